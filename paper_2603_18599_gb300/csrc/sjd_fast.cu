// Fast path of the SJD-PAC verify-and-draft step for sm_103a.
//
// Persistent CTAs (kFastThreads threads, two per SM) walk the rows of the
// step. Each row's cond/uncond slice of the allowed id range arrives in one
// shared-memory stage through a 1-D bulk asynchronous copy (the TMA engine);
// as soon as the stage has been read into registers the copy of the CTA's
// next row is issued, so HBM traffic overlaps the row's computation. The
// row then stays in registers (at most 16 KB per CTA in flight per stage):
//
//  1. guidance + temperature in fp32, each operation rounded on its own,
//     and the row maximum m;
//  2. candidates: ids with t = l - m > -34. exp(-34) < 2^-48, so every
//     other id has weight 0; the candidates are a prefix of the order
//     (l desc, id asc), hence the top-k cut can be taken among them;
//  3. top-k cut among the candidates, from registers, only when there are
//     more candidates than k;
//  4. the members are compacted into a dense shared-memory list, where the
//     weights E = rint(2^47 exp(t)) are formed without warp divergence;
//  5. top-p cut (weighted select over the list), then the kept ids are put
//     in id order with a bitmap and a popcount scan;
//  6. verification, residual resampling, proactive-drafting alternates and
//     the per-batch epilogue exactly as in the general kernel.
//
// Results are bit-identical to the general kernel (sjd_kernels.cu), which
// handles the configurations this path does not cover.

#include <cuda_bf16.h>

#include "sjd_device.cuh"

namespace sjd {
namespace {

constexpr int FT = kFastThreads;
constexpr int FNB = kFastBins;
constexpr int FCMAX = FNB / 2;          // candidates (16 bytes each) in the histogram space
constexpr float kTCut = -34.0f;         // t <= -34 => weight 0
constexpr float kBinScale = 1024.0f / 34.0f;
constexpr uint32_t kWaitLimit = 1u << 26;
static_assert(FT == kThreads, "Scratch is sized for kThreads");

// ---------------------------------------------------------------------------
// Bulk copies and the stage barrier.

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void bar_init(uint64_t* bar) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_addr(bar)));
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void bar_expect(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cta.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// Bounded wait for the barrier phase; false on timeout.
__device__ __forceinline__ bool bar_wait(uint64_t* bar, uint32_t parity) {
  for (uint32_t it = 0; it < kWaitLimit; ++it) {
    uint32_t done;
    asm volatile(
        "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}

// Issue the copies of one row's allowed-range slice into the stage.
__device__ __forceinline__ void issue_row(const DevParams& P, int row, const void* cond, const void* uncond,
                                          bool use_cfg, int esz, unsigned char* stage, uint64_t* bar) {
  const uint32_t bytes = static_cast<uint32_t>(P.nL) * esz;
  const size_t off = (static_cast<size_t>(row) * P.V + P.al0) * esz;
  bar_expect(bar, use_cfg ? 2 * bytes : bytes);
  bulk_load(stage, static_cast<const unsigned char*>(cond) + off, bytes, bar);
  if (use_cfg) bulk_load(stage + bytes, static_cast<const unsigned char*>(uncond) + off, bytes, bar);
}

// ---------------------------------------------------------------------------
// Shared-memory views.

struct FSmem {
  unsigned char* stage;
  float* list_l;              // member logits
  uint16_t* list_i;           // member local index (id - al0)
  float* list_w;              // member weight as fp32 (E * 2^-47, exact)
  float* qP;                  // q at kept ids (aliases the list)
  float* cur;                 // p^(k) of the group levels (aliases the list)
  unsigned long long* Rw;     // residual weights (aliases the list)
  uint16_t* pidx;             // kept local index, ascending
  unsigned long long* pcum;   // inclusive prefix of kept weights
  float* pp;                  // kept p (weights as fp32 before normalising)
  unsigned long long* hist;   // histogram / candidate buffer
  uint32_t* bitmap;           // one bit per local index
};

__device__ __forceinline__ FSmem fsmem_views(const DevParams& P, unsigned char* base) {
  FSmem s;
  s.stage = base + P.f_stage;
  s.list_l = reinterpret_cast<float*>(base + P.f_list_l);
  s.list_i = reinterpret_cast<uint16_t*>(base + P.f_list_i);
  s.list_w = reinterpret_cast<float*>(base + P.f_list_w);
  s.qP = reinterpret_cast<float*>(base + P.f_qP);
  s.cur = reinterpret_cast<float*>(base + P.f_cur);
  s.Rw = reinterpret_cast<unsigned long long*>(base + P.f_Rw);
  s.pidx = reinterpret_cast<uint16_t*>(base + P.f_pidx);
  s.pcum = reinterpret_cast<unsigned long long*>(base + P.f_pcum);
  s.pp = reinterpret_cast<float*>(base + P.f_pp);
  s.hist = reinterpret_cast<unsigned long long*>(base + P.f_hist);
  s.bitmap = reinterpret_cast<uint32_t*>(base + P.f_bitmap);
  return s;
}

struct FCand {
  uint32_t key;
  int idx;
  unsigned long long w;
};

// exact E of a weight stored as fp32
__device__ __forceinline__ unsigned long long w_of(float wf) { return __float2ull_rn(__fmul_rn(wf, 0x1p47f)); }

// First-level bin over t in (-34, 0]: linear in -t, monotone in l.
__device__ __forceinline__ int fbin0(float t) {
  const float x = __fmul_rn(-t, kBinScale);
  return (x < static_cast<float>(FNB - 1)) ? static_cast<int>(x) : FNB - 1;
}

// Index (local) of the need-th set bit (1-based) of the bitmap.
__device__ int nth_set_bit(const uint32_t* bitmap, int nwords, unsigned long long need, Scratch& sc) {
  if (threadIdx.x == 0) sc.bc_i[5] = INT_MAX;
  unsigned long long total;
  const uint32_t word = threadIdx.x < nwords ? bitmap[threadIdx.x] : 0u;
  const unsigned long long c = __popc(word);
  const unsigned long long ex = block_exscan_u64(c, sc, &total);
  if (ex < need && need <= ex + c) sc.bc_i[5] = threadIdx.x * 32 + __fns(word, 0, static_cast<int>(need - ex));
  __syncthreads();
  const int r = sc.bc_i[5];
  __syncthreads();
  return r;
}

// Select the cut at which the running count (or weight) of the active
// elements, in the order (key desc, local index asc), first reaches `need`
// (with need_is_tau: need = ceil(tau * total) of the level-0 total).
// src.each(f) calls f(key, idx, t, w) for this thread's active elements.
template <bool WEIGHTED, class Src>
__device__ Cut fast_select(const Src& src, const DevParams& P, float m, unsigned long long need_in,
                           bool need_is_tau, const FSmem& sm, int nwords, Scratch& sc,
                           unsigned long long* through) {
  uint32_t* h32 = reinterpret_cast<uint32_t*>(sm.hist);
  unsigned long long* h64 = sm.hist;
  FCand* cands = reinterpret_cast<FCand*>(sm.hist);
  unsigned long long need = need_in, before_all = 0;
  uint32_t klo = 0, khi = 0xFFFFFFFFu;
  for (int level = 0; level < 6; ++level) {
    const int sh = level == 0 ? 0 : max(0, 32 - __clz(khi - klo) - 10);
    for (int k = threadIdx.x; k < FNB; k += FT) {
      if (WEIGHTED) h64[k] = 0; else h32[k] = 0;
    }
    __syncthreads();
    src.each([&](uint32_t key, int idx, float t, unsigned long long w) {
      if (key < klo || key > khi) return;
      const int bk = level == 0 ? fbin0(t) : static_cast<int>((khi - key) >> sh);
      if (WEIGHTED) {
        if (w) atomicAdd(&h64[bk], w);
      } else {
        atomicAdd(&h32[bk], 1u);
      }
    });
    __syncthreads();
    constexpr int kPer = FNB / FT;
    unsigned long long loc[kPer];
    unsigned long long lsum = 0;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
      const int k = threadIdx.x * kPer + q;
      loc[q] = WEIGHTED ? h64[k] : h32[k];
      lsum += loc[q];
    }
    if (threadIdx.x == 0) {
      sc.bc_i[1] = -1;
      sc.bc_u64[0] = 0;
    }
    unsigned long long tot;
    const unsigned long long ex = block_exscan_u64(lsum, sc, &tot);
    if (level == 0 && need_is_tau) need = scale_ceil(tot, P.tau_mant, P.tau_shift);
    if (ex < need && need <= ex + lsum) {
      unsigned long long run = ex;
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        if (run < need && need <= run + loc[q]) {
          sc.bc_i[1] = threadIdx.x * kPer + q;
          sc.bc_u64[0] = run;
        }
        run += loc[q];
      }
    }
    __syncthreads();
    const int bstar = sc.bc_i[1];
    const unsigned long long bin_before = sc.bc_u64[0];
    need -= bin_before;
    before_all += bin_before;
    if (threadIdx.x == 0) {
      sc.cand_count = 0;
      sc.cand_kmin = 0xFFFFFFFFu;
      sc.cand_kmax = 0;
    }
    __syncthreads();
    uint32_t kmn = 0xFFFFFFFFu, kmx = 0;
    src.each([&](uint32_t key, int idx, float t, unsigned long long w) {
      if (key < klo || key > khi) return;
      const int bk = level == 0 ? fbin0(t) : static_cast<int>((khi - key) >> sh);
      if (bk != bstar) return;
      kmn = min(kmn, key);
      kmx = max(kmx, key);
      const uint32_t slot = atomicAdd(&sc.cand_count, 1u);
      if (slot < static_cast<uint32_t>(FCMAX)) {
        cands[slot].key = key;
        cands[slot].idx = idx;
        cands[slot].w = w;
      }
    });
    kmn = __reduce_min_sync(0xFFFFFFFFu, kmn);
    kmx = __reduce_max_sync(0xFFFFFFFFu, kmx);
    if (lane_id() == 0) {
      atomicMin(&sc.cand_kmin, kmn);
      atomicMax(&sc.cand_kmax, kmx);
    }
    __syncthreads();
    const uint32_t nc = sc.cand_count;
    const uint32_t bkmin = sc.cand_kmin, bkmax = sc.cand_kmax;
    __syncthreads();
    if (nc <= static_cast<uint32_t>(FCMAX)) {
      for (uint32_t c = threadIdx.x; c < nc; c += FT) {
        const FCand me = cands[c];
        uint32_t rank = 0;
        unsigned long long wsum = 0;
        for (uint32_t d = 0; d < nc; ++d) {
          const FCand o = cands[d];
          const bool better = o.key > me.key || (o.key == me.key && o.idx < me.idx);
          rank += better ? 1u : 0u;
          wsum += better ? o.w : 0ull;
        }
        bool pick;
        if (WEIGHTED) pick = wsum < need && need <= wsum + me.w;
        else pick = static_cast<unsigned long long>(rank) + 1 == need;
        if (pick) {
          sc.bc_u[0] = me.key;
          sc.bc_i[2] = me.idx;
          sc.bc_u64[1] = before_all + (WEIGHTED ? wsum + me.w : rank + 1);
        }
      }
      __syncthreads();
      const Cut c{sc.bc_u[0], sc.bc_i[2]};
      *through = sc.bc_u64[1];
      __syncthreads();
      return c;
    }
    klo = bkmin;
    khi = bkmax;
    if (klo == khi) {
      // every remaining element has the same value: the order is by index
      unsigned long long nth = need, wt = 1;
      if (WEIGHTED) {
        wt = quant(exp_neg(__fsub_rn(key2f(klo), m)));
        nth = (need + wt - 1) / wt;
      }
      for (int k = threadIdx.x; k < nwords; k += FT) sm.bitmap[k] = 0u;
      __syncthreads();
      src.each([&](uint32_t key, int idx, float t, unsigned long long w) {
        if (key == klo) atomicOr(&sm.bitmap[idx >> 5], 1u << (idx & 31));
      });
      __syncthreads();
      const int idx = nth_set_bit(sm.bitmap, nwords, nth, sc);
      *through = before_all + nth * wt;
      return Cut{klo, idx};
    }
  }
  *through = before_all;
  return Cut{khi, INT_MAX};
}

// Register-resident row: CPT chunks of EPC elements per thread.
template <int CPT, int EPC>
struct RegRow {
  const float* l;     // [CPT * EPC]
  float m;
  Cut kcut;
  bool members;       // false: the top-k candidates; true: members (in kcut)
  template <class F>
  __device__ __forceinline__ void each(F f) const {
#pragma unroll
    for (int i = 0; i < CPT; ++i) {
#pragma unroll
      for (int e = 0; e < EPC; ++e) {
        const float lv = l[i * EPC + e];
        const float t = __fsub_rn(lv, m);
        if (t > kTCut) {
          const uint32_t key = f2key(lv);
          const int idx = (static_cast<int>(threadIdx.x) + FT * i) * EPC + e;
          if (!members || in_cut(key, idx, kcut)) f(key, idx, t, 0ull);
        }
      }
    }
  }
};

// Member list in shared memory.
struct ListSrc {
  const float* l;
  const uint16_t* idx;
  const float* w;
  int n;
  float m;
  template <class F>
  __device__ __forceinline__ void each(F f) const {
    for (int i = threadIdx.x; i < n; i += FT) {
      const float lv = l[i];
      f(f2key(lv), static_cast<int>(idx[i]), __fsub_rn(lv, m), w_of(w[i]));
    }
  }
};

// q(v) of the stored draft row at id v (binary search in global memory).
__device__ __forceinline__ float q_lookup(const int32_t* ids, const float* pr, int n, int v, int from) {
  int lo = from, hi = n;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(ids + mid) < v) lo = mid + 1; else hi = mid;
  }
  return (lo < n && __ldg(ids + lo) == v) ? __ldg(pr + lo) : 0.0f;
}

// ---------------------------------------------------------------------------
// One row (after its logits are in registers).

template <int DT, int CPT, int MODE>
__device__ void fast_process_row(const DevParams& P, const FSmem& sm, Scratch& sc, int row,
                                 const float* l, uint32_t bad, int32_t* out_committed,
                                 int32_t* out_ncommit, int32_t* out_firstrej) {
  constexpr int EPC = DT == SJD_BF16 ? 8 : 4;
  constexpr int VPT = CPT * EPC;
  const int b = row / P.W;
  const int j = row - b * P.W;
  const int abs0 = P.abs_pos[b];
  const int slot = (abs0 + j) % P.W;
  const size_t bs = static_cast<size_t>(b) * P.W + slot;
  const uint32_t pos = static_cast<uint32_t>(abs0 + j);
  const uint32_t t = P.step_t[b];
  const int nwords = (P.nL + 31) >> 5;

  // draft group and stored draft row of this position
  int g = 1;
  int cands[kMaxK];
  int qlen = -1;
  if (MODE != kModeFromLogits) {
    g = min(max(P.gsize[bs], 1), P.K);
    for (int k = 0; k < kMaxK; ++k) cands[k] = k < g ? P.cand[bs * P.K + k] : -1;
    qlen = min(P.q_len[bs], P.S);
  }
  const int32_t* qids_g = P.q_ids + bs * P.S;
  const float* qpr_g = P.q_prob + bs * P.S;

  // ---- row maximum and the non-finite flag
  float mloc = -INFINITY;
#pragma unroll
  for (int v = 0; v < VPT; ++v) mloc = fmaxf(mloc, l[v]);
  const uint32_t kmax = block_max_u32(f2key(mloc), sc);
  bad = block_or_u32(bad, sc);
  if (bad && threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));
  const float m = key2f(kmax);
  const bool empty = kmax <= 0x007FFFFFu;  // no finite logit

  int n = 0;                   // kept ids
  unsigned long long Zk = 0;   // their total weight
  if (empty) {
    if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));
  } else {
    // ---- candidates (t > -34) and the top-k cut among them
    uint32_t ncand = 0;
#pragma unroll
    for (int v = 0; v < VPT; ++v) ncand += __fsub_rn(l[v], m) > kTCut ? 1u : 0u;
    const unsigned long long total_cand = block_sum_u64(ncand, sc);
    RegRow<CPT, EPC> regs{l, m, no_cut(), false};
    unsigned long long through;
    if (total_cand > static_cast<unsigned long long>(P.topk))
      regs.kcut = fast_select<false>(regs, P, m, static_cast<unsigned long long>(P.topk), false, sm, nwords,
                                     sc, &through);
    regs.members = true;
    // ---- dense member list, then the weights E = rint(2^47 exp(t))
    uint32_t nm = 0;
    regs.each([&](uint32_t, int, float, unsigned long long) { ++nm; });
    unsigned long long nmem;
    uint32_t at = static_cast<uint32_t>(block_exscan_u64(nm, sc, &nmem));
#pragma unroll
    for (int i = 0; i < CPT; ++i) {
#pragma unroll
      for (int e = 0; e < EPC; ++e) {
        const float lv = l[i * EPC + e];
        if (__fsub_rn(lv, m) > kTCut) {
          const int idx = (static_cast<int>(threadIdx.x) + FT * i) * EPC + e;
          if (in_cut(f2key(lv), idx, regs.kcut)) {
            if (at < static_cast<uint32_t>(P.S)) {
              sm.list_l[at] = lv;
              sm.list_i[at] = static_cast<uint16_t>(idx);
            }
            ++at;
          }
        }
      }
    }
    __syncthreads();
    if (nmem > static_cast<unsigned long long>(P.S) && threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_CAPACITY));
    const int nlist = static_cast<int>(min(nmem, static_cast<unsigned long long>(P.S)));
    unsigned long long zpart = 0;
    for (int i = threadIdx.x; i < nlist; i += FT) {
      const unsigned long long E = quant(exp_neg(__fsub_rn(sm.list_l[i], m)));
      sm.list_w[i] = dequant(E);
      zpart += E;
    }
    block_sum_u64(zpart, sc);  // (also orders the list_w writes before the reads below)
    // ---- top-p cut over the members
    Cut pcut = no_cut();
    const ListSrc list{sm.list_l, sm.list_i, sm.list_w, nlist, m};
    if (P.top_p < 1.0f) pcut = fast_select<true>(list, P, m, 0, true, sm, nwords, sc, &through);
    // ---- kept ids in id order: bitmap, per-word prefix counts, ranks
    uint32_t* word_base = reinterpret_cast<uint32_t*>(sm.hist);
    for (int k = threadIdx.x; k < nwords; k += FT) sm.bitmap[k] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < nlist; i += FT) {
      const int idx = sm.list_i[i];
      if (sm.list_w[i] > 0.0f && in_cut(f2key(sm.list_l[i]), idx, pcut))
        atomicOr(&sm.bitmap[idx >> 5], 1u << (idx & 31));
    }
    __syncthreads();
    {
      const uint32_t word = threadIdx.x < nwords ? sm.bitmap[threadIdx.x] : 0u;
      unsigned long long tot;
      const unsigned long long ex = block_exscan_u64(__popc(word), sc, &tot);
      if (threadIdx.x < nwords) word_base[threadIdx.x] = static_cast<uint32_t>(ex);
      n = static_cast<int>(tot);
    }
    if (n > P.S) {
      if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_CAPACITY));
      n = P.S;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nlist; i += FT) {
      const int idx = sm.list_i[i];
      const uint32_t word = sm.bitmap[idx >> 5];
      const uint32_t bit = 1u << (idx & 31);
      if (word & bit) {
        const int r = static_cast<int>(word_base[idx >> 5] + __popc(word & (bit - 1u)));
        if (r < P.S) {
          sm.pidx[r] = static_cast<uint16_t>(idx);
          sm.pp[r] = sm.list_w[i];
        }
      }
    }
    __syncthreads();
    // inclusive prefix of the kept weights, then p = fl(E 2^-47 / Wz)
    {
      const int per = (n + FT - 1) / FT;
      const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
      unsigned long long loc = 0;
      for (int i = i0; i < i1; ++i) loc += w_of(sm.pp[i]);
      unsigned long long tot;
      unsigned long long run = block_exscan_u64(loc, sc, &tot);
      Zk = tot;
      const float Wz = fix_to_f32(Zk);
      for (int i = i0; i < i1; ++i) {
        const float wf = sm.pp[i];
        run += w_of(wf);
        sm.pcum[i] = run;
        sm.pp[i] = __fdiv_rn(wf, Wz);
      }
    }
    __syncthreads();
  }
  auto id_of = [&](int i) { return P.al0 + static_cast<int>(sm.pidx[i]); };

  if (MODE == kModeFromLogits) {
    for (int i = threadIdx.x; i < n; i += FT) {
      P.q_ids[bs * P.S + i] = id_of(i);
      P.q_prob[bs * P.S + i] = sm.pp[i];
    }
    if (threadIdx.x == 0) {
      P.q_len[bs] = n;
      atomicAdd(&P.stats[0], 1ull);
      atomicAdd(&P.stats[2], static_cast<unsigned long long>(n));
      int x = P.lo;
      if (n > 0) {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kSynth, 0));
        x = id_of(search_excluding(sm.pcum, n, scale_floor(Zk, odd), nullptr, nullptr, 0));
      }
      P.cand[bs * P.K] = x;
      P.gsize[bs] = 1;
      P.win_tok[static_cast<size_t>(b) * P.W + j] = x;
    }
    __syncthreads();
    return;
  }

  // ---- S5/S7: verify the draft group (Sec. 3.2, Thm. 2), residual resample
  auto find_kept = [&](int c) {
    const int lc = c - P.al0;
    if (lc < 0 || lc >= P.nL) return -1;
    int lo = 0, hi = n;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (static_cast<int>(sm.pidx[mid]) < lc) lo = mid + 1; else hi = mid;
    }
    return (lo < n && static_cast<int>(sm.pidx[lo]) == lc) ? lo : -1;
  };
  int x = cands[0];
  int xidx = -1;
  if (n > 0) {
    int pidx[kMaxK];
    float qc[kMaxK];
    for (int k = 0; k < g; ++k) {
      pidx[k] = find_kept(cands[k]);
      if (qlen < 0) qc[k] = (cands[k] >= P.lo && cands[k] < P.hi) ? P.uniform_q : 0.0f;
      else qc[k] = q_lookup(qids_g, qpr_g, qlen, cands[k], 0);
    }
    const float* curk = sm.pp;
    float Sq = 0.0f, d = 1.0f;
    int removed[kMaxK];
    int nrem = 0;
    unsigned long long Rsum = 0;
    bool accepted = false;
    bool have_qP = false;
    for (int k = 1; k <= g; ++k) {
      const float q_c = k == 1 ? qc[0] : __fdiv_rn(qc[k - 1], d);
      const float p_c = pidx[k - 1] >= 0 ? curk[pidx[k - 1]] : 0.0f;
      if (q_c == 0.0f) {
        if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_INVALID_DRAFT));
      } else {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kAccept, k - 1));
        if (accept_test(odd, q_c, p_c)) {
          x = cands[k - 1];
          xidx = pidx[k - 1];
          accepted = true;
          break;
        }
      }
      if (!have_qP) {
        // q at the kept ids: each thread merges a contiguous run of kept ids
        const int per = (n + FT - 1) / FT;
        const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
        int from = 0;
        for (int i = i0; i < i1; ++i) {
          float qv = P.uniform_q;
          if (qlen >= 0) {
            const int v = id_of(i);
            int lo = from, hi = qlen;
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if (__ldg(qids_g + mid) < v) lo = mid + 1; else hi = mid;
            }
            from = lo;
            qv = (lo < qlen && __ldg(qids_g + lo) == v) ? __ldg(qpr_g + lo) : 0.0f;
          }
          sm.qP[i] = qv;
        }
        __syncthreads();
        have_qP = true;
      }
      unsigned long long part = 0;
      for (int i = threadIdx.x; i < n; i += FT) {
        float qk = sm.qP[i];
        if (k > 1) {
          bool rem = false;
          for (int e = 0; e < nrem; ++e) rem |= removed[e] == i;
          qk = rem ? 0.0f : __fdiv_rn(qk, d);
        }
        const float r = fmaxf(0.0f, __fsub_rn(curk[i], qk));
        const unsigned long long R = quant(r);
        sm.Rw[i] = R;
        part += R;
      }
      Rsum = block_sum_u64(part, sc);
      if (Rsum == 0) {  // only reachable through rounding: sample from p^(k)
        part = 0;
        for (int i = threadIdx.x; i < n; i += FT) {
          const unsigned long long R = quant(curk[i]);
          sm.Rw[i] = R;
          part += R;
        }
        Rsum = block_sum_u64(part, sc);
      }
      if (k == g) break;
      Sq = __fadd_rn(Sq, qc[k - 1]);
      if (pidx[k - 1] >= 0) removed[nrem++] = pidx[k - 1];
      const float dn = __fsub_rn(1.0f, Sq);
      if (!(dn > 0.0f)) break;
      d = dn;
      const float Wr = fix_to_f32(Rsum);
      for (int i = threadIdx.x; i < n; i += FT) sm.cur[i] = __fdiv_rn(dequant(sm.Rw[i]), Wr);
      __syncthreads();
      curk = sm.cur;
    }
    if (!accepted) {
      const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kResidual, 0));
      const unsigned long long T = scale_floor(Rsum, odd);
      const int per = (n + FT - 1) / FT;
      const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
      unsigned long long loc = 0;
      for (int i = i0; i < i1; ++i) loc += sm.Rw[i];
      if (threadIdx.x == 0) sc.bc_i[3] = -1;
      unsigned long long tot;
      unsigned long long run = block_exscan_u64(loc, sc, &tot);
      if (run <= T && T < run + loc) {
        for (int i = i0; i < i1; ++i) {
          run += sm.Rw[i];
          if (run > T) {
            sc.bc_i[3] = i;
            break;
          }
        }
      }
      __syncthreads();
      xidx = sc.bc_i[3];
      if (xidx >= 0) x = id_of(xidx);
      __syncthreads();
    }
  }

  // ---- S8: proactive-drafting alternates and the vanilla-SJD tail draw
  if (threadIdx.x == 0) {
    const int Km1 = P.K - 1;
    int32_t alts[kMaxK];
    int na = 0;
    if (n > 0 && Km1 > 0)
      na = draw_without_replacement(P, sm.pcum, id_of, n, Zk, xidx, pos, t, static_cast<uint32_t>(b), Km1, alts);
    for (int k = 0; k < na; ++k) P.res_alt[bs * Km1 + k] = alts[k];
    P.res_altn[bs] = na;
    P.res_x[bs] = x;
    P.res_dev[bs] = x != cands[0] ? 1 : 0;
    if (!P.ac) {
      int xf = x, fidx = -1;
      if (n > 0) {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kResidual, 0));
        fidx = search_excluding(sm.pcum, n, scale_floor(Zk, odd), nullptr, nullptr, 0);
        xf = id_of(fidx);
      }
      int naf = 0;
      if (n > 0 && Km1 > 0)
        naf = draw_without_replacement(P, sm.pcum, id_of, n, Zk, fidx, pos, t, static_cast<uint32_t>(b), Km1, alts);
      for (int k = 0; k < naf; ++k) P.res_altf[bs * Km1 + k] = alts[k];
      P.res_altfn[bs] = naf;
      P.res_xf[bs] = xf;
    }
    P.q_len[bs] = n;
    atomicAdd(&P.stats[0], 1ull);
    atomicAdd(&P.stats[1], static_cast<unsigned long long>(max(qlen, 0)));
    atomicAdd(&P.stats[2], static_cast<unsigned long long>(n));
  }
  // the row P^t replaces the stored draft row (which verification has read)
  for (int i = threadIdx.x; i < n; i += FT) {
    P.q_ids[bs * P.S + i] = id_of(i);
    P.q_prob[bs * P.S + i] = sm.pp[i];
  }

  // ---- last row of the batch element: S6 (+ S9 in the fused step)
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const uint32_t done = atomicAdd(P.ticket + b, 1u);
    sc.bc_i[0] = done == static_cast<uint32_t>(P.W - 1) ? 1 : 0;
  }
  __syncthreads();
  if (sc.bc_i[0]) {
    __threadfence();
    batch_epilogue(P, b, MODE == kModeStep, out_committed, out_ncommit, out_firstrej, sc);
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// The persistent kernel.

template <int DT, int CPT, int MODE>
__global__ void __launch_bounds__(FT, 2)
fast_row_kernel(DevParams P, const void* __restrict__ cond, const void* __restrict__ uncond,
                bool use_cfg, int32_t* out_committed, int32_t* out_ncommit, int32_t* out_firstrej) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ Scratch sc;
  __shared__ __align__(8) uint64_t bar;
  const FSmem sm = fsmem_views(P, smem_raw);
  constexpr int EPC = DT == SJD_BF16 ? 8 : 4;
  constexpr int VPT = CPT * EPC;
  constexpr int esz = DT == SJD_BF16 ? 2 : 4;
  const int rows = P.B * P.W;
  int row = blockIdx.x;
  if (row >= rows) return;
  if (threadIdx.x == 0) bar_init(&bar);
  __syncthreads();
  if (threadIdx.x == 0) issue_row(P, row, cond, uncond, use_cfg, esz, sm.stage, &bar);
  const int nch = P.nL / EPC;
  const bool temp = P.temp != 1.0f;
  for (uint32_t it = 0;; ++it) {
    if (!bar_wait(&bar, it & 1u)) {
      // the copy did not land: report, give it one more bounded wait, stop
      if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_TIMEOUT));
      bar_wait(&bar, it & 1u);
      return;
    }
    float l[VPT];
    uint32_t bad = 0;
#pragma unroll
    for (int i = 0; i < CPT; ++i) {
      const int c = static_cast<int>(threadIdx.x) + FT * i;
      float cv[EPC], uv[EPC];
      if (c < nch) {
        if (DT == SJD_BF16) {
          const uint4 cw = reinterpret_cast<const uint4*>(sm.stage)[c];
          const uint32_t cws[4] = {cw.x, cw.y, cw.z, cw.w};
          uint32_t uws[4] = {0u, 0u, 0u, 0u};
          if (use_cfg) {
            const uint4 uw = reinterpret_cast<const uint4*>(sm.stage + P.nL * esz)[c];
            uws[0] = uw.x; uws[1] = uw.y; uws[2] = uw.z; uws[3] = uw.w;
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            cv[2 * q] = __uint_as_float(cws[q] << 16);
            cv[2 * q + 1] = __uint_as_float(cws[q] & 0xFFFF0000u);
            uv[2 * q] = __uint_as_float(uws[q] << 16);
            uv[2 * q + 1] = __uint_as_float(uws[q] & 0xFFFF0000u);
          }
        } else {
          const float4 cw = reinterpret_cast<const float4*>(sm.stage)[c];
          float4 uw = make_float4(0.f, 0.f, 0.f, 0.f);
          if (use_cfg) uw = reinterpret_cast<const float4*>(sm.stage + P.nL * esz)[c];
          cv[0] = cw.x; cv[1] = cw.y; cv[2] = cw.z; cv[3] = cw.w;
          uv[0] = uw.x; uv[1] = uw.y; uv[2] = uw.z; uv[3] = uw.w;
        }
#pragma unroll
        for (int q = 0; q < EPC; q += 2) {
          // guidance u + s (c - u), every operation rounded on its own (the
          // packed f32x2 multiply and add would be fused by the backend)
          float o[2] = {cv[q], cv[q + 1]};
          if (use_cfg) {
            o[0] = __fadd_rn(uv[q], __fmul_rn(P.cfg, __fsub_rn(cv[q], uv[q])));
            o[1] = __fadd_rn(uv[q + 1], __fmul_rn(P.cfg, __fsub_rn(cv[q + 1], uv[q + 1])));
          }
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int v = P.al0 + c * EPC + q + h;
            float x = o[h];
            if (temp) x = __fdiv_rn(x, P.temp);
            if (v >= P.lo && v < P.hi) {
              if (!(x < INFINITY) && !(x == -INFINITY)) {
                bad = 1u;
                x = -INFINITY;
              }
            } else {
              x = pad_value();
            }
            l[i * EPC + q + h] = x;
          }
        }
      } else {
#pragma unroll
        for (int q = 0; q < EPC; ++q) l[i * EPC + q] = pad_value();
      }
    }
    __syncthreads();  // the stage has been read: fetch the next row into it
    const int next = row + static_cast<int>(gridDim.x);
    if (threadIdx.x == 0 && next < rows) {
      // order the generic-proxy reads of the stage before the async-proxy writes
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      issue_row(P, next, cond, uncond, use_cfg, esz, sm.stage, &bar);
    }
    fast_process_row<DT, CPT, MODE>(P, sm, sc, row, l, bad, out_committed, out_ncommit, out_firstrej);
    row = next;
    if (row >= rows) break;
  }
}

template <int DT, int CPT, int MODE>
cudaError_t set_one(int bytes) {
  return cudaFuncSetAttribute(fast_row_kernel<DT, CPT, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

template <int DT, int CPT>
cudaError_t set_all_modes(int bytes) {
  cudaError_t e = set_one<DT, CPT, kModeVerify>(bytes);
  if (e == cudaSuccess) e = set_one<DT, CPT, kModeStep>(bytes);
  if (e == cudaSuccess) e = set_one<DT, CPT, kModeFromLogits>(bytes);
  return e;
}

template <int DT, int CPT>
void launch_t(const DevParams& p, int mode, dim3 grid, const void* cond, const void* uncond, bool use_cfg,
              int32_t* oc, int32_t* on, int32_t* of, cudaStream_t s) {
  const dim3 block(FT);
  switch (mode) {
    case kModeVerify:
      fast_row_kernel<DT, CPT, kModeVerify><<<grid, block, p.f_smem_bytes, s>>>(p, cond, uncond, use_cfg, oc, on, of);
      break;
    case kModeStep:
      fast_row_kernel<DT, CPT, kModeStep><<<grid, block, p.f_smem_bytes, s>>>(p, cond, uncond, use_cfg, oc, on, of);
      break;
    default:
      fast_row_kernel<DT, CPT, kModeFromLogits><<<grid, block, p.f_smem_bytes, s>>>(p, cond, uncond, use_cfg, oc, on, of);
      break;
  }
}

int g_num_sms = 0;

}  // namespace


cudaError_t set_fast_row_kernel_smem(int bytes) {
  cudaError_t e = cudaSuccess;
  auto acc = [&](cudaError_t x) { if (e == cudaSuccess) e = x; };
  acc(set_all_modes<SJD_BF16, 1>(bytes));
  acc(set_all_modes<SJD_BF16, 2>(bytes));
  acc(set_all_modes<SJD_BF16, 3>(bytes));
  acc(set_all_modes<SJD_BF16, 4>(bytes));
  acc(set_all_modes<SJD_F32, 1>(bytes));
  acc(set_all_modes<SJD_F32, 2>(bytes));
  acc(set_all_modes<SJD_F32, 3>(bytes));
  acc(set_all_modes<SJD_F32, 4>(bytes));
  return e;
}

cudaError_t launch_fast_row(const DevParams& p, int mode, int dtype, const void* cond, const void* uncond,
                            bool use_cfg, int32_t* oc, int32_t* on, int32_t* of, cudaStream_t s) {
  if (g_num_sms == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const int rows = p.B * p.W;
  const dim3 grid(static_cast<unsigned>(std::min(rows, g_num_sms * std::max(p.fast_ctas, 1))));
  if (dtype == SJD_BF16) {
    switch (p.fast_cpt) {
      case 1: launch_t<SJD_BF16, 1>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 2: launch_t<SJD_BF16, 2>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 3: launch_t<SJD_BF16, 3>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      default: launch_t<SJD_BF16, 4>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
    }
  } else {
    switch (p.fast_cpt) {
      case 1: launch_t<SJD_F32, 1>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 2: launch_t<SJD_F32, 2>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 3: launch_t<SJD_F32, 3>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      default: launch_t<SJD_F32, 4>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
    }
  }
  return cudaGetLastError();
}

}  // namespace sjd
