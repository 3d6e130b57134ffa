// Fast path of the SJD-PAC verify-and-draft step for sm_103a.
//
// Persistent CTAs (kFastThreads threads, up to two per SM) walk the rows of
// the step. Each row's cond/uncond slice of the allowed id range arrives in
// one shared-memory stage through a 1-D bulk asynchronous copy (the TMA
// engine); as soon as the stage has been read into registers the copy of
// the CTA's next row is issued, so HBM traffic overlaps the computation.
//
//  1. guidance + temperature in fp32, each operation rounded on its own,
//     and the row maximum m (NaN-propagating, so one reduction also detects
//     NaN; +inf shows up as m = +inf);
//  2. candidates: ids with t = l - m > -34. exp(-34) < 2^-48, so every other
//     id has weight 0. The candidates are a prefix of the order (l desc, id
//     asc), so the top-k cut can be taken among them. They are compacted
//     into a dense shared-memory list;
//  3. top-k cut among the candidates (only when there are more than k),
//     weights E = rint(2^47 exp(t)) of the members, exact total Z;
//  4. top-p cut (weighted select over the members), then the kept ids are
//     put in id order with a bitmap and a popcount scan;
//  5. verification, residual resampling and proactive-drafting draws with
//     the decisions (and every fp64 operation) taken by one thread and
//     broadcast, the per-batch epilogue as in the general kernel.
//
// Results are bit-identical to the general kernel (sjd_kernels.cu), which
// handles the configurations this path does not cover.

#include <cuda_bf16.h>

#include "sjd_device.cuh"

namespace sjd {
namespace {

constexpr int FT = kFastThreads;
constexpr int FW = FT / 32;
constexpr int FNB = kFastBins;
constexpr int FCMAX = FNB / 2;          // candidates (16 bytes each) in the histogram space
constexpr float kTCut = -34.0f;         // t <= -34 => weight 0
constexpr float kBinScale = 1024.0f / 34.0f;
constexpr uint32_t kWaitLimit = 1u << 26;

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

// max that propagates NaN (the IEEE maximum with NaN preserved)
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// ---------------------------------------------------------------------------
// Per-CTA scratch and cheap block-wide operations (one warp combines the
// per-warp partials; results are broadcast through shared memory).

struct FScratch {
  unsigned long long red[FW];
  unsigned long long red2[FW];
  unsigned long long bc64[8];
  int bi[16];
  float bf[4];
  uint32_t cand_count, cand_kmin, cand_kmax;
  int cands[kMaxK];      // draft group of the row
  int gpidx[kMaxK];      // its positions in the kept row (-1: absent)
  float gqc[kMaxK];      // q at the group's tokens
};

__device__ __forceinline__ int lane() { return threadIdx.x & 31; }
__device__ __forceinline__ int warp() { return threadIdx.x >> 5; }

__device__ __forceinline__ unsigned long long wsum64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

// Sum over the block of one u64 per thread.
__device__ unsigned long long fsum(unsigned long long v, FScratch& s) {
  v = wsum64(v);
  if (lane() == 0) s.red[warp()] = v;
  __syncthreads();
  if (warp() == 0) {
    unsigned long long x = lane() < FW ? s.red[lane()] : 0ull;
#pragma unroll
    for (int o = FW / 2; o; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    if (lane() == 0) s.bc64[7] = x;
  }
  __syncthreads();
  return s.bc64[7];
}

// Exclusive scan of one u64 per thread in thread order; *total = the sum.
__device__ unsigned long long fexscan(unsigned long long v, FScratch& s, unsigned long long* total) {
  unsigned long long incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane() >= o) incl += y;
  }
  if (lane() == 31) s.red[warp()] = incl;
  __syncthreads();
  if (warp() == 0) {
    const unsigned long long w = lane() < FW ? s.red[lane()] : 0ull;
    unsigned long long x = w;
#pragma unroll
    for (int o = 1; o < FW; o <<= 1) {
      const unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane() >= o) x += y;
    }
    if (lane() < FW) s.red2[lane()] = x - w;
    if (lane() == FW - 1) s.bc64[4] = x;
  }
  __syncthreads();
  *total = s.bc64[4];
  return s.red2[warp()] + incl - v;
}

// Exclusive scan of one u32 per thread (counts < 2^32).
__device__ uint32_t fexscan32(uint32_t v, FScratch& s, uint32_t* total) {
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane() >= o) incl += y;
  }
  if (lane() == 31) s.red[warp()] = incl;
  __syncthreads();
  if (warp() == 0) {
    const uint32_t w = lane() < FW ? static_cast<uint32_t>(s.red[lane()]) : 0u;
    uint32_t x = w;
#pragma unroll
    for (int o = 1; o < FW; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane() >= o) x += y;
    }
    if (lane() < FW) s.red2[lane()] = x - w;
    if (lane() == FW - 1) s.bc64[3] = x;
  }
  __syncthreads();
  *total = static_cast<uint32_t>(s.bc64[3]);
  return static_cast<uint32_t>(s.red2[warp()]) + incl - v;
}

__device__ uint32_t fmax32(uint32_t v, FScratch& s) {
  v = __reduce_max_sync(0xFFFFFFFFu, v);
  if (lane() == 0) s.red[warp()] = v;
  __syncthreads();
  if (warp() == 0) {
    uint32_t x = lane() < FW ? static_cast<uint32_t>(s.red[lane()]) : 0u;
    x = __reduce_max_sync(0xFFFFFFFFu, x);
    if (lane() == 0) s.bc64[2] = x;
  }
  __syncthreads();
  return static_cast<uint32_t>(s.bc64[2]);
}

// ---------------------------------------------------------------------------
// Shared-memory views.

struct FSmem {
  unsigned char* stage;
  float* list_l;              // candidate logits
  uint16_t* list_i;           // candidate local index (id - al0)
  float* list_w;              // member weight as fp32 (E * 2^-47, exact); -1: not a member
  float* qP;                  // q at kept ids (aliases the list)
  float* cur;                 // p^(k) of the group levels (aliases the list)
  unsigned long long* Rw;     // residual weights (aliases the list)
  uint16_t* pidx;             // kept local index, ascending
  unsigned long long* pcum;   // inclusive prefix of kept weights
  float* pp;                  // kept p (weights as fp32 before normalising)
  unsigned long long* hist;   // histogram / candidate buffer / word prefix counts
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

// Local index of the need-th set bit (1-based) of the bitmap.
__device__ int nth_set_bit(const uint32_t* bitmap, int nwords, unsigned long long need, FScratch& s) {
  if (threadIdx.x == 0) s.bi[5] = INT_MAX;
  unsigned long long total;
  const uint32_t word = static_cast<int>(threadIdx.x) < nwords ? bitmap[threadIdx.x] : 0u;
  const unsigned long long c = __popc(word);
  const unsigned long long ex = fexscan(c, s, &total);
  if (ex < need && need <= ex + c) s.bi[5] = threadIdx.x * 32 + __fns(word, 0, static_cast<int>(need - ex));
  __syncthreads();
  const int r = s.bi[5];
  __syncthreads();
  return r;
}

// Select the cut at which the running count (or weight) of the active
// elements, in the order (key desc, local index asc), first reaches `need`
// (with need_is_tau: need = ceil(tau * total) of the level-0 total).
// src.each(f) calls f(key, idx, t, w) for this thread's active elements.
template <bool WEIGHTED, class Src>
__device__ Cut fast_select(const Src& src, const DevParams& P, float m, unsigned long long need_in,
                           bool need_is_tau, const FSmem& sm, int nwords, FScratch& s) {
  uint32_t* h32 = reinterpret_cast<uint32_t*>(sm.hist);
  unsigned long long* h64 = sm.hist;
  FCand* cands = reinterpret_cast<FCand*>(sm.hist);
  unsigned long long need = need_in;
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
      s.bi[1] = -1;
      s.bc64[0] = 0;
    }
    unsigned long long tot;
    const unsigned long long ex = fexscan(lsum, s, &tot);
    if (level == 0 && need_is_tau) need = scale_ceil(tot, P.tau_mant, P.tau_shift);
    if (ex < need && need <= ex + lsum) {
      unsigned long long run = ex;
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        if (run < need && need <= run + loc[q]) {
          s.bi[1] = threadIdx.x * kPer + q;
          s.bc64[0] = run;
        }
        run += loc[q];
      }
    }
    if (threadIdx.x == 0) {
      s.cand_count = 0;
      s.cand_kmin = 0xFFFFFFFFu;
      s.cand_kmax = 0;
    }
    __syncthreads();
    const int bstar = s.bi[1];
    need -= s.bc64[0];
    uint32_t kmn = 0xFFFFFFFFu, kmx = 0;
    src.each([&](uint32_t key, int idx, float t, unsigned long long w) {
      if (key < klo || key > khi) return;
      const int bk = level == 0 ? fbin0(t) : static_cast<int>((khi - key) >> sh);
      if (bk != bstar) return;
      kmn = min(kmn, key);
      kmx = max(kmx, key);
      const uint32_t slot = atomicAdd(&s.cand_count, 1u);
      if (slot < static_cast<uint32_t>(FCMAX)) {
        cands[slot].key = key;
        cands[slot].idx = idx;
        cands[slot].w = w;
      }
    });
    kmn = __reduce_min_sync(0xFFFFFFFFu, kmn);
    kmx = __reduce_max_sync(0xFFFFFFFFu, kmx);
    if (lane() == 0) {
      atomicMin(&s.cand_kmin, kmn);
      atomicMax(&s.cand_kmax, kmx);
    }
    __syncthreads();
    const uint32_t nc = s.cand_count;
    const uint32_t bkmin = s.cand_kmin, bkmax = s.cand_kmax;
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
          s.bi[2] = static_cast<int>(me.key);
          s.bi[3] = me.idx;
        }
      }
      __syncthreads();
      const Cut c{static_cast<uint32_t>(s.bi[2]), s.bi[3]};
      __syncthreads();
      return c;
    }
    __syncthreads();
    klo = bkmin;
    khi = bkmax;
    if (klo == khi) {
      // every remaining element has the same value: the order is by index
      unsigned long long nth = need;
      if (WEIGHTED) {
        const unsigned long long wt = quant(exp_neg(__fsub_rn(key2f(klo), m)));
        nth = (need + wt - 1) / wt;
      }
      for (int k = threadIdx.x; k < nwords; k += FT) sm.bitmap[k] = 0u;
      __syncthreads();
      src.each([&](uint32_t key, int idx, float t, unsigned long long w) {
        if (key == klo) atomicOr(&sm.bitmap[idx >> 5], 1u << (idx & 31));
      });
      __syncthreads();
      return Cut{klo, nth_set_bit(sm.bitmap, nwords, nth, s)};
    }
  }
  return Cut{khi, INT_MAX};
}

// Register-resident row: CPT full chunk slots plus one tail slot per thread.
template <int CPT, int EPC>
struct RegRow {
  const float* l;     // [(CPT + 1) * EPC]
  float m;
  bool tail;          // this thread holds a tail chunk
  template <class F>
  __device__ __forceinline__ void each(F f) const {
#pragma unroll
    for (int i = 0; i <= CPT; ++i) {
      if (i == CPT && !tail) break;
#pragma unroll
      for (int e = 0; e < EPC; ++e) {
        const float lv = l[i * EPC + e];
        const float t = __fsub_rn(lv, m);
        if (t > kTCut) f(f2key(lv), (static_cast<int>(threadIdx.x) + FT * i) * EPC + e, t, 0ull);
      }
    }
  }
};

// Candidate list in shared memory; with WEIGHTS only the members (w >= 0).
template <bool WEIGHTS>
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
      if (WEIGHTS) {
        const float wf = w[i];
        if (wf < 0.0f) continue;
        f(f2key(lv), static_cast<int>(idx[i]), __fsub_rn(lv, m), w_of(wf));
      } else {
        f(f2key(lv), static_cast<int>(idx[i]), __fsub_rn(lv, m), 0ull);
      }
    }
  }
};

// ---------------------------------------------------------------------------
// One row (after its logits are in registers).

template <int DT, int CPT, int MODE>
__device__ void fast_process_row(const DevParams& P, const FSmem& sm, FScratch& s, int row, float* l,
                                 float mnan, bool tail, unsigned long long* stats, int32_t* out_committed,
                                 int32_t* out_ncommit, int32_t* out_firstrej, Scratch& esc) {
  constexpr int EPC = DT == SJD_BF16 ? 8 : 4;
  const int b = row / P.W;
  const int j = row - b * P.W;
  const int abs0 = P.abs_pos[b];
  const int slot = (abs0 + j) % P.W;
  const size_t bs = static_cast<size_t>(b) * P.W + slot;
  const uint32_t pos = static_cast<uint32_t>(abs0 + j);
  const uint32_t t = P.step_t[b];
  const int nwords = (P.nL + 31) >> 5;
  const int32_t* qids_g = P.q_ids + bs * P.S;
  const float* qpr_g = P.q_prob + bs * P.S;
  const int lcap = P.f_lcap;

  // ---- row maximum (NaN-propagating); NaN / +inf are reported, then act as -inf
  uint32_t kmax = fmax32(f2key(mnan), s);
  float m = key2f(kmax);
  if (!(m < INFINITY)) {  // m is NaN or +inf (rare): recompute without them
    if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));
    float mm = -INFINITY;
#pragma unroll
    for (int i = 0; i <= CPT; ++i) {
      if (i == CPT && !tail) break;
#pragma unroll
      for (int e = 0; e < EPC; ++e) {
        const int v = P.al0 + (static_cast<int>(threadIdx.x) + FT * i) * EPC + e;
        float& x = l[i * EPC + e];
        if (v >= P.lo && v < P.hi && !(x < INFINITY) && !(x == -INFINITY)) x = -INFINITY;
        mm = fmaxf(mm, x);
      }
    }
    kmax = fmax32(f2key(mm), s);
    m = key2f(kmax);
  }
  const bool empty = kmax <= 0x007FFFFFu;  // no finite logit

  int n = 0;                   // kept ids
  unsigned long long Zk = 0;   // their total weight
  int g = 1, qlen = -1;
  if (MODE != kModeFromLogits) {
    g = min(max(P.gsize[bs], 1), P.K);
    qlen = min(P.q_len[bs], P.S);
  }
  if (empty) {
    if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));
  } else {
    // ---- candidates: flags, count, scan, write to the dense list
    const RegRow<CPT, EPC> regs{l, m, tail};
    uint32_t cmask = 0;   // candidate flags of this thread's values
#pragma unroll
    for (int i = 0; i <= CPT; ++i) {
      if (i == CPT && !tail) break;
#pragma unroll
      for (int e = 0; e < EPC; ++e)
        cmask |= (__fsub_rn(l[i * EPC + e], m) > kTCut) ? (1u << (i * EPC + e)) : 0u;
    }
    uint32_t total_cand;
    uint32_t at = fexscan32(__popc(cmask), s, &total_cand);
    Cut kcut = no_cut();
    int nlist;
    if (total_cand <= static_cast<uint32_t>(lcap)) {
#pragma unroll
      for (int i = 0; i <= CPT; ++i) {
        if (i == CPT && !tail) break;
#pragma unroll
        for (int e = 0; e < EPC; ++e) {
          if (cmask & (1u << (i * EPC + e))) {
            sm.list_l[at] = l[i * EPC + e];
            sm.list_i[at] = static_cast<uint16_t>((static_cast<int>(threadIdx.x) + FT * i) * EPC + e);
            ++at;
          }
        }
      }
      __syncthreads();
      nlist = static_cast<int>(total_cand);
      if (total_cand > static_cast<uint32_t>(P.topk)) {
        const ListSrc<false> cl{sm.list_l, sm.list_i, sm.list_w, nlist, m};
        kcut = fast_select<false>(cl, P, m, static_cast<unsigned long long>(P.topk), false, sm, nwords, s);
      }
    } else {
      // more candidates than the list holds: top-k cut from registers, then
      // only the members (at most k <= S <= list capacity) go to the list
      kcut = fast_select<false>(regs, P, m, static_cast<unsigned long long>(P.topk), false, sm, nwords, s);
      uint32_t nm = 0;
      regs.each([&](uint32_t key, int idx, float, unsigned long long) { nm += in_cut(key, idx, kcut) ? 1u : 0u; });
      uint32_t nmem;
      at = fexscan32(nm, s, &nmem);
      regs.each([&](uint32_t key, int idx, float, unsigned long long) {
        if (in_cut(key, idx, kcut)) {
          if (at < static_cast<uint32_t>(lcap)) {
            sm.list_l[at] = key2f(key);
            sm.list_i[at] = static_cast<uint16_t>(idx);
          }
          ++at;
        }
      });
      __syncthreads();
      if (nmem > static_cast<uint32_t>(lcap) && threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_CAPACITY));
      nlist = min(static_cast<int>(nmem), lcap);
    }
    // ---- member weights and their exact total
    unsigned long long zpart = 0;
    for (int i = threadIdx.x; i < nlist; i += FT) {
      const float lv = sm.list_l[i];
      float wf = -1.0f;
      if (in_cut(f2key(lv), sm.list_i[i], kcut)) {
        const unsigned long long E = quant(exp_neg(__fsub_rn(lv, m)));
        wf = dequant(E);
        zpart += E;
      }
      sm.list_w[i] = wf;
    }
    fsum(zpart, s);  // (orders the list_w writes before the reads below)
    // ---- top-p cut over the members
    Cut pcut = no_cut();
    if (P.top_p < 1.0f) {
      const ListSrc<true> ml{sm.list_l, sm.list_i, sm.list_w, nlist, m};
      pcut = fast_select<true>(ml, P, m, 0, true, sm, nwords, s);
    }
    // ---- kept ids (members in the top-p cut with weight > 0) in id order
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
      const uint32_t word = static_cast<int>(threadIdx.x) < nwords ? sm.bitmap[threadIdx.x] : 0u;
      uint32_t tot;
      const uint32_t ex = fexscan32(__popc(word), s, &tot);
      if (static_cast<int>(threadIdx.x) < nwords) word_base[threadIdx.x] = ex;
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
      unsigned long long run = fexscan(loc, s, &tot);
      Zk = tot;
      if (threadIdx.x == 0) s.bf[0] = fix_to_f32(Zk);
      __syncthreads();
      const float Wz = s.bf[0];
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
      stats[0] += 1;
      stats[2] += static_cast<unsigned long long>(n);
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

  // ---- S5/S7: verify the draft group (Sec. 3.2, Thm. 2), residual resample.
  // Thread 0 takes every decision (and every fp64 operation); all threads
  // share the per-element residual passes.
  if (threadIdx.x == 0) {
    for (int k = 0; k < g; ++k) {
      const int c = P.cand[bs * P.K + k];
      s.cands[k] = c;
      int pi = -1;
      const int lc = c - P.al0;
      if (n > 0 && lc >= 0 && lc < P.nL) {
        int lo = 0, hi = n;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (static_cast<int>(sm.pidx[mid]) < lc) lo = mid + 1; else hi = mid;
        }
        pi = (lo < n && static_cast<int>(sm.pidx[lo]) == lc) ? lo : -1;
      }
      s.gpidx[k] = pi;
      float qv;
      if (qlen < 0) {
        qv = (c >= P.lo && c < P.hi) ? P.uniform_q : 0.0f;
      } else {
        int lo = 0, hi = qlen;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (__ldg(qids_g + mid) < c) lo = mid + 1; else hi = mid;
        }
        qv = (lo < qlen && __ldg(qids_g + lo) == c) ? __ldg(qpr_g + lo) : 0.0f;
      }
      s.gqc[k] = qv;
    }
  }
  __syncthreads();
  const int c1 = s.cands[0];
  int x = c1;
  int xidx = -1;
  if (n > 0) {
    const float* curk = sm.pp;
    float d = 1.0f;
    float Sq = 0.0f;   // (thread 0)
    int nrem = 0;
    int removed[kMaxK];
    unsigned long long Rsum = 0;
    bool have_qP = false;
    bool accepted = false;
    for (int k = 1; k <= g; ++k) {
      if (threadIdx.x == 0) {
        const float q_c = k == 1 ? s.gqc[0] : __fdiv_rn(s.gqc[k - 1], d);
        const int pi = s.gpidx[k - 1];
        const float p_c = pi >= 0 ? curk[pi] : 0.0f;
        int acc = 0;
        if (q_c == 0.0f) {
          atomicOr(P.err, err_bit(SJD_ERR_INVALID_DRAFT));
        } else {
          const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kAccept, k - 1));
          acc = accept_test(odd, q_c, p_c) ? 1 : 0;
        }
        s.bi[6] = acc;
      }
      __syncthreads();
      if (s.bi[6]) {
        x = s.cands[k - 1];
        xidx = s.gpidx[k - 1];
        accepted = true;
        break;
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
      Rsum = fsum(part, s);
      if (Rsum == 0) {  // only reachable through rounding: sample from p^(k)
        part = 0;
        for (int i = threadIdx.x; i < n; i += FT) {
          const unsigned long long R = quant(curk[i]);
          sm.Rw[i] = R;
          part += R;
        }
        Rsum = fsum(part, s);
      }
      if (k == g) break;
      // adjusted draft q^(k+1): c_1..c_k removed, renormalised (thread 0
      // computes, everyone reads the same values)
      if (threadIdx.x == 0) {
        Sq = __fadd_rn(Sq, s.gqc[k - 1]);
        s.bf[2] = __fsub_rn(1.0f, Sq);
        s.bf[3] = fix_to_f32(Rsum);
      }
      __syncthreads();
      if (s.gpidx[k - 1] >= 0) removed[nrem++] = s.gpidx[k - 1];
      const float dn = s.bf[2];
      if (!(dn > 0.0f)) break;
      d = dn;
      const float Wr = s.bf[3];
      for (int i = threadIdx.x; i < n; i += FT) sm.cur[i] = __fdiv_rn(dequant(sm.Rw[i]), Wr);
      __syncthreads();
      curk = sm.cur;
    }
    if (!accepted) {
      if (threadIdx.x == 0) {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kResidual, 0));
        s.bc64[1] = scale_floor(Rsum, odd);
        s.bi[7] = -1;
      }
      const int per = (n + FT - 1) / FT;
      const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
      unsigned long long loc = 0;
      for (int i = i0; i < i1; ++i) loc += sm.Rw[i];
      unsigned long long tot;
      unsigned long long run = fexscan(loc, s, &tot);
      const unsigned long long T = s.bc64[1];
      if (run <= T && T < run + loc) {
        for (int i = i0; i < i1; ++i) {
          run += sm.Rw[i];
          if (run > T) {
            s.bi[7] = i;
            break;
          }
        }
      }
      __syncthreads();
      xidx = s.bi[7];
      if (xidx >= 0) x = id_of(xidx);
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
    P.res_dev[bs] = x != c1 ? 1 : 0;
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
    stats[0] += 1;
    stats[1] += static_cast<unsigned long long>(max(qlen, 0));
    stats[2] += static_cast<unsigned long long>(n);
  }
  // the row P^t replaces the stored draft row (which verification has read)
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += FT) {
    P.q_ids[bs * P.S + i] = id_of(i);
    P.q_prob[bs * P.S + i] = sm.pp[i];
  }

  // ---- last row of the batch element: S6 (+ S9 in the fused step)
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const uint32_t done = atomicAdd(P.ticket + b, 1u);
    s.bi[0] = done == static_cast<uint32_t>(P.W - 1) ? 1 : 0;
  }
  __syncthreads();
  if (s.bi[0]) {
    __threadfence();
    batch_epilogue(P, b, MODE == kModeStep, out_committed, out_ncommit, out_firstrej, esc);
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
  __shared__ FScratch s;
  __shared__ Scratch esc;   // for the shared per-batch epilogue
  __shared__ __align__(8) uint64_t bar;
  const FSmem sm = fsmem_views(P, smem_raw);
  constexpr int EPC = DT == SJD_BF16 ? 8 : 4;
  constexpr int esz = DT == SJD_BF16 ? 2 : 4;
  const int rows = P.B * P.W;
  int row = blockIdx.x;
  if (row >= rows) return;
  if (threadIdx.x == 0) bar_init(&bar);
  __syncthreads();
  if (threadIdx.x == 0) issue_row(P, row, cond, uncond, use_cfg, esz, sm.stage, &bar);
  const int nch = P.nL / EPC;
  const bool tail = static_cast<int>(threadIdx.x) < nch - CPT * FT;
  const bool temp = P.temp != 1.0f;
  unsigned long long stats[3] = {0ull, 0ull, 0ull};
  for (uint32_t it = 0;; ++it) {
    if (!bar_wait(&bar, it & 1u)) {
      // the copy did not land: report, give it one more bounded wait, stop
      if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_TIMEOUT));
      bar_wait(&bar, it & 1u);
      return;
    }
    float l[(CPT + 1) * EPC];
    float mnan = -INFINITY;
#pragma unroll
    for (int i = 0; i <= CPT; ++i) {
      if (i == CPT && !tail) break;
      const int c = static_cast<int>(threadIdx.x) + FT * i;
      float cv[EPC], uv[EPC];
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
      const int v0 = P.al0 + c * EPC;
      const bool inside = v0 >= P.lo && v0 + EPC <= P.hi;
#pragma unroll
      for (int q = 0; q < EPC; ++q) {
        // guidance u + s (c - u), each operation rounded on its own (a packed
        // f32x2 multiply followed by an add would be fused by the backend)
        float x = use_cfg ? __fadd_rn(uv[q], __fmul_rn(P.cfg, __fsub_rn(cv[q], uv[q]))) : cv[q];
        if (temp) x = __fdiv_rn(x, P.temp);
        if (!inside && !(v0 + q >= P.lo && v0 + q < P.hi)) x = pad_value();
        else mnan = fmax_nan(mnan, x);
        l[i * EPC + q] = x;
      }
    }
    __syncthreads();  // the stage has been read: fetch the next row into it
    const int next = row + static_cast<int>(gridDim.x);
    if (threadIdx.x == 0 && next < rows) {
      // order the generic-proxy reads of the stage before the async-proxy writes
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      issue_row(P, next, cond, uncond, use_cfg, esz, sm.stage, &bar);
    }
    fast_process_row<DT, CPT, MODE>(P, sm, s, row, l, mnan, tail, stats, out_committed, out_ncommit,
                                    out_firstrej, esc);
    row = next;
    if (row >= rows) break;
  }
  if (threadIdx.x == 0) {
    atomicAdd(&P.stats[0], stats[0]);
    if (stats[1]) atomicAdd(&P.stats[1], stats[1]);
    atomicAdd(&P.stats[2], stats[2]);
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
  acc(set_all_modes<SJD_BF16, 0>(bytes));
  acc(set_all_modes<SJD_BF16, 1>(bytes));
  acc(set_all_modes<SJD_BF16, 2>(bytes));
  acc(set_all_modes<SJD_BF16, 3>(bytes));
  acc(set_all_modes<SJD_F32, 0>(bytes));
  acc(set_all_modes<SJD_F32, 1>(bytes));
  acc(set_all_modes<SJD_F32, 2>(bytes));
  acc(set_all_modes<SJD_F32, 3>(bytes));
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
      case 0: launch_t<SJD_BF16, 0>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 1: launch_t<SJD_BF16, 1>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 2: launch_t<SJD_BF16, 2>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      default: launch_t<SJD_BF16, 3>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
    }
  } else {
    switch (p.fast_cpt) {
      case 0: launch_t<SJD_F32, 0>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 1: launch_t<SJD_F32, 1>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      case 2: launch_t<SJD_F32, 2>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
      default: launch_t<SJD_F32, 3>(p, mode, grid, cond, uncond, use_cfg, oc, on, of, s); break;
    }
  }
  return cudaGetLastError();
}

}  // namespace sjd
