// CUDA kernels of the SJD-PAC verify-and-draft step for sm_103a.
//
// One CTA processes one (batch, window-row) pair: it streams the row's
// cond/uncond logits over the allowed id range from HBM with 128-bit loads
// into shared memory (guidance and temperature applied on the way), finds
// the top-k and top-p cuts with histogram selects in shared memory,
// compacts the kept ids into a sparse row (written back as the next step's
// draft distribution), verifies the row's draft group (Sec. 3.2, Thm. 2),
// resamples from the residual on rejection, continues regardless of earlier
// rejections (adaptive continuation, Sec. 4.2) and draws the proactive
// drafting alternates (Sec. 4.1). The last CTA of each batch element (atomic
// ticket, no waiting) finds the first rejection, emits the committed tokens
// and, in the fused step, shifts and refills the window (Sec. 3.3, Alg. 1).
//
// Numerics: every value that decides an integer is formed with IEEE fp32
// operations rounded after each step (__fadd_rn / __fmul_rn / __fdiv_rn are
// never contracted; the definition's fused multiply-adds are explicit
// __fmaf_rn) and every normalising sum is an exact integer
// sum of weights quantised to units of 2^-47, so the result does not depend
// on thread count or reduction order.

#include <mutex>

#include <cuda_bf16.h>

#include "sjd_device.cuh"

namespace sjd {
namespace {

// Shared-memory views of the row kernel.

struct Cand {  // candidate of the threshold select
  uint32_t key;
  int id;
  unsigned long long w;
};

struct Smem {
  float* lv;                  // [nL] logits of ids al0.. (padding: kPad)
  unsigned long long* hist;   // [kBins] (uint32 view for counts); also Cand[kCandMax]
  int32_t* qid;               // [S] staged draft row
  float* qpr;
  int32_t* pid;               // [S] kept ids, ascending
  unsigned long long* pcum;   // [S] inclusive prefix of kept weights
  float* pp;                  // [S] p of kept ids
  float* qP;                  // [S] q at kept ids
  float* cur;                 // [S] p^(k) of the group levels
  unsigned long long* Rw;     // [S] residual weights
};

__device__ __forceinline__ Smem smem_views(const DevParams& P, unsigned char* base) {
  Smem s;
  s.lv = reinterpret_cast<float*>(base + P.off_lv);
  s.hist = reinterpret_cast<unsigned long long*>(base + P.off_hist);
  s.qid = reinterpret_cast<int32_t*>(base + P.off_qid);
  s.qpr = reinterpret_cast<float*>(base + P.off_qpr);
  s.pid = reinterpret_cast<int32_t*>(base + P.off_pid);
  s.pcum = reinterpret_cast<unsigned long long*>(base + P.off_pcum);
  s.pp = reinterpret_cast<float*>(base + P.off_pp);
  s.qP = reinterpret_cast<float*>(base + P.off_qP);
  s.cur = reinterpret_cast<float*>(base + P.off_cur);
  s.Rw = reinterpret_cast<unsigned long long*>(base + P.off_Rw);
  return s;
}

struct RowInfo {
  float m;       // largest logit
  float scale;   // bins per unit of (m - l) for the first select level
  Cut kcut;      // top-k cut
};

// Is element i of lv active for the select, and its weight.
template <bool WEIGHTED>
__device__ __forceinline__ bool sel_active(float l, uint32_t key, int id, const RowInfo& ri) {
  if (!WEIGHTED) return key > 1u;
  return key > 1u && in_cut(key, id, ri.kcut);
}
template <bool WEIGHTED>
__device__ __forceinline__ unsigned long long sel_weight(float l, const RowInfo& ri) {
  if (!WEIGHTED) return 1ull;
  return quant(exp_neg(__fsub_rn(l, ri.m)));
}

// First-level bin: linear in (m - l), monotone non-increasing in l.
__device__ __forceinline__ int bin0(float l, uint32_t key, const RowInfo& ri) {
  if (key <= kKeyNegInf) return kBins - 1;
  const float x = __fmul_rn(__fsub_rn(ri.m, l), ri.scale);
  return (x < static_cast<float>(kBins - 1)) ? static_cast<int>(x) : kBins - 1;
}

// The need-th (1-based) active element in id order with key == kt.
template <bool WEIGHTED>
__device__ int nth_tied_id(const Smem& sm, const DevParams& P, const RowInfo& ri, uint32_t kt,
                           unsigned long long need, Scratch& sc) {
  const int seg = ((P.nL + kWarps * 32 - 1) / (kWarps * 32)) * 32;
  const int w = warp_id(), lane = lane_id();
  const int beg = w * seg, end = min(P.nL, beg + seg);
  uint32_t cnt = 0;
  for (int i0 = beg; i0 < end; i0 += 32) {
    const int i = i0 + lane;
    bool hit = false;
    if (i < end) {
      const float l = sm.lv[i];
      const uint32_t key = f2key(l);
      hit = key == kt && sel_active<WEIGHTED>(l, key, P.al0 + i, ri);
    }
    cnt += __popc(__ballot_sync(0xFFFFFFFFu, hit));
  }
  if (lane == 0) sc.u32b[w] = cnt;
  __syncthreads();
  if (threadIdx.x < 32) {
    // warp 0 finds the segment and the element
    unsigned long long before = 0;
    int wsel = -1;
    for (int k = 0; k < kWarps; ++k) {
      if (before + sc.u32b[k] >= need) {
        wsel = k;
        break;
      }
      before += sc.u32b[k];
    }
    int found = INT_MAX;
    if (wsel >= 0) {
      const int b2 = wsel * seg, e2 = min(P.nL, b2 + seg);
      unsigned long long run = before;
      for (int i0 = b2; i0 < e2 && found == INT_MAX; i0 += 32) {
        const int i = i0 + lane;
        bool hit = false;
        if (i < e2) {
          const float l = sm.lv[i];
          const uint32_t key = f2key(l);
          hit = key == kt && sel_active<WEIGHTED>(l, key, P.al0 + i, ri);
        }
        const uint32_t bal = __ballot_sync(0xFFFFFFFFu, hit);
        const uint32_t n = __popc(bal);
        if (run + n >= need) {
          const int r = static_cast<int>(need - run);  // 1-based rank within this chunk
          const int pos = __fns(bal, 0, r);
          found = P.al0 + i0 + pos;
        }
        run += n;
      }
    }
    if (lane == 0) sc.bc_i[0] = found;
  }
  __syncthreads();
  const int r = sc.bc_i[0];
  __syncthreads();
  return r;
}

// Select the cut at which the running count (or weight) in the order
// (key desc, id asc) over the active elements first reaches `need`.
// Returns the cut and, through *through, the count/weight up to and
// including the cut element. `total` receives the active total (weighted).
template <bool WEIGHTED>
__device__ Cut select_cut(const Smem& sm, const DevParams& P, const RowInfo& ri,
                          unsigned long long need_in, Scratch& sc, unsigned long long* through,
                          unsigned long long* total_out, bool need_is_fraction_of_total) {
  uint32_t* h32 = reinterpret_cast<uint32_t*>(sm.hist);
  unsigned long long* h64 = sm.hist;
  Cand* cands = reinterpret_cast<Cand*>(sm.hist);
  unsigned long long need = need_in;
  unsigned long long before_all = 0;
  uint32_t klo = 0, khi = 0xFFFFFFFFu;
  int level = 0;
  for (int iter = 0; iter < 8; ++iter, ++level) {
    // --- histogram of the active elements in [klo, khi]
    const int sh = level == 0 ? 0 : max(0, 32 - __clz(khi - klo) - 11);
    for (int k = threadIdx.x; k < kBins; k += kThreads) {
      if (WEIGHTED) h64[k] = 0; else h32[k] = 0;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < P.nL; i += kThreads) {
      const float l = sm.lv[i];
      const uint32_t key = f2key(l);
      if (key < klo || key > khi) continue;
      if (!sel_active<WEIGHTED>(l, key, P.al0 + i, ri)) continue;
      const int bk = level == 0 ? bin0(l, key, ri) : static_cast<int>((khi - key) >> sh);
      if (WEIGHTED) {
        const unsigned long long w = sel_weight<WEIGHTED>(l, ri);
        if (w) atomicAdd(&h64[bk], w);
      } else {
        atomicAdd(&h32[bk], 1u);
      }
    }
    __syncthreads();
    // --- find the bin where the running total reaches need
    constexpr int kPer = kBins / kThreads;
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
    if (level == 0 && WEIGHTED && need_is_fraction_of_total) {
      // need was passed as the fraction numerator: need = ceil(tau * total)
      *total_out = tot;
      need = scale_ceil(tot, P.tau_mant, P.tau_shift);
    }
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
    // --- gather the elements of that bin
    if (threadIdx.x == 0) {
      sc.cand_count = 0;
      sc.cand_kmin = 0xFFFFFFFFu;
      sc.cand_kmax = 0;
    }
    __syncthreads();
    uint32_t kmn = 0xFFFFFFFFu, kmx = 0;
    for (int i = threadIdx.x; i < P.nL; i += kThreads) {
      const float l = sm.lv[i];
      const uint32_t key = f2key(l);
      bool hit = key >= klo && key <= khi && sel_active<WEIGHTED>(l, key, P.al0 + i, ri);
      if (hit) hit = (level == 0 ? bin0(l, key, ri) : static_cast<int>((khi - key) >> sh)) == bstar;
      if (!hit) continue;
      kmn = min(kmn, key);
      kmx = max(kmx, key);
      const uint32_t slot = atomicAdd(&sc.cand_count, 1u);
      if (slot < static_cast<uint32_t>(kCandMax)) {
        cands[slot].key = key;
        cands[slot].id = P.al0 + i;
        cands[slot].w = sel_weight<WEIGHTED>(l, ri);
      }
    }
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
    if (nc <= static_cast<uint32_t>(kCandMax)) {
      // --- resolve by ranking the candidates in (key desc, id asc)
      for (uint32_t c = threadIdx.x; c < nc; c += kThreads) {
        const Cand me = cands[c];
        uint32_t rank = 0;
        unsigned long long wsum = 0;
        for (uint32_t d = 0; d < nc; ++d) {
          const Cand o = cands[d];
          const bool better = o.key > me.key || (o.key == me.key && o.id < me.id);
          rank += better ? 1u : 0u;
          wsum += better ? o.w : 0ull;
        }
        bool pick;
        if (WEIGHTED) pick = wsum < need && need <= wsum + me.w;
        else pick = static_cast<unsigned long long>(rank) + 1 == need;
        if (pick) {
          sc.bc_u[0] = me.key;
          sc.bc_i[2] = me.id;
          sc.bc_u64[1] = before_all + (WEIGHTED ? wsum + me.w : rank + 1);
        }
      }
      __syncthreads();
      Cut c{sc.bc_u[0], sc.bc_i[2]};
      *through = sc.bc_u64[1];
      __syncthreads();
      return c;
    }
    klo = bkmin;
    khi = bkmax;
    if (klo == khi) {
      // --- all remaining candidates tie in value: resolve by id order
      unsigned long long nth = need;
      unsigned long long wt = 1;
      if (WEIGHTED) {
        wt = quant(exp_neg(__fsub_rn(key2f(klo), ri.m)));
        nth = (need + wt - 1) / wt;
      }
      const int id = nth_tied_id<WEIGHTED>(sm, P, ri, klo, nth, sc);
      *through = before_all + nth * wt;
      return Cut{klo, id};
    }
  }
  // Not reached: each integer level shrinks the key range by 2^11.
  *through = before_all;
  return Cut{khi, INT_MAX};
}

// ---------------------------------------------------------------------------
// The row kernel.

template <int DT, bool VEC, int MODE>
__global__ void __launch_bounds__(kThreads, 1)
row_kernel(DevParams P, const void* __restrict__ cond, const void* __restrict__ uncond,
           bool use_cfg, int32_t* out_committed, int32_t* out_ncommit, int32_t* out_firstrej) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  __shared__ Scratch sc;
  const Smem sm = smem_views(P, smem_raw);

  const int b = blockIdx.x / P.rows_b;
  const int jr = blockIdx.x - b * P.rows_b;  // logit row of the batch element
  const bool node_row = jr >= P.W;           // a tree node off the main path
  const int abs0 = P.abs_pos[b];
  const uint32_t t = P.step_t[b];
  const bool temp = P.temp != 1.0f;
  // A node row (node i >= 1 at depth nd) verifies the node's children, which
  // sit at window row nd, with that row's stored draft row and uniforms.
  int nd = 0, ni = 0;
  bool node_live = false;
  if (node_row) {
    int e = jr - P.W, kd = P.K;
    nd = 1;
    while (e >= kd - 1) {
      e -= kd - 1;
      kd *= P.K;
      ++nd;
    }
    ni = e + 1;
    int off = 0;  // slot of depth nd's first node
    for (int d = 1, k2 = P.K; d < nd; ++d, k2 *= P.K) off += k2;
    node_live = nd < P.tree_depth[b] && P.tree_tok[static_cast<size_t>(b) * P.tree_n + SJD_IDX(off + ni, P.tree_n)] >= 0;
  }
  const int j = node_row ? nd : jr;  // window row whose position, draft row and uniforms apply
  const int slot = (abs0 + j) % P.W;
  const size_t bs = static_cast<size_t>(b) * P.W + slot;
  const uint32_t pos = static_cast<uint32_t>(abs0 + j);

  // ---- S0: the row's draft group and stored draft distribution
  int g = 1;
  int cands[kMaxK];
  int qlen = -1;
  if (MODE != kModeFromLogits) {
    if (node_row) {
      // the node's children: depth nd + 1, slots i K .. i K + K - 1
      int off = 0;
      for (int d = 1, k2 = P.K; d <= nd; ++d, k2 *= P.K) off += k2;
      const int32_t* ch = P.tree_tok + static_cast<size_t>(b) * P.tree_n + SJD_IDX(off + ni * P.K + P.K - 1, P.tree_n) -
                          (P.K - 1);
      g = 0;
      for (int k = 0; k < kMaxK; ++k) {
        cands[k] = (node_live && k < P.K) ? ch[k] : -1;
        if (cands[k] >= 0 && g == k) ++g;
      }
    } else {
      g = min(max(P.gsize[bs], 1), P.K);
      for (int k = 0; k < kMaxK; ++k) cands[k] = k < g ? P.cand[bs * P.K + k] : -1;
    }
    qlen = min(P.q_len[bs], P.S);
    if (!node_row || node_live)
      for (int i = threadIdx.x; i < max(qlen, 0); i += kThreads) {
        sm.qid[i] = P.q_ids[bs * P.S + i];
        sm.qpr[i] = P.q_prob[bs * P.S + i];
      }
  }
  if (node_row && !node_live) {
    // no such node in this tree: the row only takes its ticket
    __syncthreads();
    if (threadIdx.x == 0) {
      __threadfence();
      const uint32_t done = atomicAdd(P.ticket + b, 1u);
      sc.bc_i[0] = done == static_cast<uint32_t>(P.rows_b - 1) ? 1 : 0;
    }
    __syncthreads();
    if (sc.bc_i[0]) {
      __threadfence();
      batch_epilogue_tree(P, b, out_committed, out_ncommit, out_firstrej, sc);
    }
    return;
  }

  // ---- S1/S2: stream the row, guidance + temperature, into shared memory
  // row start, shifted so that index v holds id v (the row layout's column 0 is id col0)
  const size_t row = static_cast<size_t>(blockIdx.x) * static_cast<size_t>(P.row_stride);
  const int c0 = P.col0;
  uint32_t kmax = 0;
  float fmin_finite = INFINITY;
  uint32_t bad = 0;
  auto put = [&](int i, float c, float u) {
    const int v = P.al0 + i;
    float l = pad_value();
    if (v >= P.lo && v < P.hi) {
      l = combine(c, u, P.cfg, use_cfg);
      if (temp) l = __fdiv_rn(l, P.temp);
      if (isnan(l) || l == INFINITY) {
        bad = 1;
        l = -INFINITY;
      }
      kmax = max(kmax, f2key(l));
      if (l != -INFINITY) fmin_finite = fminf(fmin_finite, l);
    }
    return l;
  };
  if (DT == SJD_BF16) {
    const __nv_bfloat16* cr = static_cast<const __nv_bfloat16*>(cond) + row;
    const __nv_bfloat16* ur = use_cfg ? static_cast<const __nv_bfloat16*>(uncond) + row : nullptr;
    if (VEC) {
      const int nch = P.nL >> 3;
      for (int c = threadIdx.x; c < nch; c += kThreads) {
        const uint4 cw = __ldcs(reinterpret_cast<const uint4*>(cr + (P.al0 - c0)) + c);
        uint4 uw = make_uint4(0, 0, 0, 0);
        if (use_cfg) uw = __ldcs(reinterpret_cast<const uint4*>(ur + (P.al0 - c0)) + c);
        const uint32_t cv[4] = {cw.x, cw.y, cw.z, cw.w};
        const uint32_t uv[4] = {uw.x, uw.y, uw.z, uw.w};
        float o[8];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          o[2 * e] = put(c * 8 + 2 * e, bf16_bits_to_f32(cv[e] & 0xFFFFu), bf16_bits_to_f32(uv[e] & 0xFFFFu));
          o[2 * e + 1] = put(c * 8 + 2 * e + 1, bf16_bits_to_f32(cv[e] >> 16), bf16_bits_to_f32(uv[e] >> 16));
        }
        float4* dst = reinterpret_cast<float4*>(sm.lv + c * 8);
        dst[0] = make_float4(o[0], o[1], o[2], o[3]);
        dst[1] = make_float4(o[4], o[5], o[6], o[7]);
      }
    } else {
      const uint16_t* c16 = reinterpret_cast<const uint16_t*>(cr);
      const uint16_t* u16 = reinterpret_cast<const uint16_t*>(ur);
      for (int i = threadIdx.x; i < P.nL; i += kThreads) {
        const int v = P.al0 + i;
        float l = pad_value();
        if (v >= P.lo && v < P.hi)
          l = put(i, bf16_bits_to_f32(c16[v - c0]), use_cfg ? bf16_bits_to_f32(u16[v - c0]) : 0.0f);
        sm.lv[i] = l;
      }
    }
  } else {
    const float* cr = static_cast<const float*>(cond) + row;
    const float* ur = use_cfg ? static_cast<const float*>(uncond) + row : nullptr;
    if (VEC) {
      const int nch = P.nL >> 2;
      for (int c = threadIdx.x; c < nch; c += kThreads) {
        const float4 cw = __ldcs(reinterpret_cast<const float4*>(cr + (P.al0 - c0)) + c);
        float4 uw = make_float4(0.f, 0.f, 0.f, 0.f);
        if (use_cfg) uw = __ldcs(reinterpret_cast<const float4*>(ur + (P.al0 - c0)) + c);
        float4 o;
        o.x = put(c * 4 + 0, cw.x, uw.x);
        o.y = put(c * 4 + 1, cw.y, uw.y);
        o.z = put(c * 4 + 2, cw.z, uw.z);
        o.w = put(c * 4 + 3, cw.w, uw.w);
        reinterpret_cast<float4*>(sm.lv)[c] = o;
      }
    } else {
      for (int i = threadIdx.x; i < P.nL; i += kThreads) {
        const int v = P.al0 + i;
        float l = pad_value();
        if (v >= P.lo && v < P.hi) l = put(i, cr[v - c0], use_cfg ? ur[v - c0] : 0.0f);
        sm.lv[i] = l;
      }
    }
  }
  kmax = block_max_u32(kmax, sc);
  const uint32_t kmin_f = block_min_u32(fmin_finite == INFINITY ? 0xFFFFFFFFu : f2key(fmin_finite), sc);
  bad = block_or_u32(bad, sc);
  if (bad && threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));

  RowInfo ri;
  ri.m = key2f(kmax);
  ri.kcut = no_cut();
  int n = 0;                    // kept ids
  unsigned long long Zk = 0;    // their total weight
  const bool empty = kmax <= kKeyNegInf;  // no finite logit
  if (empty) {
    if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));
  } else {
    {
      const float mn = kmin_f == 0xFFFFFFFFu ? ri.m : key2f(kmin_f);
      const float range = __fsub_rn(ri.m, mn);
      float scale = (range > 0.0f) ? __fdiv_rn(static_cast<float>(kBins), range) : 0.0f;
      if (!(scale <= 1e30f)) scale = 0.0f;
      ri.scale = scale;
    }
    // ---- S3: top-k cut (count select) and top-p cut (weighted select)
    unsigned long long through, dummy;
    if (P.topk < P.veff) ri.kcut = select_cut<false>(sm, P, ri, P.topk, sc, &through, &dummy, false);
    Cut pcut = no_cut();
    if (P.top_p < 1.0f) {
      unsigned long long tot;
      pcut = select_cut<true>(sm, P, ri, 0, sc, &through, &tot, true);
    }
    // ---- S4: compaction of the kept ids (ascending) with prefix weights;
    // a kept id's weight is its precise weight (sjd_device.cuh), from its
    // raw inputs read again
    auto kept_weight = [&](int v) -> unsigned long long {
      float c, u = 0.0f;
      const size_t e = row + static_cast<size_t>(v - P.col0);
      if (DT == SJD_BF16) {
        c = bf16_bits_to_f32(__ldg(static_cast<const unsigned short*>(cond) + e));
        if (use_cfg) u = bf16_bits_to_f32(__ldg(static_cast<const unsigned short*>(uncond) + e));
      } else {
        c = __ldg(static_cast<const float*>(cond) + e);
        if (use_cfg) u = __ldg(static_cast<const float*>(uncond) + e);
      }
      return precise_weight(c, u, use_cfg, P.cfg, temp, P.temp, ri.m);
    };
    const int seg = ((P.nL + kWarps * 32 - 1) / (kWarps * 32)) * 32;
    const int w = warp_id(), lane = lane_id();
    const int beg = w * seg, end = min(P.nL, beg + seg);
    uint32_t wc = 0;
    unsigned long long ws = 0;
    for (int i0 = beg; i0 < end; i0 += 32) {
      const int i = i0 + lane;
      bool keep = false;
      unsigned long long e = 0;
      if (i < end) {
        const float l = sm.lv[i];
        const uint32_t key = f2key(l);
        keep = key > 1u && in_cut(key, P.al0 + i, ri.kcut) && in_cut(key, P.al0 + i, pcut);
        if (keep) e = kept_weight(P.al0 + i);
        keep = e != 0;  // zero-weight ids have p = 0 and are not stored
      }
      wc += __popc(__ballot_sync(0xFFFFFFFFu, keep));
      ws += warp_sum_u64(e);
    }
    // one (count, sum) per warp, scanned across warps
    uint32_t cex, ctot;
    unsigned long long sex, stot;
    block_exscan_pair(lane == 0 ? wc : 0u, lane == 0 ? ws : 0ull, sc, &cex, &sex, &ctot, &stot);
    cex = __shfl_sync(0xFFFFFFFFu, cex, 0);
    sex = __shfl_sync(0xFFFFFFFFu, sex, 0);
    n = static_cast<int>(ctot);
    Zk = stot;
    if (n > P.S) {  // cannot happen when S >= min(k, V_eff) (checked on the host)
      if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_CAPACITY));
      n = P.S;
    }
    const float Wz = fix_to_f32(Zk);
    uint32_t run_c = cex;
    unsigned long long run_s = sex;
    for (int i0 = beg; i0 < end; i0 += 32) {
      const int i = i0 + lane;
      bool keep = false;
      unsigned long long e = 0;
      if (i < end) {
        const float l = sm.lv[i];
        const uint32_t key = f2key(l);
        keep = key > 1u && in_cut(key, P.al0 + i, ri.kcut) && in_cut(key, P.al0 + i, pcut);
        if (keep) e = kept_weight(P.al0 + i);
        keep = e != 0;
      }
      const uint32_t bal = __ballot_sync(0xFFFFFFFFu, keep);
      unsigned long long incl = e;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += y;
      }
      if (keep) {
        const int at = static_cast<int>(run_c + __popc(bal & ((1u << lane) - 1u)));
        if (at < P.S) {
          const float p = prob_of(e, Wz);
          sm.pid[at] = P.al0 + i;
          sm.pcum[at] = run_s + incl;
          sm.pp[at] = p;
        }
      }
      run_c += __popc(bal);
      run_s += __shfl_sync(0xFFFFFFFFu, incl, 31);
    }
    __syncthreads();
    // write the sparse row P^t into this position's slot (next step's q);
    // with the tree it is held apart until every row has read the old rows
    if (!node_row) {
      int32_t* qi = P.tree && MODE == kModeStep ? P.tq_ids : P.q_ids;
      float* qp = P.tree && MODE == kModeStep ? P.tq_prob : P.q_prob;
      for (int i = threadIdx.x; i < n; i += kThreads) {
        qi[bs * P.S + i] = sm.pid[i];
        qp[bs * P.S + i] = sm.pp[i];
      }
    }
  }
  if (threadIdx.x == 0 && !node_row) {
    (P.tree && MODE == kModeStep ? P.tq_len : P.q_len)[bs] = n;
    atomicAdd(&P.stats[0], 1ull);
    atomicAdd(&P.stats[1], static_cast<unsigned long long>(max(qlen, 0)));
    atomicAdd(&P.stats[2], static_cast<unsigned long long>(n));
  }

  if (MODE == kModeFromLogits) {
    if (threadIdx.x == 0) {
      int x = P.lo;
      if (n > 0) {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kSynth, 0));
        const int i = search_excluding(sm.pcum, n, scale_floor(Zk, odd), nullptr, nullptr, 0);
        x = sm.pid[SJD_IDX(i, n)];
      }
      P.cand[bs * P.K] = x;
      P.gsize[bs] = 1;
      P.win_tok[static_cast<size_t>(b) * P.W + j] = x;
    }
    return;
  }

  // ---- S5/S7: verify the draft group (Sec. 3.2, Thm. 2), residual resample
  int x = cands[0];
  int xidx = -1;  // index of x in the kept row (-1: not kept)
  if (n > 0) {
    // p and q at the candidates (every thread, from shared memory)
    int pidx[kMaxK];
    float qc[kMaxK];
    for (int k = 0; k < g; ++k) {
      pidx[k] = find_sorted(sm.pid, n, cands[k]);
      if (qlen < 0) qc[k] = (cands[k] >= P.lo && cands[k] < P.hi) ? P.uniform_q : 0.0f;
      else {
        const int qi = find_sorted(sm.qid, qlen, cands[k]);
        qc[k] = qi >= 0 ? sm.qpr[qi] : 0.0f;
      }
    }
    // p^(k) as integer weights: the kept weights (differences of sm.pcum) at
    // k = 1, then sm.Rw; the total is Wsum
    double S = 0.0;  // draft mass of the rejected candidates
    int removed[kMaxK];
    int nrem = 0;
    unsigned long long Wsum = Zk, Rsum = 0;
    bool accepted = false;
    bool have_qP = false;
    for (int k = 1; k <= g; ++k) {
      const double d = __dsub_rn(1.0, S);
      const float q_c = qc[k - 1];
      const int pi = pidx[k - 1];
      unsigned long long Wc = pi < 0 ? 0ull : (k == 1 ? weight_at(sm.pcum, pi) : sm.Rw[pi]);
      if (P.group_of) {  // the weight of the candidate's whole group (relaxed, lossy)
        const int gc = __ldg(P.group_of + cands[k - 1]);
        unsigned long long part = 0;
        for (int i = threadIdx.x; i < n; i += kThreads)
          if (__ldg(P.group_of + sm.pid[i]) == gc) part += k == 1 ? weight_at(sm.pcum, i) : sm.Rw[i];
        Wc = block_sum_u64(part, sc);
      }
      if (q_c == 0.0f && !P.group_of) {
        if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_INVALID_DRAFT));
      } else {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kAccept, k - 1));
        if (accept_exact(odd, q_c, Wsum, Wc, d)) {
          x = cands[k - 1];
          xidx = pidx[k - 1];
          accepted = true;
          break;
        }
      }
      // residual of level k: max(0, p^(k) - q^(k)) quantised
      if (!have_qP) {
        for (int i = threadIdx.x; i < n; i += kThreads) {
          float qv;
          if (qlen < 0) qv = P.uniform_q;
          else {
            const int qi = find_sorted(sm.qid, qlen, sm.pid[i]);
            qv = qi >= 0 ? sm.qpr[qi] : 0.0f;
          }
          sm.qP[i] = qv;
        }
        have_qP = true;
      }
      unsigned long long part = 0;
      if (k == 1) {
        for (int i = threadIdx.x; i < n; i += kThreads) {
          const unsigned long long R = residual_first(weight_at(sm.pcum, i), sm.qP[i], Wsum);
          sm.Rw[i] = R;
          part += R;
        }
        Rsum = block_sum_u64(part, sc);
        if (Rsum == 0) {  // only reachable through rounding: sample from p^(k)
          for (int i = threadIdx.x; i < n; i += kThreads) sm.Rw[i] = weight_at(sm.pcum, i);
          Rsum = Wsum;
        }
      } else {
        // the tokens of the rejected levels leave the draft's support; the
        // total first, so that W^(k) stays in sm.Rw if the residual is empty
        if (threadIdx.x == 0) level_scale(Wsum, d, &sc.bc_u64[2], &sc.bc_i[4]);
        __syncthreads();
        const unsigned long long A_fix = sc.bc_u64[2];
        const int G = sc.bc_i[4];
        for (int i = threadIdx.x; i < n; i += kThreads) {
          bool rem = false;
          for (int e = 0; e < nrem; ++e) rem |= removed[e] == i;
          part += rem ? sm.Rw[i] : residual_level(sm.Rw[i], sm.qP[i], A_fix, G);
        }
        Rsum = block_sum_u64(part, sc);
        if (Rsum == 0) {  // only reachable through rounding: sample from p^(k)
          Rsum = Wsum;
        } else {
          for (int i = threadIdx.x; i < n; i += kThreads) {
            bool rem = false;
            for (int e = 0; e < nrem; ++e) rem |= removed[e] == i;
            if (!rem) sm.Rw[i] = residual_level(sm.Rw[i], sm.qP[i], A_fix, G);
          }
        }
      }
      __syncthreads();
      if (k == g) break;
      S = __dadd_rn(S, f32_to_f64(qc[k - 1]));
      if (pidx[k - 1] >= 0) removed[nrem++] = pidx[k - 1];
      if (!(__dsub_rn(1.0, S) > 0.0)) break;
      Wsum = Rsum;
    }
    if (!accepted) {
      // inverse CDF over the residual weights in id order
      const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kResidual, 0));
      const unsigned long long T = scale_floor(Rsum, odd);
      const int per = (n + kThreads - 1) / kThreads;
      const int i0 = threadIdx.x * per, i1 = min(n, i0 + per);
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
      if (xidx >= 0) x = sm.pid[SJD_IDX(xidx, n)];
      __syncthreads();
    }
  }

  // ---- S8: proactive-drafting alternates and the vanilla-SJD tail draw
  if (node_row) {
    if (threadIdx.x == 0) P.res_node[static_cast<size_t>(b) * P.X + SJD_IDX(jr - P.W, P.X)] = x;
  } else if (threadIdx.x == 0) {
    if (P.tree && MODE == kModeStep) {
      // the next tree's groups off the main path, for whichever depth this
      // row takes in it: group i draws lanes i K .. i K + K - 1
      int32_t* tg = P.res_tree + bs * static_cast<size_t>(P.tree_g) * P.K;
      for (int gi = 1; gi <= P.tree_g; ++gi) {
        int32_t grp[kMaxK];
        const int nd2 = n > 0 ? draw_without_replacement(P, sm.pcum, [&](int i) { return sm.pid[i]; }, n, Zk, -1, pos,
                                                         t, static_cast<uint32_t>(b), P.K, grp, kTree, gi * P.K)
                              : 0;
        for (int k = 0; k < P.K; ++k) tg[(gi - 1) * P.K + k] = k < nd2 ? grp[k] : -1;
      }
    }
    const int Km1 = P.K - 1;
    int32_t alts[kMaxK];
    int na = 0;
    if (n > 0 && Km1 > 0)
      na = draw_without_replacement(P, sm.pcum, [&](int i) { return sm.pid[i]; }, n, Zk, xidx, pos, t, static_cast<uint32_t>(b), Km1, alts);
    for (int k = 0; k < na; ++k) P.res_alt[bs * Km1 + k] = alts[k];
    P.res_altn[bs] = na;
    P.res_x[bs] = x;
    P.res_dev[bs] = x != cands[0] ? 1 : 0;
    if (!P.ac) {
      int xf = x, fidx = -1;
      if (n > 0) {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kResidual, 0));
        fidx = search_excluding(sm.pcum, n, scale_floor(Zk, odd), nullptr, nullptr, 0);
        xf = sm.pid[SJD_IDX(fidx, n)];
      }
      int naf = 0;
      if (n > 0 && Km1 > 0)
        naf = draw_without_replacement(P, sm.pcum, [&](int i) { return sm.pid[i]; }, n, Zk, fidx, pos, t, static_cast<uint32_t>(b), Km1, alts);
      for (int k = 0; k < naf; ++k) P.res_altf[bs * Km1 + k] = alts[k];
      P.res_altfn[bs] = naf;
      P.res_xf[bs] = xf;
    }
  }

  // ---- last CTA of the batch element: S6 (+ S9 in the fused step)
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const uint32_t done = atomicAdd(P.ticket + b, 1u);
    sc.bc_i[0] = done == static_cast<uint32_t>(P.rows_b - 1) ? 1 : 0;
  }
  __syncthreads();
  if (sc.bc_i[0]) {
    __threadfence();
    // the row's logits (and everything aliased over them) are dead here
    if (P.tree && MODE == kModeStep)
      batch_epilogue_tree(P, b, out_committed, out_ncommit, out_firstrej, sc);
    else
      batch_epilogue_staged(P, b, MODE == kModeStep, out_committed, out_ncommit, out_firstrej, sc,
                            reinterpret_cast<int32_t*>(smem_raw + P.off_lv), static_cast<size_t>(P.nL));
  }
}

// ---------------------------------------------------------------------------
// Small kernels.

__global__ void init_kernel(DevParams P) {
  const int b = blockIdx.x;
  const int abs0 = P.abs_pos[b];
  const uint32_t t = P.step_t[b];
  if (P.tree && threadIdx.x == 0) P.tree_depth[b] = 0;
  for (int r = threadIdx.x; r < P.W; r += blockDim.x) {
    const int slot = (abs0 + r) % P.W;
    const size_t bs = static_cast<size_t>(b) * P.W + slot;
    const uint64_t r64 = rand64(P, static_cast<uint32_t>(abs0 + r), t, static_cast<uint32_t>(b), kInit);
    const int x = P.lo + static_cast<int>(__umul64hi(r64, static_cast<unsigned long long>(P.veff)));
    P.cand[bs * P.K] = x;
    P.gsize[bs] = 1;
    P.q_len[bs] = -1;
    P.win_tok[static_cast<size_t>(b) * P.W + r] = x;
  }
}

__global__ void refresh_kernel(DevParams P) {
  __shared__ Scratch sc;
  const int b = blockIdx.x;
  batch_refresh(P, b, P.first_rej[b], P.n_commit[b], sc);
}

__global__ void get_window_kernel(DevParams P, int32_t* tokens, int32_t* cands, int32_t* group,
                                  int32_t* abs_pos, int32_t* prev) {
  const int b = blockIdx.x;
  const int abs0 = P.abs_pos[b];
  for (int r = threadIdx.x; r < P.W; r += blockDim.x) {
    const size_t bs = static_cast<size_t>(b) * P.W + (abs0 + r) % P.W;
    const size_t o = static_cast<size_t>(b) * P.W + r;
    const int g = P.gsize[bs];
    tokens[o] = P.cand[bs * P.K];
    if (group) group[o] = g;
    if (cands)
      for (int k = 0; k < P.K; ++k) cands[o * P.K + k] = k < g ? P.cand[bs * P.K + k] : -1;
  }
  if (threadIdx.x == 0) {
    if (abs_pos) abs_pos[b] = abs0;
    if (prev) prev[b] = P.last_tok[b];
  }
}

__global__ void get_rows_kernel(DevParams P, int32_t* ids, float* probs, int32_t* len) {
  const int b = blockIdx.x / P.W;
  const int r = blockIdx.x - b * P.W;
  const size_t bs = static_cast<size_t>(b) * P.W + (P.abs_pos[b] + r) % P.W;
  const size_t o = static_cast<size_t>(b) * P.W + r;
  const int n = P.q_len[bs];
  if (threadIdx.x == 0) len[o] = n;
  for (int i = threadIdx.x; i < P.S; i += blockDim.x) {
    ids[o * P.S + i] = i < n ? P.q_ids[bs * P.S + i] : -1;
    probs[o * P.S + i] = i < n ? P.q_prob[bs * P.S + i] : 0.0f;
  }
}

// Append the committed tokens of the last step to the output grid.
__global__ void append_kernel(DevParams P, const int32_t* abs_before, int32_t n_tokens,
                              int32_t* grid, int32_t* accept_len_row) {
  const int b = blockIdx.x;
  const int base = abs_before[b];
  const int nc = P.n_commit[b];
  const int take = max(0, min(nc, n_tokens - base));
  for (int i = threadIdx.x; i < take; i += blockDim.x)
    grid[static_cast<size_t>(b) * n_tokens + base + i] = P.committed[static_cast<size_t>(b) * P.W + i];
  if (threadIdx.x == 0 && accept_len_row) accept_len_row[b] = take;
}

// The dynamic shared-memory limit of a kernel is a setting of the whole
// process (per device): contexts of different configurations only ever
// raise it, one at a time.
std::mutex g_smem_attr_mutex;

template <int DT, bool VEC, int MODE>
cudaError_t raise_smem_one(int bytes) {
  cudaFuncAttributes a;
  cudaError_t e = cudaFuncGetAttributes(&a, row_kernel<DT, VEC, MODE>);
  if (e != cudaSuccess || a.maxDynamicSharedSizeBytes >= bytes) return e;
  return cudaFuncSetAttribute(row_kernel<DT, VEC, MODE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              bytes);
}

template <int DT, bool VEC>
cudaError_t launch_row_t(const DevParams& p, int mode, const void* cond, const void* uncond,
                         bool use_cfg, int32_t* oc, int32_t* on, int32_t* of, cudaStream_t s) {
  const dim3 grid(p.B * p.rows_b), block(kThreads);
  switch (mode) {
    case kModeVerify:
      row_kernel<DT, VEC, kModeVerify><<<grid, block, p.smem_bytes, s>>>(p, cond, uncond, use_cfg, oc, on, of);
      break;
    case kModeStep:
      row_kernel<DT, VEC, kModeStep><<<grid, block, p.smem_bytes, s>>>(p, cond, uncond, use_cfg, oc, on, of);
      break;
    default:
      row_kernel<DT, VEC, kModeFromLogits><<<grid, block, p.smem_bytes, s>>>(p, cond, uncond, use_cfg, oc, on, of);
      break;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t raise_row_kernel_smem_all(int bytes) {
  std::lock_guard<std::mutex> lock(g_smem_attr_mutex);
  cudaError_t e = cudaSuccess;
  auto acc = [&](cudaError_t x) { if (e == cudaSuccess) e = x; };
  acc(raise_smem_one<SJD_F32, true, kModeVerify>(bytes));
  acc(raise_smem_one<SJD_F32, true, kModeStep>(bytes));
  acc(raise_smem_one<SJD_F32, true, kModeFromLogits>(bytes));
  acc(raise_smem_one<SJD_F32, false, kModeVerify>(bytes));
  acc(raise_smem_one<SJD_F32, false, kModeStep>(bytes));
  acc(raise_smem_one<SJD_F32, false, kModeFromLogits>(bytes));
  acc(raise_smem_one<SJD_BF16, true, kModeVerify>(bytes));
  acc(raise_smem_one<SJD_BF16, true, kModeStep>(bytes));
  acc(raise_smem_one<SJD_BF16, true, kModeFromLogits>(bytes));
  acc(raise_smem_one<SJD_BF16, false, kModeVerify>(bytes));
  acc(raise_smem_one<SJD_BF16, false, kModeStep>(bytes));
  acc(raise_smem_one<SJD_BF16, false, kModeFromLogits>(bytes));
  return e;
}

cudaError_t raise_row_kernel_smem(int bytes) {
  std::lock_guard<std::mutex> lock(g_smem_attr_mutex);
  cudaError_t e = cudaSuccess;
  auto acc = [&](cudaError_t x) { if (e == cudaSuccess) e = x; };
  acc(raise_smem_one<SJD_F32, true, kModeStep>(bytes));
  acc(raise_smem_one<SJD_F32, false, kModeStep>(bytes));
  acc(raise_smem_one<SJD_BF16, true, kModeStep>(bytes));
  acc(raise_smem_one<SJD_BF16, false, kModeStep>(bytes));
  return e;
}

cudaError_t launch_row(const DevParams& p, int mode, int dtype, bool vec, const void* cond,
                       const void* uncond, bool use_cfg, int32_t* oc, int32_t* on, int32_t* of,
                       cudaStream_t s) {
  if (dtype == SJD_BF16)
    return vec ? launch_row_t<SJD_BF16, true>(p, mode, cond, uncond, use_cfg, oc, on, of, s)
               : launch_row_t<SJD_BF16, false>(p, mode, cond, uncond, use_cfg, oc, on, of, s);
  return vec ? launch_row_t<SJD_F32, true>(p, mode, cond, uncond, use_cfg, oc, on, of, s)
             : launch_row_t<SJD_F32, false>(p, mode, cond, uncond, use_cfg, oc, on, of, s);
}

cudaError_t launch_init(const DevParams& p, cudaStream_t s) {
  init_kernel<<<p.B, 256, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_refresh(const DevParams& p, cudaStream_t s) {
  refresh_kernel<<<p.B, kThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_get_window(const DevParams& p, int32_t* tokens, int32_t* cands, int32_t* group,
                              int32_t* abs_pos, int32_t* prev, cudaStream_t s) {
  get_window_kernel<<<p.B, 256, 0, s>>>(p, tokens, cands, group, abs_pos, prev);
  return cudaGetLastError();
}

cudaError_t launch_get_rows(const DevParams& p, int32_t* ids, float* probs, int32_t* len,
                            cudaStream_t s) {
  get_rows_kernel<<<p.B * p.W, 256, 0, s>>>(p, ids, probs, len);
  return cudaGetLastError();
}

cudaError_t launch_append(const DevParams& p, const int32_t* abs_before, int32_t n_tokens,
                          int32_t* grid, int32_t* accept_len_row, cudaStream_t s) {
  append_kernel<<<p.B, 256, 0, s>>>(p, abs_before, n_tokens, grid, accept_len_row);
  return cudaGetLastError();
}

}  // namespace sjd
