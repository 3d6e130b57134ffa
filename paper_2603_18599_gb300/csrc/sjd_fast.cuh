#pragma once

// Streaming fast path of the SJD-PAC verify-and-draft step for sm_103a
// (the kernel templates; sjd_fast_part.cu instantiates them).
//
// One CTA per (batch, window-row) pair: 128 threads and about 32 KB of
// shared memory, so seven CTAs share an SM and every row of a 1024-row step
// is in flight at once (or 512 threads, one CTA per SM, when the step has at
// most two rows per SM). Each row is read once from HBM, with 128-bit
// streaming loads two pairs of rounds ahead of the arithmetic:
//
//  1. guidance in fp32 as the definition has it (fl(c - u), then one fused
//     multiply-add), temperature, the allowed-range mask;
//  2. a shared running maximum (atomicMax on order-preserving keys; a stale
//     value is never above the final maximum m) filters candidates on the
//     fly: ids with l - m_running > -34 go to a dense shared-memory list
//     (continued in the workspace). exp(-34) 2^47 < 0.5, so every other id
//     has weight 0. The first pair of rounds, a sample of the row, also gives
//     a conservative bound of the k-th largest logit that keeps the list
//     short, checked once the row is in (and the row streamed again without
//     it when it excluded too much);
//  3. weights E = rint(2^47 EXP(t)) of the listed candidates (two at a time
//     on packed fp32 pairs) and their exact total; members with t > -9 also
//     go to a small head buffer. A top-k cut
//     (more than k candidates) comes from the 16-bit counts of the weights
//     below 1024 when it lies there, else from 128 bins over t and an exact
//     ranking inside the bin that holds it, else from an exact select;
//  4. top-p cut: from the head, ranked one entry per thread, when its mass
//     reaches the target; otherwise a weighted select over all members;
//  5. kept ids in id order, verification, residual resampling and the
//     proactive-drafting draws (one warp for up to 32 kept ids, the block
//     otherwise; decisions and fp64 operations by one thread), and the
//     per-batch epilogue shared with the general kernel.
//
// Steps 1-4 read the step's logits alone: with the caller's early-logits
// guarantee they run while the previous step finishes (programmatic
// dependent launch), and only step 5 waits for it.
//
// Results are bit-identical to the general kernel (sjd_kernels.cu), which
// handles the configurations this path does not cover.


#include <cuda_bf16.h>

#include "sjd_device.cuh"

namespace sjd {
namespace {

// Wait for the grids this one depends on (programmatic dependent launch);
// returns at once when they are complete.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

constexpr int kMaxWarps = 16;           // scratch sized for up to 512 threads per CTA
__device__ __forceinline__ int nthr() { return static_cast<int>(blockDim.x); }
__device__ __forceinline__ int nwarp() { return static_cast<int>(blockDim.x >> 5); }
constexpr int NB = kFastBins;           // select bins
constexpr int CMAX = NB / 2;            // select candidates (16 bytes each) in the histogram space
constexpr int HCAP = 128;               // head buffer
constexpr int QREG = 2;                 // draft-row entries prefetched per thread
constexpr float kTCut = -34.0f;         // t <= -34 => weight 0
constexpr float kTHead = -9.0f;         // head: t > -9
constexpr float kTHead2 = -6.0f;        // rebuilt head (too many ids above -9)
constexpr float kBinScale = static_cast<float>(NB) / 34.0f;

// ---------------------------------------------------------------------------
// Per-CTA scratch and block-wide operations (one warp combines the per-warp
// partials; results are broadcast through shared memory).

struct FScratch {
  unsigned long long red[kMaxWarps];
  unsigned long long red2[kMaxWarps];
  unsigned long long bc64[8];
  int bi[24];             // [17]: G of a later group level
  float bf[4];
  uint32_t mkey;          // running maximum (order-preserving key)
  uint32_t list_count;    // candidates appended (may exceed the capacity)
  uint32_t head_count;
  unsigned long long head_mass;
  uint32_t cand_count, cand_kmin, cand_kmax;
  uint32_t rnd[5][4];     // Philox blocks of the row: ACCEPT lanes 0-3 / 4-7, RESIDUAL, PD 0-3 / 4-7
  float lbound;           // lower bound estimate of the k-th largest logit (-inf: none)
  float cut_est;          // estimate of the k-th largest logit, a bin's upper edge (+inf: none)
  int cands[kMaxK];       // draft group of the row
  int gpidx[kMaxK];       // its positions in the kept row (-1: absent)
  float gqc[kMaxK];       // q at the group's tokens
  int alts[kMaxK];        // proactive-drafting draws (thread 0)
  int excl[kMaxK];        // positions excluded from a draw and their weights (thread 0)
  unsigned long long exw[kMaxK];
};

__device__ __forceinline__ int lane() { return threadIdx.x & 31; }
__device__ __forceinline__ int warp() { return threadIdx.x >> 5; }

__device__ __forceinline__ unsigned long long wsum64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

__device__ unsigned long long fsum(unsigned long long v, FScratch& s) {
  v = wsum64(v);
  if (lane() == 0) s.red[warp()] = v;
  __syncthreads();
  if (warp() == 0) {
    unsigned long long x = lane() < nwarp() ? s.red[lane()] : 0ull;
#pragma unroll
    for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
    if (lane() == 0) s.bc64[7] = x;
  }
  __syncthreads();
  return s.bc64[7];
}

// Block sums of two u64 per thread (one pair of barriers).
__device__ void fsum2(unsigned long long a, unsigned long long b, FScratch& s, unsigned long long* ra,
                      unsigned long long* rb) {
  a = wsum64(a);
  b = wsum64(b);
  if (lane() == 0) {
    s.red[warp()] = a;
    s.red2[warp()] = b;
  }
  __syncthreads();
  if (warp() == 0) {
    unsigned long long x = lane() < nwarp() ? s.red[lane()] : 0ull;
    unsigned long long y = lane() < nwarp() ? s.red2[lane()] : 0ull;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      x += __shfl_xor_sync(0xFFFFFFFFu, x, o);
      y += __shfl_xor_sync(0xFFFFFFFFu, y, o);
    }
    if (lane() == 0) {
      s.bc64[5] = x;
      s.bc64[6] = y;
    }
  }
  __syncthreads();
  *ra = s.bc64[5];
  *rb = s.bc64[6];
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
    const int nw = nwarp();
    const unsigned long long w = lane() < nw ? s.red[lane()] : 0ull;
    unsigned long long x = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, x, o);
      if (lane() >= o) x += y;
    }
    if (lane() < nw) s.red2[lane()] = x - w;
    if (lane() == nw - 1) s.bc64[4] = x;
  }
  __syncthreads();
  *total = s.bc64[4];
  return s.red2[warp()] + incl - v;
}

// ---------------------------------------------------------------------------
// Shared-memory views and the kept-row arrays.

struct KeptArrays {           // kept row (capacity S) and its verification arrays
  uint16_t* pidx;             // local index (id - al0), ascending
  unsigned long long* pcum;   // inclusive prefix of the weights
  float* pp;                  // p (weights as fp32 before normalising)
  float* qP;                  // q at the kept ids
  float* cur;                 // p^(k) of the group levels
  unsigned long long* Rw;     // residual weights
};

struct FSmem {
  uint2* list;                // candidates: {logit bits, local index}; the general kept pass
                              // replaces the logit by the kept weight (fp32) or -1
  unsigned long long* hist;   // histogram / select candidates / word prefix counts
  unsigned long long* head;   // head buffer: HCAP x {key, idx, E} (16 bytes)
  uint32_t* bitmap;           // one bit per local index
  int32_t* qs_ids;            // staged draft row (up to f_qcap entries)
  float* qs_pr;
  KeptArrays small;           // kept arrays in shared memory (capacity f_kcap)
};

__device__ __forceinline__ FSmem fsmem_views(const DevParams& P, unsigned char* base) {
  FSmem s;
  s.list = reinterpret_cast<uint2*>(base + P.f_list_l);
  s.hist = reinterpret_cast<unsigned long long*>(base + P.f_hist);
  s.head = reinterpret_cast<unsigned long long*>(base + P.f_list_w);
  s.bitmap = reinterpret_cast<uint32_t*>(base + P.f_bitmap);
  s.qs_ids = reinterpret_cast<int32_t*>(base + P.f_stage);
  s.qs_pr = reinterpret_cast<float*>(base + P.f_stage + 4 * P.f_qcap);
  s.small.pidx = reinterpret_cast<uint16_t*>(base + P.f_pidx);
  s.small.pcum = reinterpret_cast<unsigned long long*>(base + P.f_pcum);
  s.small.pp = reinterpret_cast<float*>(base + P.f_pp);
  s.small.qP = reinterpret_cast<float*>(base + P.f_qP);
  s.small.cur = reinterpret_cast<float*>(base + P.f_cur);
  s.small.Rw = reinterpret_cast<unsigned long long*>(base + P.f_Rw);
  return s;
}

// Kept arrays of row `row` in the workspace (for kept rows above f_kcap).
__device__ __forceinline__ KeptArrays global_kept(const DevParams& P, int row) {
  unsigned char* base = reinterpret_cast<unsigned char*>(P.f_scratch) + static_cast<size_t>(row) * P.f_row_bytes;
  const size_t S = static_cast<size_t>(P.S);
  KeptArrays k;
  k.pcum = reinterpret_cast<unsigned long long*>(base);
  k.Rw = reinterpret_cast<unsigned long long*>(base + 8 * S);
  k.pp = reinterpret_cast<float*>(base + 16 * S);
  k.qP = reinterpret_cast<float*>(base + 20 * S);
  k.cur = reinterpret_cast<float*>(base + 24 * S);
  k.pidx = reinterpret_cast<uint16_t*>(base + 28 * S);
  return k;
}

struct FCand {
  uint32_t key;
  int idx;
  unsigned long long w;
};

// First-level bin over t in (-34, 0]: linear in -t, monotone in l.
__device__ __forceinline__ int fbin0(float t) {
  const float x = __fmul_rn(-t, kBinScale);
  return (x < static_cast<float>(NB - 1)) ? static_cast<int>(x) : NB - 1;
}

// Weight of a member: E = rint(2^47 exp(t)) (the exponential of the shared
// exp_neg definition) and E 2^-47 as fp32, without conversion instructions.
// rint(a) for |a| <= 64 is fl(a + 1.5 2^23) - 1.5 2^23 (the sum lies in a
// binade of spacing 1, so the addition rounds to an integer, ties to even),
// and its integer value is the difference of the bit patterns. For
// y >= 2^-24, y 2^47 is an integer and E is y's significand shifted; below,
// fl(y + 2^-24) rounds y to the grid 2^-47 (ties to even on the significand,
// whose last bit is E's), E is the difference of the bit patterns and
// E 2^-47 = fl(y + 2^-24) - 2^-24 exactly (Sterbenz). Both identities hold
// for every input float (checked exhaustively against rintf and against the
// integer rounding of quant()/dequant()).
__device__ __forceinline__ float exp_weight(float t, unsigned long long* E) {
  const float a = __fmul_rn(t, 0x1.715476p+0f);  // fl32(log2 e)
  if (!(a >= -64.0f)) {
    *E = 0ull;
    return 0.0f;
  }
  const float r = __fadd_rn(a, 0x1.8p23f);
  const float n = __fsub_rn(r, 0x1.8p23f);
  const int ni = static_cast<int>(__float_as_uint(r) - __float_as_uint(0x1.8p23f));
  const float f = __fsub_rn(a, n);
  float y = 0x1.ffcbfcp-17f;
  y = __fmaf_rn(y, f, 0x1.430912p-13f);
  y = __fmaf_rn(y, f, 0x1.5d87fep-10f);
  y = __fmaf_rn(y, f, 0x1.3b2ab6p-7f);
  y = __fmaf_rn(y, f, 0x1.c6b08ep-5f);
  y = __fmaf_rn(y, f, 0x1.ebfbe0p-3f);
  y = __fmaf_rn(y, f, 0x1.62e430p-1f);
  y = __fmaf_rn(y, f, 1.0f);
  y = __fmul_rn(y, __int_as_float((ni + 127) << 23));
  const uint32_t b = __float_as_uint(y);
  if (y >= 0x1p-24f) {
    *E = static_cast<unsigned long long>((b & 0x7FFFFFu) | 0x800000u) << ((b >> 23) - 103u);
    return y;
  }
  const float sg = __fadd_rn(y, 0x1p-24f);
  *E = static_cast<unsigned long long>(__float_as_uint(sg) - __float_as_uint(0x1p-24f));
  return __fsub_rn(sg, 0x1p-24f);
}

// The weights E0, E1 of two members at once: the operations of exp_weight
// (same roundings, element by element), with the additions, subtractions and
// the Horner steps on packed pairs and no branches. The product t log2 e stays
// a scalar multiply (a packed multiply followed by a packed add might be
// contracted); y 2^n is exact, so its product needs no such care. Below
// a = -64 the weight is 0, as in exp_weight.
__device__ __forceinline__ void exp_weight2(float t0, float t1, unsigned long long* E0, unsigned long long* E1) {
  const float a0 = __fmul_rn(t0, 0x1.715476p+0f), a1 = __fmul_rn(t1, 0x1.715476p+0f);
  [[maybe_unused]] float n0, n1, f0, f1;
  float r0, r1, y0, y1;
  asm("{\n\t.reg .b64 a2, c2, r2, n2, f2, y2, k2;\n\t"
      "mov.b64 a2, {%8, %9};\n\t"
      "mov.b64 c2, {%10, %10};\n\t"
      "add.rn.f32x2 r2, a2, c2;\n\t"
      "sub.rn.f32x2 n2, r2, c2;\n\t"
      "sub.rn.f32x2 f2, a2, n2;\n\t"
      "mov.b64 y2, {%11, %11};\n\t"
      "mov.b64 k2, {%12, %12};\n\t"
      "fma.rn.f32x2 y2, y2, f2, k2;\n\t"
      "mov.b64 k2, {%13, %13};\n\t"
      "fma.rn.f32x2 y2, y2, f2, k2;\n\t"
      "mov.b64 k2, {%14, %14};\n\t"
      "fma.rn.f32x2 y2, y2, f2, k2;\n\t"
      "mov.b64 k2, {%15, %15};\n\t"
      "fma.rn.f32x2 y2, y2, f2, k2;\n\t"
      "mov.b64 k2, {%16, %16};\n\t"
      "fma.rn.f32x2 y2, y2, f2, k2;\n\t"
      "mov.b64 k2, {%17, %17};\n\t"
      "fma.rn.f32x2 y2, y2, f2, k2;\n\t"
      "mov.b64 k2, {%18, %18};\n\t"
      "fma.rn.f32x2 y2, y2, f2, k2;\n\t"
      "mov.b64 {%0, %1}, r2;\n\t"
      "mov.b64 {%2, %3}, n2;\n\t"
      "mov.b64 {%4, %5}, f2;\n\t"
      "mov.b64 {%6, %7}, y2;\n\t}"
      : "=f"(r0), "=f"(r1), "=f"(n0), "=f"(n1), "=f"(f0), "=f"(f1), "=f"(y0), "=f"(y1)
      : "f"(a0), "f"(a1), "f"(0x1.8p23f), "f"(0x1.ffcbfcp-17f), "f"(0x1.430912p-13f), "f"(0x1.5d87fep-10f),
        "f"(0x1.3b2ab6p-7f), "f"(0x1.c6b08ep-5f), "f"(0x1.ebfbe0p-3f), "f"(0x1.62e430p-1f), "f"(1.0f));
  const int ni0 = static_cast<int>(__float_as_uint(r0) - __float_as_uint(0x1.8p23f));
  const int ni1 = static_cast<int>(__float_as_uint(r1) - __float_as_uint(0x1.8p23f));
  y0 = __fmul_rn(y0, __int_as_float((ni0 + 127) << 23));
  y1 = __fmul_rn(y1, __int_as_float((ni1 + 127) << 23));
  auto quantize = [](float y, float a) -> unsigned long long {
    const uint32_t b = __float_as_uint(y);
    const int sh = static_cast<int>(b >> 23) - 103;
    const unsigned long long big = static_cast<unsigned long long>((b & 0x7FFFFFu) | 0x800000u) << max(sh, 0);
    const unsigned long long small =
        static_cast<unsigned long long>(__float_as_uint(__fadd_rn(y, 0x1p-24f)) - __float_as_uint(0x1p-24f));
    const unsigned long long e = y >= 0x1p-24f ? big : small;
    return a >= -64.0f ? e : 0ull;
  };
  *E0 = quantize(y0, a0);
  *E1 = quantize(y1, a1);
}

// Bins of the top-k cut search: t in (-34, 0], linear in -t, monotone in l.
constexpr int kTBins = 128;
__device__ __forceinline__ int tbin(float t) {
  const int b = __float2int_rz(__fmul_rn(-t, static_cast<float>(kTBins) / 34.0f));
  return min(b, kTBins - 1);
}

// Index of the need-th set bit (1-based) of the bitmap (nwords words).
__device__ int nth_set_bit(const uint32_t* bitmap, int nwords, unsigned long long need, FScratch& s) {
  const int per = (nwords + nthr() - 1) / nthr();
  const int w0 = min(nwords, static_cast<int>(threadIdx.x) * per), w1 = min(nwords, w0 + per);
  unsigned long long c = 0;
  for (int w = w0; w < w1; ++w) c += __popc(bitmap[w]);
  if (threadIdx.x == 0) s.bi[5] = INT_MAX;
  unsigned long long total;
  unsigned long long run = fexscan(c, s, &total);
  if (run < need && need <= run + c) {
    for (int w = w0; w < w1; ++w) {
      const uint32_t word = bitmap[w];
      const unsigned long long pc = __popc(word);
      if (run + pc >= need) {
        s.bi[5] = w * 32 + __fns(word, 0, static_cast<int>(need - run));
        break;
      }
      run += pc;
    }
  }
  __syncthreads();
  const int r = s.bi[5];
  __syncthreads();
  return r;
}

// Select the cut at which the running count (or weight) of the active
// elements, in the order (key desc, local index asc), first reaches `need`.
// src.each(f) calls f(key, idx, t, w) for this thread's active elements.
template <bool WEIGHTED, class Src>
__device__ Cut fast_select(const Src& src, float m, unsigned long long need_in, const FSmem& sm, int nwords,
                           FScratch& s) {
  uint32_t* h32 = reinterpret_cast<uint32_t*>(sm.hist);
  unsigned long long* h64 = sm.hist;
  FCand* cands = reinterpret_cast<FCand*>(sm.hist);
  unsigned long long need = need_in;
  uint32_t klo = 0, khi = 0xFFFFFFFFu;
  for (int level = 0; level < 8; ++level) {
    const int sh = level == 0 ? 0 : max(0, 32 - __clz(khi - klo) - 8);
    for (int k = threadIdx.x; k < NB; k += nthr()) {
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
    // thread t owns bins [t kPer, t kPer + kPer) (kPer = 2 for 128 threads, 1 for more)
    const int kPer = nthr() >= NB ? 1 : NB / nthr();
    unsigned long long loc[2];
    unsigned long long lsum = 0;
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const int k = threadIdx.x * kPer + q;
      loc[q] = (q < kPer && k < NB) ? (WEIGHTED ? h64[k] : h32[k]) : 0ull;
      lsum += loc[q];
    }
    if (threadIdx.x == 0) {
      s.bi[1] = -1;
      s.bc64[0] = 0;
    }
    unsigned long long tot;
    const unsigned long long ex = fexscan(lsum, s, &tot);
    if (ex < need && need <= ex + lsum) {
      unsigned long long run = ex;
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        if (q < kPer && run < need && need <= run + loc[q]) {
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
      if (slot < static_cast<uint32_t>(CMAX)) {
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
    if (nc <= static_cast<uint32_t>(CMAX)) {
      for (uint32_t c = threadIdx.x; c < nc; c += nthr()) {
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
      for (int k = threadIdx.x; k < nwords; k += nthr()) sm.bitmap[k] = 0u;
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

// ---------------------------------------------------------------------------
// Streaming loads.

template <int DT>
struct Chunk {  // one 16-byte chunk of cond and of uncond
  uint4 c, u;
};

template <int DT>
__device__ __forceinline__ Chunk<DT> load_chunk(const uint4* cr, const uint4* ur, bool use_cfg, int c, int nch) {
  Chunk<DT> k;
  k.c = make_uint4(0u, 0u, 0u, 0u);
  k.u = make_uint4(0u, 0u, 0u, 0u);
  if (c < nch) {
    k.c = __ldcs(cr + c);
    if (use_cfg) k.u = __ldcs(ur + c);
  }
  return k;
}

// Scalars of the logit arithmetic, held in registers for the streaming loops.
struct RowArith {
  float cfg, temp;
  int lo, hi, al0;
  bool use_cfg, use_temp;
};

__device__ __forceinline__ RowArith row_arith(const DevParams& P, bool use_cfg) {
  return RowArith{P.cfg, P.temp, P.lo, P.hi, P.al0, use_cfg, P.temp != 1.0f};
}

__device__ __forceinline__ float max_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Logits of one chunk (EPC values; ids outside the allowed range get the
// padding value) and their NaN-propagating maximum (-inf if none).
template <int DT>
__device__ __forceinline__ void chunk_logits(const RowArith& A, const Chunk<DT>& k, int c, float* out, float* cmax) {
  constexpr int EPC = DT == SJD_BF16 ? 8 : 4;
  float cv[EPC], uv[EPC];
  if (DT == SJD_BF16) {
    const uint32_t cw[4] = {k.c.x, k.c.y, k.c.z, k.c.w};
    const uint32_t uw[4] = {k.u.x, k.u.y, k.u.z, k.u.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      cv[2 * q] = __uint_as_float(cw[q] << 16);
      cv[2 * q + 1] = __uint_as_float(cw[q] & 0xFFFF0000u);
      uv[2 * q] = __uint_as_float(uw[q] << 16);
      uv[2 * q + 1] = __uint_as_float(uw[q] & 0xFFFF0000u);
    }
  } else {
    cv[0] = __uint_as_float(k.c.x); cv[1] = __uint_as_float(k.c.y);
    cv[2] = __uint_as_float(k.c.z); cv[3] = __uint_as_float(k.c.w);
    uv[0] = __uint_as_float(k.u.x); uv[1] = __uint_as_float(k.u.y);
    uv[2] = __uint_as_float(k.u.z); uv[3] = __uint_as_float(k.u.w);
  }
  float x[EPC];
#pragma unroll
  for (int q = 0; q < EPC; ++q)  // guidance: fl(c - u), then one fused multiply-add s (c - u) + u
    x[q] = A.use_cfg ? __fmaf_rn(A.cfg, __fsub_rn(cv[q], uv[q]), uv[q]) : cv[q];
  if (A.use_temp) {
#pragma unroll
    for (int q = 0; q < EPC; ++q) x[q] = __fdiv_rn(x[q], A.temp);
  }
  const int v0 = A.al0 + c * EPC;
  if (v0 >= A.lo && v0 + EPC <= A.hi) {
#pragma unroll
    for (int q = 0; q < EPC; ++q) out[q] = x[q];
  } else {
#pragma unroll
    for (int q = 0; q < EPC; ++q) {
      const bool ok = v0 + q >= A.lo && v0 + q < A.hi;
      out[q] = ok ? x[q] : pad_value();
      x[q] = ok ? x[q] : -INFINITY;
    }
  }
  // pairwise maximum (NaN-propagating, so the order does not matter)
#pragma unroll
  for (int w = 1; w < EPC; w <<= 1)
#pragma unroll
    for (int q = 0; q + w < EPC; q += 2 * w) x[q] = max_nan(x[q], x[q + w]);
  *cmax = x[0];
}

// ---------------------------------------------------------------------------
// Element sources for the selects.

// Candidates (t > -34) of the whole row, read again (128-bit loads, mostly
// from L2) with the final maximum.
template <int DT>
struct GlobalRow {
  const DevParams* P;
  const uint4* cr;
  const uint4* ur;
  bool use_cfg;
  float m;
  template <class F>
  __device__ __forceinline__ void each(F f) const {
    constexpr int EPC = DT == SJD_BF16 ? 8 : 4;
    const int nch = P->nL / EPC;
    const RowArith A = row_arith(*P, use_cfg);
    for (int c = threadIdx.x; c < nch; c += nthr()) {
      Chunk<DT> k;
      k.c = __ldg(cr + c);
      k.u = use_cfg ? __ldg(ur + c) : make_uint4(0u, 0u, 0u, 0u);
      float lv[EPC], cm;
      chunk_logits<DT>(A, k, c, lv, &cm);
#pragma unroll
      for (int q = 0; q < EPC; ++q) {
        const float t = __fsub_rn(lv[q], m);
        if (t > kTCut) f(f2key(lv[q]), c * EPC + q, t, 0ull);
      }
    }
  }
};

// The candidate list: entries [0, lcap) in shared memory (logit, local
// index), the rest in the row's workspace scratch (8 bytes each; written and
// read by this CTA only, ordered by its barriers).
struct ListView {
  uint2* sh;
  uint2* g;
  int lcap;
  bool early;  // the grid may still overlap the previous one: wait before writing g
  __device__ __forceinline__ void get(int i, float& l, int& idx) const {
    const uint2 e = i < lcap ? sh[i] : g[i - lcap];
    l = __uint_as_float(e.x);
    idx = static_cast<int>(e.y);
  }
  __device__ __forceinline__ void put(int i, float l, int idx) const {
    const uint2 e = make_uint2(__float_as_uint(l), static_cast<uint32_t>(idx));
    if (i < lcap) {
      sh[i] = e;
    } else {
      // the previous step's CTA of this row may still read this scratch
      if (early) griddep_wait();
      g[i - lcap] = e;
    }
  }
  // the kept pass replaces an entry by (precise weight << 16) | local index
  __device__ __forceinline__ void put_weight(int i, unsigned long long E, int idx) const {
    const uint2 e = make_uint2(static_cast<uint32_t>(E << 16) | static_cast<uint32_t>(idx),
                               static_cast<uint32_t>(E >> 16));
    if (i < lcap) sh[i] = e;
    else g[i - lcap] = e;
  }
  __device__ __forceinline__ void get_weight(int i, unsigned long long& E, int& idx) const {
    const uint2 e = i < lcap ? sh[i] : g[i - lcap];
    idx = static_cast<int>(e.x & 0xFFFFu);
    E = (static_cast<unsigned long long>(e.y) << 16) | (e.x >> 16);
  }
};

// Precise weight (sjd_device.cuh) of the id at local index idx of the row,
// from its raw inputs read again (mostly from L2).
template <int DT>
__device__ __forceinline__ unsigned long long kept_weight(const uint4* cr, const uint4* ur, int idx,
                                                          const RowArith& A, float m) {
  float c, u = 0.0f;
  if (DT == SJD_BF16) {
    c = bf16_bits_to_f32(__ldg(reinterpret_cast<const unsigned short*>(cr) + idx));
    if (A.use_cfg) u = bf16_bits_to_f32(__ldg(reinterpret_cast<const unsigned short*>(ur) + idx));
  } else {
    c = __ldg(reinterpret_cast<const float*>(cr) + idx);
    if (A.use_cfg) u = __ldg(reinterpret_cast<const float*>(ur) + idx);
  }
  return precise_weight(c, u, A.use_cfg, A.cfg, A.use_temp, A.temp, m);
}

// Every list entry (the list of a stream pass that overflowed).
struct ListAll {
  ListView L;
  int n;
  float m;
  template <class F>
  __device__ __forceinline__ void each(F f) const {
    for (int i = threadIdx.x; i < n; i += nthr()) {
      float lv;
      int idx;
      L.get(i, lv, idx);
      f(f2key(lv), idx, __fsub_rn(lv, m), 0ull);
    }
  }
};

// Candidate list (entries with t > -34 under the final maximum).
struct ListCand {
  ListView L;
  int n;
  float m;
  template <class F>
  __device__ __forceinline__ void each(F f) const {
    for (int i = threadIdx.x; i < n; i += nthr()) {
      float lv;
      int idx;
      L.get(i, lv, idx);
      const float t = __fsub_rn(lv, m);
      if (t > kTCut) f(f2key(lv), idx, t, 0ull);
    }
  }
};

// Members of the candidate list (t > -34, inside the top-k cut) with their
// weights recomputed.
struct ListMembers {
  ListView L;
  int n;
  float m;
  Cut kcut;
  template <class F>
  __device__ __forceinline__ void each(F f) const {
    for (int i = threadIdx.x; i < n; i += nthr()) {
      float lv;
      int id;
      L.get(i, lv, id);
      const float t = __fsub_rn(lv, m);
      if (!(t > kTCut)) continue;
      const uint32_t key = f2key(lv);
      if (!in_cut(key, id, kcut)) continue;
      unsigned long long E;
      exp_weight(t, &E);
      f(key, id, t, E);
    }
  }
};

// ---------------------------------------------------------------------------
// The row kernel.

template <int DT, int MODE, bool CFG, int NT>
__global__ void __launch_bounds__(NT, NT == 128 ? 7 : 1)
stream_row_kernel(DevParams P, const void* __restrict__ cond, const void* __restrict__ uncond,
                  int32_t* out_committed, int32_t* out_ncommit, int32_t* out_firstrej) {
  constexpr bool use_cfg = CFG;  // guidance with an unconditional branch (compile time)
  constexpr int ST = NT;         // threads per CTA: 128 (many rows, 7 per SM) or 512 (few rows)
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __shared__ FScratch s;
  __shared__ Scratch esc;  // for the per-batch epilogue shared with the general kernel
  // Programmatic dependent launch: this grid may start while the previous
  // kernel of the stream drains, and the next launch may start as soon as
  // every CTA of this grid has begun. Everything below may depend on the
  // previous kernel (the window state of the previous step, or logits a
  // forward has just written), so the wait comes before the first global
  // read; when the caller guarantees that the logits were written before
  // that kernel started (P.early_logits), S1-S4 (which read the logits
  // alone) run at once, and the wait comes before the first read or write
  // of the decode state or of the row's workspace scratch.
  const bool early = P.early_logits != 0;
  if (!early) griddep_wait();
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const FSmem sm = fsmem_views(P, smem_raw);
  constexpr int EPC = DT == SJD_BF16 ? 8 : 4;
  const int row = blockIdx.x;
  const size_t rowoff = static_cast<size_t>(row) * static_cast<size_t>(P.row_stride);
  const int nch = P.nL / EPC;
  const int esz = DT == SJD_BF16 ? 2 : 4;
  const size_t first = rowoff + static_cast<size_t>(P.al0 - P.col0);  // element of id al0
  const uint4* cr = reinterpret_cast<const uint4*>(static_cast<const unsigned char*>(cond) + first * esz);
  const uint4* ur = use_cfg ? reinterpret_cast<const uint4*>(static_cast<const unsigned char*>(uncond) + first * esz)
                            : nullptr;
  // the window position and step go first; the stream's first two pairs of
  // rounds follow. What depends on the position (the draft group, the
  // stored draft row, the random words) is set up during the stream, so
  // that its dependent loads never hold up the first rounds.
  const int b = row / P.W;
  const int j = row - b * P.W;
  int abs0 = 0;      // the window position and step: state, read in row_setup
  uint32_t t = 0;
  Chunk<DT> a0 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x, nch);
  Chunk<DT> a1 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + ST, nch);
  Chunk<DT> b0, b1;  // the second pair is requested once the first is in (below)
  b0.c = b0.u = b1.c = b1.u = make_uint4(0u, 0u, 0u, 0u);
  const int nwords = (P.nL + 31) >> 5;
  const int lcap = P.f_lcap;

  // ---- row set-up: counters now; draft group, stored draft row and random
  // words once the first pair of rounds is in (row_setup), the draft row's
  // prefetch after the stream (stage_setup)
  int g = 1, qlen = -1;
  int slot = 0;
  size_t bs = 0;
  uint32_t pos = 0;
  if (threadIdx.x == 0) {
    s.mkey = 0u;
    s.lbound = -INFINITY;
    s.cut_est = INFINITY;
    s.list_count = 0u;
    s.head_count = 0u;
    s.head_mass = 0ull;
  }
  for (int k = threadIdx.x; k < NB; k += ST) reinterpret_cast<uint32_t*>(smem_raw + P.f_hist)[k] = 0u;
  bool row_set = false;
  auto row_setup = [&]() {
    row_set = true;
    abs0 = P.abs_pos[b];
    t = P.step_t[b];
    slot = (abs0 + j) % P.W;
    bs = static_cast<size_t>(b) * P.W + slot;
    pos = static_cast<uint32_t>(abs0 + j);
    if (MODE != kModeFromLogits) {
      g = min(max(P.gsize[bs], 1), P.K);
      qlen = min(P.q_len[bs], P.S);
    }
    if (threadIdx.x < 5 && MODE != kModeFromLogits) {
      const uint32_t purpose[5] = {kAccept, kAccept + 8u, kResidual, kPd, kPd + 8u};
      const uint4 r = philox4x32_10(make_uint4(pos, t, static_cast<uint32_t>(b), purpose[threadIdx.x]), P.seed_lo,
                                    P.seed_hi);
      s.rnd[threadIdx.x][0] = r.x;
      s.rnd[threadIdx.x][1] = r.y;
      s.rnd[threadIdx.x][2] = r.z;
      s.rnd[threadIdx.x][3] = r.w;
    }
  };
  const int32_t* qids_g = nullptr;
  const float* qpr_g = nullptr;
  bool qstaged = false, q_in_smem = false;
  int32_t qreg_id[QREG];
  float qreg_p[QREG];
  int cand_reg = 0;  // the row's draft-group candidate k (thread k < g), fetched with the row
  // the stored draft row, when short, is fetched into registers and staged
  // in shared memory (over the dead candidate list) for verification
  auto stage_setup = [&]() {
    if (MODE != kModeFromLogits && static_cast<int>(threadIdx.x) < g) cand_reg = P.cand[bs * P.K + threadIdx.x];
    qids_g = P.q_ids + bs * P.S;
    qpr_g = P.q_prob + bs * P.S;
    qstaged = qlen >= 0 && qlen <= QREG * ST;   // prefetched into registers
    q_in_smem = qlen >= 0 && qlen <= P.f_qcap;  // staged before verification
#pragma unroll
    for (int e = 0; e < QREG; ++e) {
      const int i = threadIdx.x + e * ST;
      qreg_id[e] = 0;
      qreg_p[e] = 0.0f;
      if (qstaged && i < qlen) {
        qreg_id[e] = __ldg(qids_g + i);
        qreg_p[e] = __ldg(qpr_g + i);
      }
    }
  };

  // ---- S1-S2 streaming pass: logits, running maximum, candidate list
  const int rounds = (nch + ST - 1) / ST;
  volatile uint32_t* mkey_v = &s.mkey;
  uint32_t bad = 0;
  float mfix = 0.0f;  // second pass: the final maximum
  // Listed values are >= lmin. The first pass sets it from the first pair of
  // rounds: a conservative estimate of the row's k-th largest logit (the
  // sample's rank k*ns/nL, plus a quarter and 16 for safety). The estimate is
  // checked once the row is streamed: when fewer than k candidates were
  // listed while it excluded some, the row is streamed again without it.
  float lmin = -INFINITY;
  float lmin_below = -INFINITY;  // the float below lmin
  uint32_t* hsamp = reinterpret_cast<uint32_t*>(sm.hist);  // [NB] sample histogram (first pass)
  const RowArith arith = row_arith(P, use_cfg);
  const ListView Lst{sm.list,
                     reinterpret_cast<uint2*>(P.f_scratch + static_cast<size_t>(row) * P.f_row_bytes + P.f_glist),
                     lcap, early};
  const int lmax = lcap + P.f_gcap;  // list capacity
  const uint32_t lanes_below = (1u << lane()) - 1u;
  // One pair of rounds (chunks c0 = threadIdx.x + r ST and c1 = c0 + ST).
  // First pass: publish the warp maximum and filter with the running
  // maximum (never above the final one). Second pass: filter with the final
  // maximum, so that exactly the candidates are listed.
  auto process = [&](const Chunk<DT>& ka, const Chunk<DT>& kb, int r, bool fixed) {
    float lv[2][EPC];
    float cm0 = -INFINITY, cm1 = -INFINITY;
    const int c0 = threadIdx.x + r * ST, c1 = c0 + ST;
    if (c1 < nch) {  // both chunks inside the row: every pair but the last
      chunk_logits<DT>(arith, ka, c0, lv[0], &cm0);
      chunk_logits<DT>(arith, kb, c1, lv[1], &cm1);
    } else {
      // A warp whose lanes all lie past the last full pair (after the first
      // pair): at most one chunk per lane, few lanes with one. Each thread
      // publishes its maximum and lists its candidates itself, without warp
      // collectives, so the last ragged chunks cost no full round.
      if (r > 0 && static_cast<int>(threadIdx.x & ~31u) + (r + 1) * ST >= nch) {
        if (c0 >= nch) return;
        float l1[EPC];
        chunk_logits<DT>(arith, ka, c0, l1, &cm0);
        float mt = mfix;
        if (!fixed) {
          float cm = cm0;
          if (cm != cm) {  // NaN in the allowed range: flag, then NaN acts as -inf
            bad = 1u;
            cm = -INFINITY;
#pragma unroll
            for (int q = 0; q < EPC; ++q)
              if (l1[q] == l1[q]) cm = fmaxf(cm, l1[q]);
          }
          const uint32_t k1 = f2key(cm);
          if (k1 > *mkey_v) atomicMax(&s.mkey, k1);
          mt = key2f(*mkey_v);
        }
        const float th = fmaxf(fabsf(mt) < 4.0e6f ? __fadd_rn(mt, -34.5f) : -INFINITY, lmin_below);
        uint32_t n1 = 0;
#pragma unroll
        for (int q = 0; q < EPC; ++q) n1 += l1[q] > th ? 1u : 0u;
        if (n1) {
          uint32_t at = atomicAdd(&s.list_count, n1);
#pragma unroll
          for (int q = 0; q < EPC; ++q)
            if (l1[q] > th) {
              if (at < static_cast<uint32_t>(lmax)) Lst.put(static_cast<int>(at), l1[q], c0 * EPC + q);
              ++at;
            }
        }
        return;
      }
#pragma unroll
      for (int q = 0; q < EPC; ++q) {
        lv[0][q] = pad_value();
        lv[1][q] = pad_value();
      }
      if (c0 < nch) chunk_logits<DT>(arith, ka, c0, lv[0], &cm0);
    }
    float mth = mfix;
    if (!fixed) {
      float cm = fmaxf(cm0, cm1);
      if (cm0 != cm0 || cm1 != cm1) {  // NaN in the allowed range (rare): flag, then NaN acts as -inf
        bad = 1u;
        cm = -INFINITY;
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int q = 0; q < EPC; ++q)
            if (lv[h][q] == lv[h][q]) cm = fmaxf(cm, lv[h][q]);
      }
      const uint32_t wk = __reduce_max_sync(0xFFFFFFFFu, f2key(cm));
      if (lane() == 0 && wk > *mkey_v) atomicMax(&s.mkey, wk);
      if (r == 0) {
        __syncthreads();  // the first pair of rounds sets a good threshold for everyone
        mth = key2f(*mkey_v);
        // histogram of the sample (this pair) over t in (-34, 0] below its maximum
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int q = 0; q < EPC; ++q) {
            const float tq = __fsub_rn(lv[h][q], mth);
            if (tq > kTCut) atomicAdd(&hsamp[fbin0(tq)], 1u);
          }
        __syncthreads();
        if (warp() == 0) {
          constexpr int PER = NB / 32;
          const uint32_t ns = static_cast<uint32_t>(min(P.nL, 2 * ST * EPC));
          uint32_t c = 0;
#pragma unroll
          for (int q = 0; q < PER; ++q) c += hsamp[lane() * PER + q];
          uint32_t ci = c;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, ci, o);
            if (lane() >= o) ci += y;
          }
          const uint32_t total = __shfl_sync(0xFFFFFFFFu, ci, 31);  // candidates in the sample
          // only rows whose sample projects more than 1.5 k candidates need the bound
          const bool want = static_cast<unsigned long long>(total) * static_cast<uint32_t>(P.nL) >
                            static_cast<unsigned long long>(ns) * static_cast<uint32_t>(P.topk + P.topk / 2);
          if (want) {
            // ranks in the sample (k ns <= 16384 x 8192 fits 32 bits)
            const uint32_t kp = (static_cast<uint32_t>(P.topk) * ns + static_cast<uint32_t>(P.nL) - 1u) /
                                static_cast<uint32_t>(P.nL);
            const uint32_t ks = kp + kp / 4 + 16;
            uint32_t ce = ci - c;
            if (ce < ks && ks <= ci) {
#pragma unroll
              for (int q = 0; q < PER; ++q) {
                const uint32_t nq = hsamp[lane() * PER + q];
                if (ce < ks && ks <= ce + nq)
                  s.lbound = __fadd_rn(mth, -static_cast<float>(lane() * PER + q + 1) * (34.0f / NB));
                ce += nq;
              }
            }
            ce = ci - c;
            if (ce < kp && kp <= ci) {  // the sample's rank k ns / nL: where the cut is expected
#pragma unroll
              for (int q = 0; q < PER; ++q) {
                const uint32_t nq = hsamp[lane() * PER + q];
                if (ce < kp && kp <= ce + nq)
                  s.cut_est = __fadd_rn(mth, -static_cast<float>(lane() * PER + q) * (34.0f / NB));
                ce += nq;
              }
            }
          }
        }
        __syncthreads();
        lmin = s.lbound;
        lmin_below = nextafterf(lmin, -INFINITY);
      } else {
        mth = key2f(*mkey_v);
      }
    }
    // One comparison lists every id that can have t > -34 under the final
    // maximum m >= mth: such an id has l > m - 34 - 2^-18 (fl(l - m) > -34),
    // while fl(mth - 34.5) <= mth - 34.25 for |mth| < 4e6. Listed ids are
    // tested exactly later. Values below lmin are not listed (l >= lmin is
    // l > the float below lmin); padding and NaN compare false.
    const float thr = fmaxf(fabsf(mth) < 4.0e6f ? __fadd_rn(mth, -34.5f) : -INFINITY, lmin_below);
    uint32_t cnt = 0;
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int q = 0; q < EPC; ++q) cnt += lv[h][q] > thr ? 1u : 0u;
    // append to the list: one reservation per warp, consecutive entries per lane
    uint32_t incl = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
      if (lane() >= o) incl += y;
    }
    const uint32_t wtotal = __shfl_sync(0xFFFFFFFFu, incl, 31);
    if (wtotal) {
      uint32_t base = 0;
      if (lane() == 31) base = atomicAdd(&s.list_count, wtotal);
      base = __shfl_sync(0xFFFFFFFFu, base, 31);
      uint32_t at = base + incl - cnt;
      if (base + wtotal <= static_cast<uint32_t>(lcap)) {
        // consecutive entries from this lane's slot: a predicated store and
        // pointer step per value
        uint2* dst = sm.list + at;
        const uint32_t i0 = static_cast<uint32_t>(c0 * EPC), i1 = static_cast<uint32_t>(c1 * EPC);
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int q = 0; q < EPC; ++q)
            if (lv[h][q] > thr) *dst++ = make_uint2(__float_as_uint(lv[h][q]), (h ? i1 : i0) + q);
      } else {
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int q = 0; q < EPC; ++q)
            if (lv[h][q] > thr) {
              if (at < static_cast<uint32_t>(lmax)) Lst.put(static_cast<int>(at), lv[h][q], ((h ? c1 : c0) * EPC) + q);
              ++at;
            }
      }
    }
  };
  uint32_t appended = 0;
  bool exact_list = false;  // second pass: the list holds every top-k member (and maybe more)
  bool tau_active = false;  // the estimate excluded candidates (the top-k cut lies well above -34)
  for (int pass = 0; pass < 2; ++pass) {
    const bool fixed = pass == 1;
    __syncthreads();  // counters initialised (first pass) or reset (second)
    // two pairs of rounds in flight: the next pair was issued one pair of
    // processing earlier, so taking it over does not wait on memory; one
    // copy of the processing keeps the hot code small
    if (fixed) {
      a0 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x, nch);
      a1 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + ST, nch);
      b0 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + 2 * ST, nch);
      b1 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + 3 * ST, nch);
    }
#pragma unroll 1
    for (int r = 0; r < rounds; r += 2) {
      if (r == 0 && !fixed) {
        // every row's first pair is requested at once; each row asks for its
        // second pair only when its first has arrived, so the first pairs
        // do not queue behind the second ones
        asm volatile("" ::"r"(a0.c.x), "r"(a0.u.x));
        b0 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + 2 * ST, nch);
        b1 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + 3 * ST, nch);
      }
      process(a0, a1, r, fixed);
      if (!row_set && !early) row_setup();
      a0 = b0;
      a1 = b1;
      b0 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + (r + 4) * ST, nch);
      b1 = load_chunk<DT>(cr, ur, use_cfg, threadIdx.x + (r + 5) * ST, nch);
    }
    __syncthreads();
    appended = s.list_count;
    if (fixed) {
      exact_list = true;
      break;
    }
    mfix = key2f(s.mkey);
    if (!(mfix < INFINITY) || s.mkey <= 0x007FFFFFu) break;
    tau_active = lmin > __fadd_rn(mfix, -(34.0f + fmaxf(1.0f, fabsf(mfix) * 0x1p-20f)));
    if (appended > static_cast<uint32_t>(lmax)) {
      // The list overflowed. Its k-th largest value is at most the row's
      // k-th largest, so streaming the row again (mostly from L2) and listing
      // only the candidates at or above it keeps every top-k member.
      const ListAll la{Lst, lmax, mfix};
      lmin = key2f(fast_select<false>(la, mfix, static_cast<unsigned long long>(P.topk), sm, nwords, s).key);
      lmin_below = nextafterf(lmin, -INFINITY);
    } else if (tau_active) {
      // The estimate may have excluded candidates: it holds when at least k
      // candidates (under the final maximum) are listed above it. With lmin
      // above fl(m - 33.5) (>= m - 33.625 for |m| < 4e6), every listed value
      // has fl(l - m) > -34: the listed entries are the candidates.
      if (lmin >= __fadd_rn(mfix, -33.5f) && fabsf(mfix) < 4.0e6f) {
        if (appended >= static_cast<uint32_t>(P.topk)) break;
      } else {
        uint32_t nc = 0;
        const ListCand lc0{Lst, static_cast<int>(appended), mfix};
        lc0.each([&](uint32_t, int, float, unsigned long long) { ++nc; });
        if (fsum(nc, s) >= static_cast<unsigned long long>(P.topk)) break;
      }
      lmin = -INFINITY;
      lmin_below = -INFINITY;
      tau_active = false;
    } else {
      break;
    }
    if (threadIdx.x == 0) {
      s.list_count = 0u;
      atomicAdd(P.stats + kStatsPaths, 1ull);  // this row is streamed a second time
    }
  }
  // with early logits, the cuts, the kept row and its exact weights (S3-S4)
  // depend on this step's logits alone and run before the wait too; the
  // decode state is set up once the previous step is complete (below)
  if (!early) {
    if (!row_set) row_setup();
    stage_setup();
  }
  if (bad) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));
  const float m = key2f(s.mkey);

  int n = 0;                  // kept ids
  unsigned long long Zk = 0;  // their total weight
  KeptArrays K = sm.small;   // aliases the candidate list: used once the list is dead
  bool short_row = false;     // at most 32 kept ids from the head: warp 0 finishes the row
  if (!(m < INFINITY) || s.mkey <= 0x007FFFFFu) {
    // +inf logit, or no finite logit at all
    if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_NONFINITE));
  } else {
    int nlist;
    Cut kcut = no_cut();
    bool kcut_known = true;   // false: the members are the candidates except some of weight e* > 0
    bool from_global = false;  // the list holds the members only (kcut taken over the row)
    bool head_stale = false;   // the head was built before a top-k cut above t = -9 was known
    if (appended <= static_cast<uint32_t>(lmax)) {
      // every candidate, or (second pass) every candidate at or above a
      // bound of the k-th largest: in both cases every top-k member
      nlist = static_cast<int>(appended);
    } else {
      // more top-k candidates than the list holds (massive ties): the top-k
      // cut is taken over the row (read again), then only the members are listed
      const GlobalRow<DT> gr{&P, cr, ur, use_cfg, m};
      kcut = fast_select<false>(gr, m, static_cast<unsigned long long>(P.topk), sm, nwords, s);
      if (threadIdx.x == 0) s.list_count = 0u;
      __syncthreads();
      gr.each([&](uint32_t key, int idx, float, unsigned long long) {
        if (!in_cut(key, idx, kcut)) return;
        const uint32_t at = atomicAdd(&s.list_count, 1u);
        if (at < static_cast<uint32_t>(lmax)) Lst.put(static_cast<int>(at), key2f(key), idx);
      });
      __syncthreads();
      if (s.list_count > static_cast<uint32_t>(lmax) && threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_CAPACITY));
      nlist = min(static_cast<int>(s.list_count), lmax);
      from_global = true;
      if (threadIdx.x == 0) atomicAdd(P.stats + kStatsPaths + 1, 1ull);
    }
    const ListCand lcn{Lst, nlist, m};
    // ---- S3-S4: weights of the listed candidates inside kcut, their count
    // and exact total, the head buffer (t > -9) and, when a top-k cut may
    // follow, the counts of the small weights E < ecap (one per value) and,
    // when the cut may lie above them, per-bin counts and weight totals over
    // t (128 bins) (the list keeps the logits)
    // per bin: count, and the totals of the low and high 24 bits of E
    // (32-bit counters: exact while a bin holds fewer than 256 entries)
    uint32_t* tb_cnt = reinterpret_cast<uint32_t*>(sm.hist);                // [128]
    uint32_t* tb_lo = tb_cnt + kTBins;                                      // [128]
    uint32_t* tb_hi = tb_lo + kTBins;                                       // [128]
    // counts of E = 0 .. ecap-1, 16 bits each (a row has at most 65535
    // candidates): after the t-bins (ecap 256), or over the whole histogram
    // space when no t-bins are kept (ecap 1024)
    uint32_t* hE = reinterpret_cast<uint32_t*>(sm.hist);
    int ecap = 1024;
    auto weights_pass = [&](bool with_hist, bool with_tbins, unsigned long long* cnt, unsigned long long* tot) {
      if (threadIdx.x == 0) {
        s.head_count = 0u;
        s.head_mass = 0ull;
      }
      if (with_tbins) {
        for (int k = threadIdx.x; k < kTBins; k += ST) {
          tb_cnt[k] = 0u;
          tb_lo[k] = 0u;
          tb_hi[k] = 0u;
        }
      }
      if (with_hist) {
        hE = with_tbins ? tb_hi + kTBins : reinterpret_cast<uint32_t*>(sm.hist);
        ecap = with_tbins ? 256 : 1024;
        for (int k = threadIdx.x; k < (ecap >> 1); k += ST) hE[k] = 0u;
      }
      __syncthreads();
      unsigned long long zpart = 0;
      uint32_t cpart = 0;
      const bool cut_on = kcut.key != no_cut().key || kcut.id != no_cut().id;
      // the bookkeeping of one entry with its weight E (valid: a list entry)
      auto book = [&](float lv, float tt, int idx, bool valid, unsigned long long E) {
        if (!valid || !(tt > kTCut)) return;
        if (cut_on && !in_cut(f2key(lv), idx, kcut)) return;
        zpart += E;
        ++cpart;
        if (with_hist) {
          if (E < static_cast<unsigned long long>(ecap))
            atomicAdd(&hE[E >> 1], 1u << ((static_cast<uint32_t>(E) & 1u) << 4));
          if (with_tbins) {
            const int tb = tbin(tt);
            atomicAdd(&tb_cnt[tb], 1u);
            atomicAdd(&tb_lo[tb], static_cast<uint32_t>(E) & 0xFFFFFFu);
            atomicAdd(&tb_hi[tb], static_cast<uint32_t>(E >> 24));
          }
        }
        if (tt > kTHead) {
          const uint32_t h = atomicAdd(&s.head_count, 1u);
          if (h < static_cast<uint32_t>(HCAP)) {
            sm.head[2 * h] = (static_cast<unsigned long long>(f2key(lv)) << 32) | static_cast<uint32_t>(idx);
            sm.head[2 * h + 1] = E;
            atomicAdd(&s.head_mass, E);
          }
        }
      };
      // shared-memory part, four entries per step (two packed pairs of
      // independent exponentials)
      const int ns = min(nlist, lcap);
      for (int i0 = threadIdx.x; i0 < ns; i0 += 4 * ST) {
        float lv[4], tt[4];
        int id[4];
        unsigned long long E[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int i = min(i0 + u * ST, ns - 1);
          const uint2 en = sm.list[i];
          lv[u] = __uint_as_float(en.x);
          id[u] = static_cast<int>(en.y);
          tt[u] = __fsub_rn(lv[u], m);
        }
        exp_weight2(tt[0], tt[1], &E[0], &E[1]);
        exp_weight2(tt[2], tt[3], &E[2], &E[3]);
#pragma unroll
        for (int u = 0; u < 4; ++u) book(lv[u], tt[u], id[u], i0 + u * ST < ns, E[u]);
      }
      for (int i = lcap + static_cast<int>(threadIdx.x); i < nlist; i += ST) {
        float lv;
        int idx;
        Lst.get(i, lv, idx);
        const float tt = __fsub_rn(lv, m);
        unsigned long long E;
        exp_weight(tt, &E);
        book(lv, tt, idx, true, E);
      }
      fsum2(cpart, zpart, s, cnt, tot);
    };
    const bool may_cut = !from_global && appended > static_cast<uint32_t>(P.topk);
    unsigned long long ncand, Z;
    // many listed candidates: the cut may lie above the counted weights,
    // unless the sample puts it well below weight 1024 (t < -25.64)
    const bool many = may_cut && (tau_active || exact_list || appended > static_cast<uint32_t>(P.topk) + 1024u) &&
                      !(__fsub_rn(s.cut_est, m) < -24.5f);
    weights_pass(may_cut, many, &ncand, &Z);
    if (may_cut && ncand > static_cast<unsigned long long>(P.topk)) {
      // The top-k cut drops the excl = ncand - k last listed candidates,
      // whose weights are the excl smallest (E is monotone in t).
      // (a) When they all lie below ecap, the counts give their exact total X:
      //     Z = Zcand - X, and the cut falls among the candidates of weight
      //     e*, the largest dropped one. With e* = 0 the cut changes nothing
      //     else (weight-0 ids are never kept); otherwise it is taken exactly
      //     once something depends on it.
      // (b) Otherwise the t-bin b* holding the k-th candidate is found from
      //     the bin counts; its candidates are ranked exactly, which gives
      //     the cut and, with the totals of the bins above, Z.
      const unsigned long long excl = ncand - static_cast<unsigned long long>(P.topk);
      const uint32_t kk = static_cast<uint32_t>(P.topk);
      if (threadIdx.x == 0) {
        s.bi[10] = -1;
        s.bi[11] = -1;
      }
      __syncthreads();
      if (warp() == 0) {
        // each lane takes vpl = ecap/32 consecutive weight values (two per
        // word); counts and weight totals fit 32 bits (at most 16384 x 1023)
        const int pw = ecap >> 6;
        const int vpl = 2 * pw;
        const uint32_t ex = static_cast<uint32_t>(excl);  // below the list capacity
        const uint4* h4 = reinterpret_cast<const uint4*>(hE + lane() * pw);
        uint32_t c = 0, w = 0;
        for (int q = 0; q < (pw >> 2); ++q) {
          const uint4 x4 = h4[q];
          const uint32_t xs[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
          for (int r2 = 0; r2 < 4; ++r2) {
            const uint32_t e0 = 2u * static_cast<uint32_t>(lane() * pw + 4 * q + r2);
            const uint32_t lo = xs[r2] & 0xFFFFu, hi = xs[r2] >> 16;
            c += lo + hi;
            w += (lo + hi) * e0 + hi;
          }
        }
        uint32_t ci = c, wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t yc = __shfl_up_sync(0xFFFFFFFFu, ci, o);
          const uint32_t yw = __shfl_up_sync(0xFFFFFFFFu, wi, o);
          if (lane() >= o) {
            ci += yc;
            wi += yw;
          }
        }
        // the lane whose values hold the excl-th smallest; then one value per
        // lane inside it: e*, the largest dropped weight, and X
        const uint32_t bal = __ballot_sync(0xFFFFFFFFu, ci - c < ex && ex <= ci);
        if (bal != 0u) {
          const int L = __ffs(bal) - 1;
          const uint32_t cL = __shfl_sync(0xFFFFFFFFu, ci - c, L);
          const uint32_t wL = __shfl_sync(0xFFFFFFFFu, wi - w, L);
          uint32_t n = 0, e = 0;
          if (lane() < vpl) {
            e = static_cast<uint32_t>(L * vpl + lane());
            n = (hE[e >> 1] >> ((e & 1u) << 4)) & 0xFFFFu;
          }
          uint32_t ni = n, nw = n * e;
#pragma unroll
          for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y1 = __shfl_up_sync(0xFFFFFFFFu, ni, o);
            const uint32_t y2 = __shfl_up_sync(0xFFFFFFFFu, nw, o);
            if (lane() >= o) {
              ni += y1;
              nw += y2;
            }
          }
          const uint32_t cb = cL + ni - n;
          if (lane() < vpl && cb < ex && ex <= cb + n) {
            s.bi[10] = static_cast<int>(e);
            s.bc64[2] = static_cast<unsigned long long>(wL + nw - n * e) + static_cast<unsigned long long>(ex - cb) * e;
          }
        }
      } else if (warp() == 1 && many) {
        // bins in order of decreasing t, four per lane
        uint32_t c4[kTBins / 32];
        unsigned long long w4[kTBins / 32];
        uint32_t c = 0;
        unsigned long long w = 0;
        bool crowded = false;
#pragma unroll
        for (int q = 0; q < kTBins / 32; ++q) {
          const int k = lane() * (kTBins / 32) + q;
          c4[q] = tb_cnt[k];
          w4[q] = (static_cast<unsigned long long>(tb_hi[k]) << 24) + tb_lo[k];
          crowded |= c4[q] >= 256u;
          c += c4[q];
          w += w4[q];
        }
        crowded = __any_sync(0xFFFFFFFFu, crowded);
        uint32_t ci = c;
        unsigned long long wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t yc = __shfl_up_sync(0xFFFFFFFFu, ci, o);
          const unsigned long long yw = __shfl_up_sync(0xFFFFFFFFu, wi, o);
          if (lane() >= o) {
            ci += yc;
            wi += yw;
          }
        }
        uint32_t ce = ci - c;
        unsigned long long we = wi - w;
        if (!crowded && ce < kk && kk <= ci) {
#pragma unroll
          for (int q = 0; q < kTBins / 32; ++q) {
            if (ce < kk && kk <= ce + c4[q]) {
              s.bi[11] = lane() * (kTBins / 32) + q;
              s.bi[12] = static_cast<int>(kk - ce);  // rank of the cut inside the bin (1-based)
              s.bc64[3] = we;                        // total weight of the bins above
            }
            ce += c4[q];
            we += w4[q];
          }
        }
      }
      __syncthreads();
      const int estar = s.bi[10];
      const int bstar = s.bi[11];
      if (estar >= 0) {
        Z -= s.bc64[2];
        kcut_known = estar == 0;
      } else if (bstar < 0) {
        // no bin counts: the exact select, then the weights again
        kcut = fast_select<false>(lcn, m, static_cast<unsigned long long>(P.topk), sm, nwords, s);
        weights_pass(false, false, &ncand, &Z);
      } else {
        // (b): rank the candidates of bin b* (one per thread)
        const uint32_t need = static_cast<uint32_t>(s.bi[12]);
        const unsigned long long above = s.bc64[3];
        FCand* cands = reinterpret_cast<FCand*>(sm.hist);
        if (threadIdx.x == 0) s.cand_count = 0u;
        __syncthreads();
        for (int i = threadIdx.x; i < nlist; i += ST) {
          float lv;
          int idx;
          Lst.get(i, lv, idx);
          const float tt = __fsub_rn(lv, m);
          if (!(tt > kTCut) || tbin(tt) != bstar) continue;
          // t rides in the weight field: only members of the cut need their weight
          const uint32_t at = atomicAdd(&s.cand_count, 1u);
          if (at < static_cast<uint32_t>(CMAX)) cands[at] = FCand{f2key(lv), idx, __float_as_uint(tt)};
        }
        __syncthreads();
        const uint32_t nc = s.cand_count;
        if (nc <= static_cast<uint32_t>(CMAX)) {
          unsigned long long incl = 0;
          if (threadIdx.x < nc) {
            const FCand me = cands[threadIdx.x];
            uint32_t rank = 0;
#pragma unroll 4
            for (uint32_t d = 0; d < nc; ++d) {
              const FCand o = cands[d];
              rank += (o.key > me.key || (o.key == me.key && o.idx < me.idx)) ? 1u : 0u;
            }
            if (rank < need) exp_weight(__uint_as_float(static_cast<uint32_t>(me.w)), &incl);
            if (rank + 1 == need) {
              s.bi[2] = static_cast<int>(me.key);
              s.bi[3] = me.idx;
            }
          }
          Z = above + fsum(incl, s);
          kcut = Cut{static_cast<uint32_t>(s.bi[2]), s.bi[3]};
          head_stale = bstar <= tbin(kTHead);
        } else {
          // a crowded bin: the exact select, then the weights again
          kcut = fast_select<false>(lcn, m, static_cast<unsigned long long>(P.topk), sm, nwords, s);
          weights_pass(false, false, &ncand, &Z);
        }
      }
    }
    auto need_kcut = [&]() {
      if (!kcut_known) {
        kcut = fast_select<false>(lcn, m, static_cast<unsigned long long>(P.topk), sm, nwords, s);
        kcut_known = true;
      }
    };
    // ---- top-p cut
    Cut pcut = no_cut();
    bool head_done = false;
    if (P.top_p < 1.0f) {
      const unsigned long long target = scale_ceil(Z, P.tau_mant, P.tau_shift);
      // rebuild the head: with the top-k cut, when that cut (found after the
      // head was built) reaches above t = -9; with t > -6 when more than HCAP
      // ids lie above -9. The top-p cut is taken from the head only when the
      // head's mass reaches the target, by a weighted select otherwise.
      auto rebuild_head = [&](float thr) {
        __syncthreads();
        if (threadIdx.x == 0) {
          s.head_count = 0u;
          s.head_mass = 0ull;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < nlist; i += ST) {
          float lv;
          int idx;
          Lst.get(i, lv, idx);
          const float tt = __fsub_rn(lv, m);
          if (!(tt > thr)) continue;
          const uint32_t key = f2key(lv);
          if (!in_cut(key, idx, kcut)) continue;
          unsigned long long E;
          exp_weight(tt, &E);
          const uint32_t h = atomicAdd(&s.head_count, 1u);
          if (h < static_cast<uint32_t>(HCAP)) {
            sm.head[2 * h] = (static_cast<unsigned long long>(key) << 32) | static_cast<uint32_t>(idx);
            sm.head[2 * h + 1] = E;
            atomicAdd(&s.head_mass, E);
          }
        }
        __syncthreads();
      };
      if (head_stale) rebuild_head(kTHead);
      if (s.head_count > static_cast<uint32_t>(HCAP)) rebuild_head(kTHead2);
      const uint32_t nh = s.head_count;
      if (nh <= static_cast<uint32_t>(HCAP) && s.head_mass >= target) {
        // the cut lies in the head: rank the head (key desc, index asc), one entry per thread
        for (uint32_t e = threadIdx.x; e < nh; e += ST) {
          const unsigned long long me = sm.head[2 * e];
          const unsigned long long mw = sm.head[2 * e + 1];
          const uint32_t mk = static_cast<uint32_t>(me >> 32);
          const int mi = static_cast<int>(me & 0xFFFFFFFFu);
          unsigned long long before = 0;
#pragma unroll 4
          for (uint32_t d = 0; d < nh; ++d) {
            const unsigned long long o = sm.head[2 * d];
            const uint32_t ok = static_cast<uint32_t>(o >> 32);
            const int oi = static_cast<int>(o & 0xFFFFFFFFu);
            if (ok > mk || (ok == mk && oi < mi)) before += sm.head[2 * d + 1];
          }
          if (before < target && target <= before + mw) {
            s.bi[8] = static_cast<int>(mk);
            s.bi[9] = mi;
          }
        }
        __syncthreads();
        pcut = Cut{static_cast<uint32_t>(s.bi[8]), s.bi[9]};
        head_done = true;
      }
      if (!head_done) {
        // the cut lies below the head: weighted select over every member
        need_kcut();
        const ListMembers mg{Lst, nlist, m, kcut};
        pcut = fast_select<true>(mg, m, target, sm, nwords, s);
      }
    } else {
      need_kcut();
    }
    // ---- S4: kept ids (members in the top-p cut with precise weight > 0) in
    // id order; K.pcum holds their precise weights until the prefix pass
    if (head_done) {
      // the kept ids are all in the head: their precise weights replace the
      // head's (0 outside the top-p cut), then one entry per thread takes its rank
      const uint32_t nh = s.head_count;
      for (uint32_t e = threadIdx.x; e < nh; e += ST) {
        const unsigned long long me = sm.head[2 * e];
        const int mi = static_cast<int>(me & 0xFFFFFFFFu);
        sm.head[2 * e + 1] =
            in_cut(static_cast<uint32_t>(me >> 32), mi, pcut) ? kept_weight<DT>(cr, ur, mi, arith, m) : 0ull;
      }
      __syncthreads();
      uint32_t nk = 0;
      for (uint32_t e = threadIdx.x; e < nh; e += ST) {
        const int mi = static_cast<int>(sm.head[2 * e] & 0xFFFFFFFFu);
        const unsigned long long mw = sm.head[2 * e + 1];
        if (mw == 0) continue;
        ++nk;
        int rank = 0;
#pragma unroll 4
        for (uint32_t d = 0; d < nh; ++d)
          if (sm.head[2 * d + 1] != 0 && static_cast<int>(sm.head[2 * d] & 0xFFFFFFFFu) < mi) ++rank;
        K.pidx[SJD_IDX(rank, P.f_kcap)] = static_cast<uint16_t>(mi);
        K.pcum[SJD_IDX(rank, P.f_kcap)] = mw;
      }
      n = static_cast<int>(fsum(nk, s));
    } else {
      // general: the list's logits become kept weights (-1 otherwise), then a
      // bitmap over the local indices, word prefix counts and ranks
      uint32_t* word_base = reinterpret_cast<uint32_t*>(sm.hist);
      for (int k = threadIdx.x; k < nwords; k += ST) sm.bitmap[k] = 0u;
      __syncthreads();
      for (int i = threadIdx.x; i < nlist; i += ST) {
        float lv;
        int idx;
        Lst.get(i, lv, idx);
        const float tt = __fsub_rn(lv, m);
        unsigned long long E = 0;
        if (tt > kTCut) {
          const uint32_t key = f2key(lv);
          if (in_cut(key, idx, kcut) && in_cut(key, idx, pcut)) {
            E = kept_weight<DT>(cr, ur, idx, arith, m);
            if (E) atomicOr(&sm.bitmap[idx >> 5], 1u << (idx & 31));
          }
        }
        Lst.put_weight(i, E, idx);
      }
      __syncthreads();
      {
        const int per = (nwords + ST - 1) / ST;
        const int w0 = min(nwords, static_cast<int>(threadIdx.x) * per), w1 = min(nwords, w0 + per);
        unsigned long long c = 0;
        for (int w = w0; w < w1; ++w) c += __popc(sm.bitmap[w]);
        unsigned long long tot;
        unsigned long long run = fexscan(c, s, &tot);
        for (int w = w0; w < w1; ++w) {
          word_base[w] = static_cast<uint32_t>(run);
          run += __popc(sm.bitmap[w]);
        }
        n = static_cast<int>(tot);
      }
      if (n > P.S) {
        if (threadIdx.x == 0) atomicOr(P.err, err_bit(SJD_ERR_CAPACITY));
        n = P.S;
      }
      // the kept arrays: in shared memory when the layout holds them apart
      // from the list, else in the row's workspace scratch
      const bool k_shared = P.f_kwide && n <= P.f_kcap;
      // the previous step's CTA of this row may still use the row's scratch
      if (early && !k_shared) griddep_wait();
      K = k_shared ? sm.small : global_kept(P, row);
      __syncthreads();
      for (int i = threadIdx.x; i < nlist; i += ST) {
        unsigned long long E;
        int idx;
        Lst.get_weight(i, E, idx);
        if (E == 0) continue;
        const uint32_t word = sm.bitmap[idx >> 5];
        const int r = static_cast<int>(word_base[idx >> 5] + __popc(word & ((1u << (idx & 31)) - 1u)));
        if (r < n) {
          K.pidx[r] = static_cast<uint16_t>(idx);
          K.pcum[r] = E;
        }
      }
      __syncthreads();
    }
    // inclusive prefix of the kept weights, then p = fl(fl(E) 2^-47 / Wz)
    // (a short kept row from the head does it in warp 0, with verification)
    short_row = head_done && MODE != kModeFromLogits && n <= 32;
    if (!short_row) {
      const int per = (n + ST - 1) / ST;
      const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
      unsigned long long loc = 0;
      for (int i = i0; i < i1; ++i) loc += K.pcum[i];
      unsigned long long tot;
      unsigned long long run = fexscan(loc, s, &tot);
      Zk = tot;
      if (threadIdx.x == 0) s.bf[0] = fix_to_f32(Zk);
      __syncthreads();
      const float Wz = s.bf[0];
      for (int i = i0; i < i1; ++i) {
        const unsigned long long E = K.pcum[i];
        run += E;
        K.pcum[i] = run;
        K.pp[i] = prob_of(E, Wz);
      }
    }
    __syncthreads();
  }
  auto id_of = [&](int i) { return P.al0 + static_cast<int>(K.pidx[SJD_IDX(i, n)]); };
  if (early) {
    griddep_wait();  // the previous step is complete: its state may be read
    row_setup();
    stage_setup();
  }

  if (MODE == kModeFromLogits) {
    for (int i = threadIdx.x; i < n; i += ST) {
      P.q_ids[bs * P.S + i] = id_of(i);
      P.q_prob[bs * P.S + i] = K.pp[i];
    }
    if (threadIdx.x == 0) {
      P.q_len[bs] = n;
      unsigned long long* st = P.stats + kStatsSpread + 3 * (row & (kStatsSlots - 1));
      atomicAdd(st + 0, 1ull);
      atomicAdd(st + 2, static_cast<unsigned long long>(n));
      int x = P.lo;
      if (n > 0) {
        const uint32_t odd = odd24(rand32(P, pos, t, static_cast<uint32_t>(b), kSynth, 0));
        x = id_of(search_excluding(K.pcum, n, scale_floor(Zk, odd), nullptr, nullptr, 0));
      }
      P.cand[bs * P.K] = x;
      P.gsize[bs] = 1;
      P.win_tok[static_cast<size_t>(b) * P.W + j] = x;
    }
    return;
  }

  // ---- S5/S7: verify the draft group (Sec. 3.2, Thm. 2), residual resample.
  // Thread 0 takes every decision (and every fp64 operation); all threads
  // share the per-element residual passes.
  if (static_cast<int>(threadIdx.x) < g) s.cands[threadIdx.x] = cand_reg;
  if (qstaged) {
#pragma unroll
    for (int e = 0; e < QREG; ++e) {
      const int i = threadIdx.x + e * ST;
      if (i < qlen) {
        sm.qs_ids[i] = qreg_id[e];
        sm.qs_pr[i] = qreg_p[e];
      }
    }
  } else if (q_in_smem) {
    for (int i = threadIdx.x; i < qlen; i += ST) {
      sm.qs_ids[i] = __ldg(qids_g + i);
      sm.qs_pr[i] = __ldg(qpr_g + i);
    }
  }
  __syncthreads();
  auto q_at = [&](int v, int from) -> float {
    if (qlen < 0) return (v >= P.lo && v < P.hi) ? P.uniform_q : 0.0f;
    int lo = from, hi = qlen;
    if (q_in_smem) {
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (sm.qs_ids[mid] < v) lo = mid + 1; else hi = mid;
      }
      return (lo < qlen && sm.qs_ids[lo] == v) ? sm.qs_pr[lo] : 0.0f;
    }
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (__ldg(qids_g + mid) < v) lo = mid + 1; else hi = mid;
    }
    return (lo < qlen && __ldg(qids_g + lo) == v) ? __ldg(qpr_g + lo) : 0.0f;
  };
  if (!short_row && static_cast<int>(threadIdx.x) < g) {
    // candidate k's kept position and draft probability, one thread each
    {
      const int k = static_cast<int>(threadIdx.x);
      const int c = s.cands[k];
      int pi = -1;
      const int lc = c - P.al0;
      if (n > 0 && lc >= 0 && lc < P.nL) {
        int lo = 0, hi = n;
        while (lo < hi) {
          const int mid = (lo + hi) >> 1;
          if (static_cast<int>(K.pidx[mid]) < lc) lo = mid + 1; else hi = mid;
        }
        pi = (lo < n && static_cast<int>(K.pidx[lo]) == lc) ? lo : -1;
      }
      s.gpidx[k] = pi;
      s.gqc[k] = q_at(c, 0);
    }
  }
  if (!short_row) __syncthreads();
  if (n > 0 && n <= 32) {
    // ---- a short kept row (the common case: top-p keeps a few ids): warp 0
    // verifies, resamples and draws with one kept position per lane and the
    // same operations as the block path below, without block barriers
    if (warp() == 0) {
      const int ln = lane();
      const bool mine = ln < n;
      if (short_row) {
        // inclusive prefix of the kept weights, p = fl(fl(E) 2^-47 / Wz)
        const unsigned long long w = mine ? K.pcum[ln] : 0ull;
        unsigned long long inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, inc, o);
          if (ln >= o) inc += y;
        }
        Zk = __shfl_sync(0xFFFFFFFFu, inc, 31);
        float Wz = 0.0f;
        if (ln == 0) Wz = fix_to_f32(Zk);
        Wz = __shfl_sync(0xFFFFFFFFu, Wz, 0);
        if (mine) {
          K.pcum[ln] = inc;
          K.pp[ln] = prob_of(w, Wz);
        }
        __syncwarp();
        // the draft group: candidates, their kept positions and q
        if (ln < g) {
          const int c = s.cands[ln];
          int pi = -1;
          const int lc = c - P.al0;
          if (lc >= 0 && lc < P.nL) {
            int lo = 0, hi = n;
            while (lo < hi) {
              const int mid = (lo + hi) >> 1;
              if (static_cast<int>(K.pidx[mid]) < lc) lo = mid + 1; else hi = mid;
            }
            pi = (lo < n && static_cast<int>(K.pidx[lo]) == lc) ? lo : -1;
          }
          s.cands[ln] = c;
          s.gpidx[ln] = pi;
          s.gqc[ln] = q_at(c, 0);
        }
        __syncwarp();
      }
      const int c1 = s.cands[0];
      int x = c1, xidx = -1;
      const unsigned long long pc = mine ? K.pcum[ln] : 0ull;
      const unsigned long long w = mine ? weight_at(K.pcum, ln) : 0ull;
      unsigned long long Wk = w, Wsum = Zk;  // p^(k) as integer weights (my position; total)
      float qP = 0.0f;
      bool have_qP = false, accepted = false;
      double S = 0.0;  // draft mass of the rejected candidates
      unsigned long long R = 0, Rsum = 0;
      const int grp = (P.group_of && mine) ? __ldg(P.group_of + id_of(ln)) : 0;  // relaxed test: my id's group
      for (int k = 1; k <= g; ++k) {
        const int pi = s.gpidx[k - 1];
        unsigned long long Wc = __shfl_sync(0xFFFFFFFFu, Wk, max(pi, 0) & 31);
        if (P.group_of) {  // the weight of the candidate's whole group (relaxed, lossy)
          const int gc = __ldg(P.group_of + s.cands[k - 1]);
          Wc = wsum64(mine && grp == gc ? Wk : 0ull);
        }
        const double d = __dsub_rn(1.0, S);
        int acc = 0;
        if (ln == 0) {
          const float q_c = s.gqc[k - 1];
          if (q_c == 0.0f && !P.group_of) {
            atomicOr(P.err, err_bit(SJD_ERR_INVALID_DRAFT));
          } else {
            acc = accept_exact(odd24(s.rnd[(k - 1) >> 2][(k - 1) & 3]), q_c, Wsum,
                               (pi >= 0 || P.group_of) ? Wc : 0ull, d) ? 1 : 0;
          }
        }
        if (__shfl_sync(0xFFFFFFFFu, acc, 0)) {
          x = s.cands[k - 1];
          xidx = pi;
          accepted = true;
          break;
        }
        if (!have_qP) {
          if (mine) qP = q_at(id_of(ln), 0);
          have_qP = true;
        }
        if (k == 1) {
          R = mine ? residual_first(Wk, qP, Wsum) : 0ull;
        } else {
          // the tokens of the rejected levels leave the draft's support
          unsigned long long A_fix = 0;
          int G = 0;
          if (ln == 0) level_scale(Wsum, d, &A_fix, &G);
          A_fix = __shfl_sync(0xFFFFFFFFu, A_fix, 0);
          G = __shfl_sync(0xFFFFFFFFu, G, 0);
          bool rem = false;
          for (int e = 0; e < k - 1; ++e) rem |= s.gpidx[e] == ln;
          R = mine ? (rem ? Wk : residual_level(Wk, qP, A_fix, G)) : 0ull;
        }
        Rsum = wsum64(R);
        if (Rsum == 0) {  // only reachable through rounding: sample from p^(k)
          R = Wk;
          Rsum = Wsum;
        }
        if (k == g) break;
        S = __dadd_rn(S, f32_to_f64(s.gqc[k - 1]));
        if (!(__dsub_rn(1.0, S) > 0.0)) break;
        Wk = R;
        Wsum = Rsum;
      }
      // inclusive prefix over the lanes (positions) of a u64
      auto lane_incl = [&](unsigned long long v) {
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, v, o);
          if (ln >= o) v += y;
        }
        return v;
      };
      // first position whose value exceeds T (the last one when none does)
      auto first_over = [&](unsigned long long v, unsigned long long T) {
        const uint32_t hit = __ballot_sync(0xFFFFFFFFu, mine && v > T);
        return hit ? __ffs(hit) - 1 : n - 1;
      };
      if (!accepted) {
        const unsigned long long T = scale_floor(Rsum, odd24(s.rnd[2][0]));
        const unsigned long long incl = lane_incl(R);  // every lane takes part in the shuffles
        const uint32_t hit = __ballot_sync(0xFFFFFFFFu, mine && incl > T);
        xidx = hit ? __ffs(hit) - 1 : -1;
        if (xidx >= 0) x = id_of(xidx);
      }
      // ---- S8: proactive-drafting alternates and the vanilla-SJD tail draw
      const int Km1 = P.K - 1;
      auto draw = [&](int first_idx, int32_t* out) {
        unsigned long long tot = Zk;
        uint32_t exmask = 0;  // excluded positions
        if (first_idx >= 0) {
          exmask = 1u << first_idx;
          tot -= __shfl_sync(0xFFFFFFFFu, w, first_idx);
        }
        int drawn = 0;
        for (int kk = 1; kk <= Km1; ++kk) {
          if (tot == 0) break;
          const unsigned long long T = scale_floor(tot, odd24(s.rnd[3 + (kk >> 2)][kk & 3]));
          // C'(i) = pcum[i] minus the weights of the excluded positions up to i
          const unsigned long long cx = pc - lane_incl(((exmask >> ln) & 1u) ? w : 0ull);
          const int i = first_over(cx, T);
          if (ln == 0) out[drawn] = id_of(i);
          ++drawn;
          exmask |= 1u << i;
          tot -= __shfl_sync(0xFFFFFFFFu, w, i);
        }
        return drawn;
      };
      const int na = Km1 > 0 ? draw(xidx, s.alts) : 0;
      __syncwarp();
      if (ln == 0) {
        for (int k = 0; k < na; ++k) P.res_alt[bs * Km1 + k] = s.alts[k];
        P.res_altn[bs] = na;
        P.res_x[bs] = x;
        P.res_dev[bs] = x != c1 ? 1 : 0;
      }
      if (!P.ac) {
        const int fidx = first_over(pc, scale_floor(Zk, odd24(s.rnd[2][0])));
        const int xf = id_of(fidx);
        __syncwarp();
        const int naf = Km1 > 0 ? draw(fidx, s.alts) : 0;
        __syncwarp();
        if (ln == 0) {
          for (int k = 0; k < naf; ++k) P.res_altf[bs * Km1 + k] = s.alts[k];
          P.res_altfn[bs] = naf;
          P.res_xf[bs] = xf;
        }
      }
      if (ln == 0) {
        P.q_len[bs] = n;
        unsigned long long* st = P.stats + kStatsSpread + 3 * (row & (kStatsSlots - 1));
        atomicAdd(st + 0, 1ull);
        atomicAdd(st + 1, static_cast<unsigned long long>(max(qlen, 0)));
        atomicAdd(st + 2, static_cast<unsigned long long>(n));
      }
    }
  } else {
  const int c1 = s.cands[0];
  int x = c1;
  int xidx = -1;
  if (n > 0) {
    // p^(k) as integer weights: the kept weights (differences of K.pcum) at
    // k = 1, then K.Rw; the total is Wsum
    unsigned long long Wsum = Zk, Rsum = 0;
    // draft mass of the rejected candidates and d = 1 - S, in thread 0 only
    // (fp64 runs at a small fraction of the fp32 rate; the other threads
    // learn of the loop's end through shared memory)
    double S = 0.0, d = 1.0;
    bool have_qP = false;
    bool accepted = false;
    for (int k = 1; k <= g; ++k) {
      if (threadIdx.x == 0) d = __dsub_rn(1.0, S);
      unsigned long long WG = 0;
      if (P.group_of) {  // the weight of the candidate's whole group (relaxed, lossy)
        const int gc = __ldg(P.group_of + s.cands[k - 1]);
        unsigned long long part = 0;
        for (int i = threadIdx.x; i < n; i += ST)
          if (__ldg(P.group_of + id_of(i)) == gc) part += k == 1 ? weight_at(K.pcum, i) : K.Rw[i];
        WG = fsum(part, s);
      }
      if (threadIdx.x == 0) {
        const float q_c = s.gqc[k - 1];
        const int pi = s.gpidx[k - 1];
        const unsigned long long Wc =
            P.group_of ? WG : (pi < 0 ? 0ull : (k == 1 ? weight_at(K.pcum, pi) : K.Rw[pi]));
        int acc = 0;
        if (q_c == 0.0f && !P.group_of) {
          atomicOr(P.err, err_bit(SJD_ERR_INVALID_DRAFT));
        } else {
          const uint32_t odd = odd24(s.rnd[(k - 1) >> 2][(k - 1) & 3]);
          acc = accept_exact(odd, q_c, Wsum, Wc, d) ? 1 : 0;
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
        // q at the kept ids: each thread merges its contiguous run of kept ids
        // (ascending) with the stored draft row (ascending): one search, then
        // a forward walk
        const int per = (n + ST - 1) / ST;
        const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
        if (qlen < 0) {
          for (int i = i0; i < i1; ++i) {
            const int v = id_of(i);
            K.qP[i] = (v >= P.lo && v < P.hi) ? P.uniform_q : 0.0f;
          }
        } else if (i0 < i1) {
          const int32_t* qi = q_in_smem ? sm.qs_ids : qids_g;
          const float* qp = q_in_smem ? sm.qs_pr : qpr_g;
          int lo = 0, hi = qlen;
          const int v0 = id_of(i0);
          while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (qi[mid] < v0) lo = mid + 1; else hi = mid;
          }
          for (int i = i0; i < i1; ++i) {
            const int v = id_of(i);
            while (lo < qlen && qi[lo] < v) ++lo;
            K.qP[i] = (lo < qlen && qi[lo] == v) ? qp[lo] : 0.0f;
          }
        }
        __syncthreads();
        have_qP = true;
      }
      unsigned long long part = 0;
      if (k == 1) {
        for (int i = threadIdx.x; i < n; i += ST) {
          const unsigned long long R = residual_first(weight_at(K.pcum, i), K.qP[i], Wsum);
          K.Rw[i] = R;
          part += R;
        }
        Rsum = fsum(part, s);
        if (Rsum == 0) {  // only reachable through rounding: sample from p^(k)
          for (int i = threadIdx.x; i < n; i += ST) K.Rw[i] = weight_at(K.pcum, i);
          Rsum = Wsum;
        }
      } else {
        // the tokens of the rejected levels leave the draft's support; the
        // total first, so that W^(k) stays in K.Rw if the residual is empty
        if (threadIdx.x == 0) level_scale(Wsum, d, &s.bc64[3], &s.bi[17]);
        __syncthreads();
        const unsigned long long A_fix = s.bc64[3];
        const int G = s.bi[17];
        for (int i = threadIdx.x; i < n; i += ST) {
          bool rem = false;
          for (int e = 0; e < k - 1; ++e) rem |= s.gpidx[e] == i;
          part += rem ? K.Rw[i] : residual_level(K.Rw[i], K.qP[i], A_fix, G);
        }
        Rsum = fsum(part, s);
        if (Rsum == 0) {  // only reachable through rounding: sample from p^(k)
          Rsum = Wsum;
        } else {
          for (int i = threadIdx.x; i < n; i += ST) {
            bool rem = false;
            for (int e = 0; e < k - 1; ++e) rem |= s.gpidx[e] == i;
            if (!rem) K.Rw[i] = residual_level(K.Rw[i], K.qP[i], A_fix, G);
          }
        }
      }
      if (threadIdx.x == 0 && k < g) {
        S = __dadd_rn(S, f32_to_f64(s.gqc[k - 1]));
        s.bi[18] = __dsub_rn(1.0, S) > 0.0 ? 0 : 1;  // the group's draft mass is spent
      }
      __syncthreads();
      if (k == g || s.bi[18]) break;
      Wsum = Rsum;
    }
    if (!accepted) {
      if (threadIdx.x == 0) {
        s.bc64[1] = scale_floor(Rsum, odd24(s.rnd[2][0]));
        s.bi[7] = -1;
      }
      const int per = (n + ST - 1) / ST;
      const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
      unsigned long long loc = 0;
      for (int i = i0; i < i1; ++i) loc += K.Rw[i];
      unsigned long long tot;
      unsigned long long run = fexscan(loc, s, &tot);
      const unsigned long long T = s.bc64[1];
      if (run <= T && T < run + loc) {
        for (int i = i0; i < i1; ++i) {
          run += K.Rw[i];
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

  // ---- S8: proactive-drafting alternates and the vanilla-SJD tail draw.
  // Each draw: the thread whose contiguous run of kept positions holds the
  // first position with C'(i) > T finds it (C' = the inclusive prefix of the
  // weights minus the excluded ones, non-decreasing; C'(n-1) = tot > T).
  {
    const int Km1 = P.K - 1;
    const int per = (n + ST - 1) / ST;
    const int i0 = min(n, static_cast<int>(threadIdx.x) * per), i1 = min(n, i0 + per);
    auto bdraw = [&](int first_idx, int32_t* out) {
      unsigned long long tot = Zk;
      int nex = 0;
      if (first_idx >= 0) {
        const unsigned long long w0 = weight_at(K.pcum, first_idx);
        if (threadIdx.x == 0) {
          s.excl[0] = first_idx;
          s.exw[0] = w0;
        }
        tot -= w0;
        nex = 1;
      }
      __syncthreads();
      int drawn = 0;
      for (int kk = 1; kk <= Km1; ++kk) {
        if (tot == 0) break;
        const unsigned long long T = scale_floor(tot, odd24(s.rnd[3 + (kk >> 2)][kk & 3]));
        auto Cx = [&](int i) {
          unsigned long long c = K.pcum[i];
          for (int e = 0; e < nex; ++e)
            if (s.excl[e] <= i) c -= s.exw[e];
          return c;
        };
        if (i0 < i1 && (i0 == 0 || Cx(i0 - 1) <= T) && Cx(i1 - 1) > T) {
          for (int i = i0; i < i1; ++i)
            if (Cx(i) > T) {
              s.bi[15] = i;
              break;
            }
        }
        __syncthreads();
        const int i = s.bi[15];
        const unsigned long long wi = weight_at(K.pcum, i);
        if (threadIdx.x == 0) {
          out[drawn] = id_of(i);
          s.excl[nex] = i;
          s.exw[nex] = wi;
        }
        ++drawn;
        tot -= wi;
        ++nex;
        __syncthreads();
      }
      return drawn;
    };
    const int na = (n > 0 && Km1 > 0) ? bdraw(xidx, s.alts) : 0;
    if (threadIdx.x == 0) {
      for (int k = 0; k < na; ++k) P.res_alt[bs * Km1 + k] = s.alts[k];
      P.res_altn[bs] = na;
      P.res_x[bs] = x;
      P.res_dev[bs] = x != c1 ? 1 : 0;
    }
    if (!P.ac) {
      int xf = x, fidx = -1;
      if (n > 0) {
        const unsigned long long T = scale_floor(Zk, odd24(s.rnd[2][0]));
        if (i0 < i1 && (i0 == 0 || K.pcum[i0 - 1] <= T) && K.pcum[i1 - 1] > T) {
          for (int i = i0; i < i1; ++i)
            if (K.pcum[i] > T) {
              s.bi[16] = i;
              break;
            }
        }
        __syncthreads();
        fidx = s.bi[16];
        xf = id_of(fidx);
      }
      __syncthreads();  // the alternates above are read by thread 0 before bdraw reuses them
      const int naf = (n > 0 && Km1 > 0) ? bdraw(fidx, s.alts) : 0;
      if (threadIdx.x == 0) {
        for (int k = 0; k < naf; ++k) P.res_altf[bs * Km1 + k] = s.alts[k];
        P.res_altfn[bs] = naf;
        P.res_xf[bs] = xf;
      }
    }
    if (threadIdx.x == 0) {
      P.q_len[bs] = n;
      unsigned long long* st = P.stats + kStatsSpread + 3 * (row & (kStatsSlots - 1));
      atomicAdd(st + 0, 1ull);
      atomicAdd(st + 1, static_cast<unsigned long long>(max(qlen, 0)));
      atomicAdd(st + 2, static_cast<unsigned long long>(n));
    }
  }
  }
  // the row P^t replaces the stored draft row (which verification has read)
  __syncthreads();
  for (int i = threadIdx.x; i < n; i += ST) {
    P.q_ids[bs * P.S + i] = id_of(i);
    P.q_prob[bs * P.S + i] = K.pp[i];
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
    batch_epilogue_staged(P, b, MODE == kModeStep, out_committed, out_ncommit, out_firstrej, esc,
                          reinterpret_cast<int32_t*>(smem_raw + P.f_list_l), P.f_region_bytes / 4);
  }
}

// Raise (never lower) the dynamic shared-memory limit of one kernel.
template <class Kern>
cudaError_t raise_limit(Kern* k, int bytes) {
  cudaFuncAttributes a;
  cudaError_t e = cudaFuncGetAttributes(&a, k);
  if (e != cudaSuccess || a.maxDynamicSharedSizeBytes >= bytes) return e;
  return cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

template <int DT, int MODE>
cudaError_t set_one(int bytes) {
  cudaError_t e = raise_limit(stream_row_kernel<DT, MODE, true, 128>, bytes);
  if (e == cudaSuccess) e = raise_limit(stream_row_kernel<DT, MODE, false, 128>, bytes);
  if (e == cudaSuccess) e = raise_limit(stream_row_kernel<DT, MODE, true, 512>, bytes);
  if (e == cudaSuccess) e = raise_limit(stream_row_kernel<DT, MODE, false, 512>, bytes);
  return e;
}


// Launched with programmatic stream serialization: the grid may begin while
// the previous kernel in the stream finishes (the kernel waits for it before
// its first global read).
template <int DT, int MODE, bool CFG, int NT>
cudaError_t launch_pdl(const DevParams& p, const void* cond, const void* uncond, int32_t* oc, int32_t* on,
                       int32_t* of, cudaStream_t s) {
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3(p.B * p.W);
  lc.blockDim = dim3(NT);
  lc.dynamicSmemBytes = p.f_smem_bytes;
  lc.stream = s;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  lc.attrs = at;
  lc.numAttrs = 1;
  return cudaLaunchKernelEx(&lc, stream_row_kernel<DT, MODE, CFG, NT>, p, cond, uncond, oc, on, of);
}

template <int DT, int MODE, int NT>
cudaError_t launch_n(const DevParams& p, const void* cond, const void* uncond, bool use_cfg, int32_t* oc,
                     int32_t* on, int32_t* of, cudaStream_t s) {
  return use_cfg ? launch_pdl<DT, MODE, true, NT>(p, cond, uncond, oc, on, of, s)
                 : launch_pdl<DT, MODE, false, NT>(p, cond, uncond, oc, on, of, s);
}

template <int DT, int MODE>
cudaError_t launch_m(const DevParams& p, const void* cond, const void* uncond, bool use_cfg, int32_t* oc,
                     int32_t* on, int32_t* of, cudaStream_t s) {
  return p.f_nt == 512 ? launch_n<DT, MODE, 512>(p, cond, uncond, use_cfg, oc, on, of, s)
                       : launch_n<DT, MODE, 128>(p, cond, uncond, use_cfg, oc, on, of, s);
}

}  // namespace

// The (dtype, mode) variants, instantiated one pair per translation unit
// (sjd_fast_part.cu) so that they compile in parallel.
template <int DT, int MODE>
cudaError_t fast_launch(const DevParams& p, const void* cond, const void* uncond, bool use_cfg, int32_t* oc,
                        int32_t* on, int32_t* of, cudaStream_t s) {
  return launch_m<DT, MODE>(p, cond, uncond, use_cfg, oc, on, of, s);
}

template <int DT, int MODE>
cudaError_t fast_raise_smem(int bytes) {
  return set_one<DT, MODE>(bytes);
}

}  // namespace sjd
