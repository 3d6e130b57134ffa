// Device helpers shared by the row kernels: Philox, the arithmetic of the
// method's definition, block-wide reductions and scans, prefix searches and
// the per-batch epilogue (first rejection, commit, window refill).
#pragma once

#include <climits>

#include "sjd_exp2_table.h"
#include "sjd_internal.h"

namespace sjd {
namespace {

// ---------------------------------------------------------------------------
// Philox-4x32-10 (Salmon et al., SC'11): multipliers and Weyl key increments.
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += kPhiloxW0;
      k1 += kPhiloxW1;
    }
    const uint32_t hi0 = __umulhi(kPhiloxM0, c.x), lo0 = kPhiloxM0 * c.x;
    const uint32_t hi1 = __umulhi(kPhiloxM1, c.z), lo1 = kPhiloxM1 * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// Word `lane` of the block addressed by (position, step, batch, purpose).
__device__ __forceinline__ uint32_t rand32(const DevParams& P, uint32_t pos, uint32_t t,
                                           uint32_t b, uint32_t purpose, uint32_t lane) {
  const uint4 r = philox4x32_10(make_uint4(pos, t, b, purpose + 8u * (lane >> 2)), P.seed_lo,
                                P.seed_hi);
  switch (lane & 3u) {
    case 0: return r.x;
    case 1: return r.y;
    case 2: return r.z;
    default: return r.w;
  }
}

// Lanes 0 and 1 joined as (lane0 << 32) | lane1.
__device__ __forceinline__ uint64_t rand64(const DevParams& P, uint32_t pos, uint32_t t,
                                           uint32_t b, uint32_t purpose) {
  const uint4 r = philox4x32_10(make_uint4(pos, t, b, purpose), P.seed_lo, P.seed_hi);
  return (static_cast<uint64_t>(r.x) << 32) | r.y;
}

// Odd numerator of the uniform u = (2m+1) / 2^24, m = r >> 9.
__device__ __forceinline__ uint32_t odd24(uint32_t r) { return ((r >> 9) << 1) | 1u; }

// ---------------------------------------------------------------------------
// Bounds-checked build (compiled with SJD_CHECKS): an index a kernel takes
// from data is tested against its array's length; one outside latches
// SJD_ERR_BOUNDS in the status word and is clamped into the array, so that
// the kernel never traps and the host learns of it at the next sjd_sync.
// Without SJD_CHECKS the macro is the index itself.
#ifdef SJD_CHECKS
__device__ __forceinline__ int checked_idx(const DevParams& P, long long i, long long n) {
  if (i < 0 || i >= n) {
    atomicOr(P.err, err_bit(SJD_ERR_BOUNDS));
    return n > 0 && i >= n ? static_cast<int>(n - 1) : 0;
  }
  return static_cast<int>(i);
}
#define SJD_IDX(i, n) checked_idx(P, (i), (n))
#else
#define SJD_IDX(i, n) (i)
#endif

// ---------------------------------------------------------------------------
// Arithmetic of the method's definition.

// exp(t) for t <= 0: base-2 range reduction (Cody & Waite) and the Taylor
// polynomial of 2^f on |f| <= 1/2, coefficients fl32((ln 2)^k / k!),
// evaluated by Horner's rule with one fused multiply-add per step.
__device__ __forceinline__ float exp_neg(float t) {
  const float a = __fmul_rn(t, 0x1.715476p+0f);  // fl32(log2 e)
  if (!(a >= -64.0f)) return 0.0f;
  const float n = rintf(a);
  const float f = __fsub_rn(a, n);
  float y = 0x1.ffcbfcp-17f;
  y = __fmaf_rn(y, f, 0x1.430912p-13f);
  y = __fmaf_rn(y, f, 0x1.5d87fep-10f);
  y = __fmaf_rn(y, f, 0x1.3b2ab6p-7f);
  y = __fmaf_rn(y, f, 0x1.c6b08ep-5f);
  y = __fmaf_rn(y, f, 0x1.ebfbe0p-3f);
  y = __fmaf_rn(y, f, 0x1.62e430p-1f);
  y = __fmaf_rn(y, f, 1.0f);
  return __fmul_rn(y, __int_as_float((static_cast<int>(n) + 127) << 23));
}

// rint(x * 2^47) (half to even) of x = +0 or a finite fp32 in [0, 2), with
// integer operations only (64-bit float/integer conversions run on the fp64
// unit): x = m * 2^(ex - 23) with a 24-bit m, so x * 2^47 = m * 2^(ex + 24).
__device__ __forceinline__ unsigned long long quant(float x) {
  const uint32_t b = __float_as_uint(x);
  if (b < 0x00800000u) return 0ull;  // +0 and subnormals (< 2^-126) round to 0
  const uint32_t m = (b & 0x7FFFFFu) | 0x800000u;
  const int sh = static_cast<int>(b >> 23) - 127 + 24;
  if (sh >= 0) return static_cast<unsigned long long>(m) << sh;
  const int s = -sh;
  if (s > 24) return 0ull;
  const uint32_t q = m >> s, rem = m & ((1u << s) - 1u), half = 1u << (s - 1);
  return q + ((rem > half || (rem == half && (q & 1u))) ? 1u : 0u);
}
// w * 2^-47 as fp32 for a weight w made by quant() (at most 24 significant
// bits, so the value is exact): split into two exact 32-bit halves.
__device__ __forceinline__ float dequant(unsigned long long w) {
  const float hi = __uint2float_rn(static_cast<uint32_t>(w >> 32));
  const float lo = __uint2float_rn(static_cast<uint32_t>(w));
  return __fmul_rn(__fadd_rn(__fmul_rn(hi, 0x1p32f), lo), 0x1p-47f);
}
// x rounded to the nearest value with `bits` significant bits (ties to even),
// for x != 0; *p is the position of its leading bit afterwards. Integer
// operations only: on this GPU a u64 to double conversion takes about 165
// cycles and a dependent fp64 add or multiply 64 (measured), against about 5
// for an fp32 fused multiply-add.
__device__ __forceinline__ unsigned long long round_bits(unsigned long long x, int bits, int* p) {
  int lead = 63 - __clzll(static_cast<long long>(x));
  if (lead >= bits) {
    const int sh = lead - bits + 1;
    const unsigned long long q = x >> sh, rem = x & ((1ull << sh) - 1ull), half = 1ull << (sh - 1);
    unsigned long long r = q + ((rem > half || (rem == half && (q & 1ull))) ? 1ull : 0ull);
    if (r >> bits) {  // the rounding carried into a new leading bit
      r >>= 1;
      ++lead;
    }
    x = r << (lead - bits + 1);
  }
  *p = lead;
  return x;
}
// fp32 of x (ties to even), as __ull2float_rn: a finite float (x < 2^64).
__device__ __forceinline__ float u64_to_f32_rn(unsigned long long x) {
  if (x == 0ull) return 0.0f;
  int p;
  const unsigned long long r = round_bits(x, 24, &p);  // r = m 2^(p-23), 2^23 <= m < 2^24
  const uint32_t m = static_cast<uint32_t>(p >= 23 ? r >> (p - 23) : r << (23 - p));
  return __uint_as_float((static_cast<uint32_t>(p + 127) << 23) | (m & 0x7FFFFFu));
}
// The double nearest x (ties to even), as __ull2double_rn, with integer
// operations only.
__device__ __forceinline__ double u64_to_f64_rn(unsigned long long x) {
  if (x == 0ull) return 0.0;
  int p;
  const unsigned long long r = round_bits(x, 53, &p);  // r = m 2^(p-52), 2^52 <= m < 2^53
  const unsigned long long m = p >= 52 ? r >> (p - 52) : r << (52 - p);
  return __longlong_as_double(static_cast<long long>((static_cast<unsigned long long>(p + 1023) << 52) |
                                                     (m & 0xFFFFFFFFFFFFFull)));
}
// A float widened to double (exact), with integer operations for finite
// values.
__device__ __forceinline__ double f32_to_f64(float f) {
  const uint32_t b = __float_as_uint(f);
  const uint32_t ex = (b >> 23) & 0xFFu;
  const unsigned long long sign = static_cast<unsigned long long>(b >> 31) << 63;
  if (ex == 0xFFu) return static_cast<double>(f);
  uint32_t mant = b & 0x7FFFFFu;
  int e = static_cast<int>(ex) - 127;
  if (ex == 0u) {  // zero or subnormal: value = mant 2^-149
    if (mant == 0u) return __longlong_as_double(static_cast<long long>(sign));
    const int lead = 31 - __clz(static_cast<int>(mant));
    e = lead - 149;
    mant = (mant << (23 - lead)) & 0x7FFFFFu;
  }
  return __longlong_as_double(static_cast<long long>(sign | (static_cast<unsigned long long>(e + 1023) << 52) |
                                                     (static_cast<unsigned long long>(mant) << 29)));
}

// fl32(fl64(total) 2^-47) with integer operations: the rounding to 53 bits,
// then to 24 (both ties to even), then the exact scaling.
__device__ __forceinline__ float fix_to_f32(unsigned long long total) {
  if (total == 0ull) return 0.0f;
  int p;
  const unsigned long long r53 = round_bits(total, 53, &p);
  const unsigned long long r = round_bits(r53, 24, &p);
  const uint32_t m = static_cast<uint32_t>(p >= 23 ? r >> (p - 23) : r << (23 - p));
  return __uint_as_float((static_cast<uint32_t>(p - 47 + 127) << 23) | (m & 0x7FFFFFu));
}
// floor(odd * total / 2^24) (the product fits in 88 bits).
__device__ __forceinline__ unsigned long long scale_floor(unsigned long long total, uint32_t odd) {
  const unsigned long long lo = total * odd;
  const unsigned long long hi = __umul64hi(total, static_cast<unsigned long long>(odd));
  return (hi << 40) | (lo >> 24);
}
// ceil(mant * total / 2^shift), shift >= 24.
__device__ __forceinline__ unsigned long long scale_ceil(unsigned long long total, uint32_t mant,
                                                         int shift) {
  const unsigned long long lo = total * mant;
  const unsigned long long hi = __umul64hi(total, static_cast<unsigned long long>(mant));
  unsigned long long q;
  bool rem;
  if (shift >= 128) {
    q = 0;
    rem = (lo | hi) != 0;
  } else if (shift >= 64) {
    const int s = shift - 64;
    q = s ? (hi >> s) : hi;
    rem = lo != 0 || (s && (hi & ((1ull << s) - 1)) != 0);
  } else {
    q = (hi << (64 - shift)) | (lo >> shift);
    rem = (lo & ((1ull << shift) - 1)) != 0;
  }
  return q + (rem ? 1 : 0);
}
// ---------------------------------------------------------------------------
// Precise weights of the kept ids: E = round(2^47 exp(l - m)) with l the
// guided logit taken exactly from the inputs (double-float arithmetic: a
// value is an unevaluated sum hi + lo of two fp32) and exp evaluated to
// about 1e-12 relative, so that every decision taken on these weights (the
// acceptance test, the residual draw, the alternates) agrees with the
// real-number sampler except within about 1e-12 of its threshold.

// Knuth's TwoSum: a + b = s + e exactly.
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = __fadd_rn(a, b);
  const float ap = __fsub_rn(s, b);
  const float bp = __fsub_rn(s, ap);
  e = __fadd_rn(__fsub_rn(a, ap), __fsub_rn(b, bp));
}

// |x| 2^k truncated toward zero (x given by its bits; normal or zero, the
// result below 2^64).
__device__ __forceinline__ unsigned long long f32_fix_mag(uint32_t b, int k) {
  const uint32_t ex = (b >> 23) & 0xFFu;
  if (ex == 0u) return 0ull;
  const unsigned long long mnt = (b & 0x7FFFFFu) | 0x800000u;
  const int sh = static_cast<int>(ex) - 150 + k;
  if (sh >= 0) return mnt << sh;
  return sh > -32 ? (mnt >> -sh) : 0ull;
}

// exp(th + tl) 2^47 rounded to an integer, for th + tl <= about 0 (0 below
// t = -44). Base-2 reduction x = t log2(e) = n + j/64 + g with |g| <=
// 1/128, e^(g ln 2) by its Taylor series to the fifth power, 2^(j/64) from
// the double-float table, all in double-float; the value (rh + rl) 2^(47+n)
// is then rounded with 16 fractional bits.
__device__ __forceinline__ unsigned long long exp_weight_df(float th, float tl) {
  const float xh = __fmul_rn(th, kLog2eHi);
  const float xe = __fmaf_rn(th, kLog2eHi, -xh);
  const float xl = __fmaf_rn(th, kLog2eLo, __fmaf_rn(tl, kLog2eHi, xe));
  if (!(xh >= -64.0f)) return 0ull;
  const float rn = __fadd_rn(xh, 0x1.8p23f);
  const float n = __fsub_rn(rn, 0x1.8p23f);
  const int ni = static_cast<int>(__float_as_uint(rn) - __float_as_uint(0x1.8p23f));
  const float fh = __fsub_rn(xh, n);  // exact, |fh| <= 1/2
  const float rj = __fadd_rn(__fmul_rn(fh, 64.0f), 0x1.8p23f);
  const float jf = __fsub_rn(rj, 0x1.8p23f);
  const int ji = static_cast<int>(__float_as_uint(rj) - __float_as_uint(0x1.8p23f));
  const float gh = __fmaf_rn(jf, -0x1p-6f, fh);  // exact, |gh| <= 1/128
  const float yh = __fmul_rn(gh, kLn2Hi);
  const float ye = __fmaf_rn(gh, kLn2Hi, -yh);
  const float yl = __fmaf_rn(gh, kLn2Lo, __fmaf_rn(xl, kLn2Hi, ye));
  const float y1 = __fadd_rn(yh, yl);  // the polynomial's argument (yl is not below ulp(yh))
  float pp = __fmaf_rn(y1, kInv120, kInv24);
  pp = __fmaf_rn(pp, y1, kInv6);
  pp = __fmaf_rn(pp, y1, 0.5f);
  const float q = __fmul_rn(__fmul_rn(y1, y1), pp);  // y^2 (1/2 + y/6 + y^2/24 + y^3/120)
  const float sh = __fadd_rn(1.0f, yh);
  const float se = __fsub_rn(yh, __fsub_rn(sh, 1.0f));
  const float sl = __fadd_rn(se, __fadd_rn(yl, q));
  const float2 T = kExp2Table[ji + 32];
  const float rh = __fmul_rn(T.x, sh);
  const float re = __fmaf_rn(T.x, sh, -rh);
  const float rl = __fmaf_rn(T.x, sl, __fmaf_rn(T.y, sh, re));
  const int k = 47 + ni + 16;
  const uint32_t bl = __float_as_uint(rl);
  const unsigned long long a = f32_fix_mag(__float_as_uint(rh), k);
  const unsigned long long l = f32_fix_mag(bl, k);
  return (((bl >> 31) ? a - l : a + l) + 0x8000ull) >> 16;
}

// Precise weight of one id from its raw inputs: l = u + s (c - u) (or c
// without guidance), divided by T when temp, minus the row's stage-one
// maximum m (any reference point gives the same probabilities).
__device__ __forceinline__ unsigned long long precise_weight(float c, float u, bool cfg, float s, bool temp,
                                                             float T, float m) {
  float lh, ll;
  if (cfg) {
    float dh, dl;
    two_sum(c, -u, dh, dl);                 // c - u = dh + dl
    const float ph = __fmul_rn(s, dh);
    float pe = __fmaf_rn(s, dh, -ph);       // s dh = ph + pe
    pe = __fmaf_rn(s, dl, pe);
    float le;
    two_sum(u, ph, lh, le);
    ll = __fadd_rn(le, pe);
  } else {
    lh = c;
    ll = 0.0f;
  }
  if (temp) {
    const float qh = __fdiv_rn(lh, T);
    const float r = __fmaf_rn(-qh, T, lh);  // exact remainder
    ll = __fdiv_rn(__fadd_rn(r, ll), T);
    lh = qh;
  }
  float th, te;
  two_sum(lh, -m, th, te);
  return exp_weight_df(th, __fadd_rn(te, ll));
}

// The stored probability of a kept id: fl(fl(E 2^-47) / Wz).
__device__ __forceinline__ float prob_of(unsigned long long E, float Wz) {
  return __fdiv_rn(__fmul_rn(u64_to_f32_rn(E), 0x1p-47f), Wz);
}

// Acceptance test of candidate k of a group (Sec. 3.2, Thm. 2): u <
// p^(k)(c)/q^(k)(c) with p^(k)(c) = Wc / Wsum (integer weights) and
// q^(k)(c) = q / d, taken as u q Wsum < Wc d in fp64 (u q is exact; d = 1
// at the first level, so there the test is u q fl(Wsum) < Wc).
__device__ __forceinline__ bool accept_exact(uint32_t odd, float q, unsigned long long Wsum, unsigned long long Wc,
                                             double d) {
  // (the conversions are exact or round as the casts do, without the fp64
  // unit: odd 2^-24 is exact, as is the widened q)
  const double u = __longlong_as_double(__double_as_longlong(u64_to_f64_rn(odd)) - (24ll << 52));
  const double uq = __dmul_rn(u, f32_to_f64(q));
  return __dmul_rn(uq, u64_to_f64_rn(Wsum)) < __dmul_rn(u64_to_f64_rn(Wc), d);
}

// ceil(q * total) of an fp32 q in [0, 1] and an integer total (exact).
__device__ __forceinline__ unsigned long long ceil_q_times(float q, unsigned long long total) {
  const uint32_t b = __float_as_uint(q);
  const uint32_t ex = (b >> 23) & 0xFFu;
  const uint32_t mant = ex ? ((b & 0x7FFFFFu) | 0x800000u) : (b & 0x7FFFFFu);
  if (mant == 0u) return 0ull;
  return scale_ceil(total, mant, 150 - static_cast<int>(ex ? ex : 1u));
}

// Residual weight of one id at the first level: max(0, E - ceil(q Z)).
__device__ __forceinline__ unsigned long long residual_first(unsigned long long E, float q, unsigned long long Z) {
  const unsigned long long c = ceil_q_times(q, Z);
  return E > c ? E - c : 0ull;
}

// A = fl64(fl64(Wsum) / d) of a later group level, as A = A_fix 2^-G with
// A_fix in [2^62, 2^63) (exact: A has 53 significant bits). One division
// per level; the per-id residuals below are then integer operations.
__device__ __forceinline__ void level_scale(unsigned long long Wsum, double d, unsigned long long* A_fix, int* G) {
  const double A = __ddiv_rn(u64_to_f64_rn(Wsum), d);
  const unsigned long long b = static_cast<unsigned long long>(__double_as_longlong(A));
  *G = 62 - (static_cast<int>((b >> 52) & 0x7FFull) - 1023);
  *A_fix = ((b & 0xFFFFFFFFFFFFFull) | 0x10000000000000ull) << 10;
}

// Residual weight of one id at a later level: max(0, W - ceil(q A)), the
// weight of p^(k) - q^(k) with q^(k) Wsum = (q / d) Wsum = q A.
__device__ __forceinline__ unsigned long long residual_level(unsigned long long W, float q, unsigned long long A_fix,
                                                             int G) {
  const uint32_t b = __float_as_uint(q);
  const uint32_t ex = (b >> 23) & 0xFFu;
  const uint32_t mant = ex ? ((b & 0x7FFFFFu) | 0x800000u) : (b & 0x7FFFFFu);
  if (mant == 0u) return W;
  const int shift = G + 150 - static_cast<int>(ex ? ex : 1u);  // q A = mant A_fix 2^-shift
  if (shift < 24) return 0ull;                                  // q A >= 2^62 > W
  const unsigned long long c = scale_ceil(A_fix, mant, shift);
  return W > c ? W - c : 0ull;
}

// Order-preserving key: larger l <-> larger key; -0 sorts with +0. The
// shared-memory padding (NaN bit pattern 0xFFFFFFFF) maps to key 0, below
// every real value including -inf.
__device__ __forceinline__ uint32_t f2key(float f) {
  uint32_t u = __float_as_uint(f);
  if (u == 0x80000000u) u = 0u;
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float key2f(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}
constexpr uint32_t kKeyNegInf = 0x007FFFFFu;  // key of -inf
__device__ __forceinline__ float pad_value() { return __uint_as_float(0xFFFFFFFFu); }

__device__ __forceinline__ float bf16_bits_to_f32(uint32_t h) { return __uint_as_float(h << 16); }

__device__ __forceinline__ float combine(float c, float u, float s, bool cfg) {
  return cfg ? __fmaf_rn(s, __fsub_rn(c, u), u) : c;
}

// ---------------------------------------------------------------------------
// Block-wide helpers (any block of at most kThreads threads).

struct Scratch {
  unsigned long long u64[kWarps];
  unsigned long long u64b[kWarps];
  uint32_t u32[kWarps];
  uint32_t u32b[kWarps];
  float f32[kWarps];
  // broadcast slots
  unsigned long long bc_u64[4];
  int bc_i[8];
  uint32_t bc_u[4];
  float bc_f[4];
  uint32_t cand_count;
  uint32_t cand_kmin, cand_kmax;
};

__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }
__device__ __forceinline__ int warp_id() { return threadIdx.x >> 5; }
__device__ __forceinline__ int num_warps() { return static_cast<int>(blockDim.x) >> 5; }

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
  return v;
}

__device__ __forceinline__ unsigned long long block_sum_u64(unsigned long long v, Scratch& sc) {
  v = warp_sum_u64(v);
  if (lane_id() == 0) sc.u64[warp_id()] = v;
  __syncthreads();
  unsigned long long r = 0;
#pragma unroll
  for (int i = 0; i < num_warps(); ++i) r += sc.u64[i];
  __syncthreads();
  return r;
}

__device__ __forceinline__ uint32_t block_max_u32(uint32_t v, Scratch& sc) {
  v = __reduce_max_sync(0xFFFFFFFFu, v);
  if (lane_id() == 0) sc.u32[warp_id()] = v;
  __syncthreads();
  uint32_t r = 0;
#pragma unroll
  for (int i = 0; i < num_warps(); ++i) r = max(r, sc.u32[i]);
  __syncthreads();
  return r;
}

__device__ __forceinline__ uint32_t block_min_u32(uint32_t v, Scratch& sc) {
  v = __reduce_min_sync(0xFFFFFFFFu, v);
  if (lane_id() == 0) sc.u32[warp_id()] = v;
  __syncthreads();
  uint32_t r = 0xFFFFFFFFu;
#pragma unroll
  for (int i = 0; i < num_warps(); ++i) r = min(r, sc.u32[i]);
  __syncthreads();
  return r;
}

__device__ __forceinline__ uint32_t block_or_u32(uint32_t v, Scratch& sc) {
  v = __reduce_or_sync(0xFFFFFFFFu, v);
  if (lane_id() == 0) sc.u32[warp_id()] = v;
  __syncthreads();
  uint32_t r = 0;
#pragma unroll
  for (int i = 0; i < num_warps(); ++i) r |= sc.u32[i];
  __syncthreads();
  return r;
}

// Exclusive scan of one u64 per thread (thread order); *total gets the sum.
__device__ __forceinline__ unsigned long long block_exscan_u64(unsigned long long v, Scratch& sc,
                                                               unsigned long long* total) {
  unsigned long long incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane_id() >= o) incl += y;
  }
  if (lane_id() == 31) sc.u64[warp_id()] = incl;
  __syncthreads();
  unsigned long long base = 0, tot = 0;
  for (int i = 0; i < num_warps(); ++i) {
    const unsigned long long s = sc.u64[i];
    if (i < warp_id()) base += s;
    tot += s;
  }
  __syncthreads();
  *total = tot;
  return base + incl - v;
}

// Exclusive scan of a (u32 count, u64 sum) pair per thread.
__device__ __forceinline__ void block_exscan_pair(uint32_t c, unsigned long long s, Scratch& sc,
                                                  uint32_t* c_ex, unsigned long long* s_ex,
                                                  uint32_t* c_tot, unsigned long long* s_tot) {
  uint32_t ci = c;
  unsigned long long si = s;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t yc = __shfl_up_sync(0xFFFFFFFFu, ci, o);
    const unsigned long long ys = __shfl_up_sync(0xFFFFFFFFu, si, o);
    if (lane_id() >= o) {
      ci += yc;
      si += ys;
    }
  }
  if (lane_id() == 31) {
    sc.u32b[warp_id()] = ci;
    sc.u64b[warp_id()] = si;
  }
  __syncthreads();
  uint32_t cb = 0, ct = 0;
  unsigned long long sb = 0, st = 0;
  for (int i = 0; i < num_warps(); ++i) {
    if (i < warp_id()) {
      cb += sc.u32b[i];
      sb += sc.u64b[i];
    }
    ct += sc.u32b[i];
    st += sc.u64b[i];
  }
  __syncthreads();
  *c_ex = cb + ci - c;
  *s_ex = sb + si - s;
  *c_tot = ct;
  *s_tot = st;
}

// ---------------------------------------------------------------------------
// Threshold in the order (key desc, id asc): an element belongs to the
// selected prefix iff key > key_t or (key == key_t and id <= id_t).
struct Cut {
  uint32_t key;
  int id;
};

__device__ __forceinline__ bool in_cut(uint32_t key, int id, Cut c) {
  return key > c.key || (key == c.key && id <= c.id);
}

// The prefix is "everything real" when no cut applies (key 1 is never used
// by a real value: real keys are >= the key of -inf).
__device__ __forceinline__ Cut no_cut() { return Cut{1u, INT_MAX}; }


// Inclusive-prefix search: first i in [0, n) with C'(i) > T, where
// C'(i) = pcum[i] - (sum of weights of excluded indices <= i).
__device__ __forceinline__ int search_excluding(const unsigned long long* pcum, int n,
                                                unsigned long long T, const int* excl,
                                                const unsigned long long* exw, int nexcl) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    unsigned long long c = pcum[mid];
    for (int e = 0; e < nexcl; ++e)
      if (excl[e] <= mid) c -= exw[e];
    if (c > T) hi = mid; else lo = mid + 1;
  }
  return lo;
}

__device__ __forceinline__ int find_sorted(const int32_t* ids, int n, int v) {
  int lo = 0, hi = n;
  while (lo < hi) {
    const int mid = (lo + hi) >> 1;
    if (ids[mid] < v) lo = mid + 1; else hi = mid;
  }
  return (lo < n && ids[lo] == v) ? lo : -1;
}

__device__ __forceinline__ unsigned long long weight_at(const unsigned long long* pcum, int i) {
  return pcum[i] - (i ? pcum[i - 1] : 0ull);
}

// Draw up to `count` tokens without replacement from the kept row (integer
// weights) excluding index `first_idx` (-1: none); returns the number drawn.
// Draw k (1-based) takes word lane0 + k - 1 of purpose `purpose` (the
// proactive-drafting alternates: purpose kPd from lane 1).
template <class IdOf>
__device__ int draw_without_replacement(const DevParams& P, const unsigned long long* pcum, IdOf id_of, int n,
                                        unsigned long long Z, int first_idx, uint32_t pos,
                                        uint32_t t, uint32_t b, int count, int32_t* out,
                                        uint32_t purpose = kPd, int lane0 = 1) {
  int excl[kMaxK];
  unsigned long long exw[kMaxK];
  int nex = 0;
  unsigned long long tot = Z;
  if (first_idx >= 0) {
    excl[0] = first_idx;
    exw[0] = weight_at(pcum, first_idx);
    tot -= exw[0];
    nex = 1;
  }
  int drawn = 0;
  for (int k = 1; k <= count; ++k) {
    if (tot == 0) break;
    const uint32_t odd = odd24(rand32(P, pos, t, b, purpose, static_cast<uint32_t>(lane0 + k - 1)));
    const unsigned long long T = scale_floor(tot, odd);
    const int i = search_excluding(pcum, n, T, excl, exw, nex);
    out[drawn++] = id_of(i);
    excl[nex] = i;
    exw[nex] = weight_at(pcum, i);
    tot -= exw[nex];
    ++nex;
  }
  return drawn;
}

// ---------------------------------------------------------------------------
// Per-batch epilogue: first rejection, committed tokens (S6) and, in the
// fused step, the window refill (S8-S9).

__device__ void batch_refresh(const DevParams& P, int b, int first, int ncommit, Scratch& sc) {
  const int W = P.W;
  const int old_abs = P.abs_pos[b];
  const int new_abs = old_abs + ncommit;
  const uint32_t t = P.step_t[b];
  const int Km1 = P.K - 1;
  for (int r = threadIdx.x; r < W; r += blockDim.x) {
    const int slot = (new_abs + r) % W;
    const size_t bs = static_cast<size_t>(b) * W + slot;
    int32_t* cg = P.cand + bs * P.K;
    int x;
    if (r < W - ncommit) {
      const int j = r + ncommit;
      const bool fresh_tail = !P.ac && first >= 0 && j > first;
      x = fresh_tail ? __ldcg(P.res_xf + bs) : __ldcg(P.res_x + bs);
      int g = 1;
      if (first >= 0 && j <= first + P.D && Km1 > 0) {
        const int na = fresh_tail ? __ldcg(P.res_altfn + bs) : __ldcg(P.res_altn + bs);
        const int32_t* src = (fresh_tail ? P.res_altf : P.res_alt) + bs * Km1;
        for (int k = 0; k < na; ++k) cg[1 + k] = __ldcg(src + k);
        g = 1 + na;
      }
      cg[0] = x;
      P.gsize[bs] = g;
    } else {
      const uint32_t a = static_cast<uint32_t>(new_abs + r);
      const uint64_t r64 = rand64(P, a, t, static_cast<uint32_t>(b), kInit);
      x = P.lo + static_cast<int>(__umul64hi(r64, static_cast<unsigned long long>(P.veff)));
      cg[0] = x;
      P.gsize[bs] = 1;
      P.q_len[bs] = -1;
    }
    P.win_tok[static_cast<size_t>(b) * W + r] = x;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    const int last_slot = (old_abs + ncommit - 1) % W;
    P.last_tok[b] = __ldcg(P.res_x + static_cast<size_t>(b) * W + last_slot);
    P.abs_pos[b] = new_abs;
    P.step_t[b] = t + 1;
  }
}

__device__ void batch_epilogue(const DevParams& P, int b, bool fused, int32_t* out_committed,
                               int32_t* out_ncommit, int32_t* out_firstrej, Scratch& sc) {
  const int W = P.W;
  const int abs0 = P.abs_pos[b];
  uint32_t first = 0xFFFFFFFFu;
  for (int j = threadIdx.x; j < W; j += blockDim.x) {
    const int slot = (abs0 + j) % W;
    if (__ldcg(P.res_dev + static_cast<size_t>(b) * W + slot)) first = min(first, static_cast<uint32_t>(j));
  }
  first = block_min_u32(first, sc);
  const int fr = first == 0xFFFFFFFFu ? -1 : static_cast<int>(first);
  const int nc = fr < 0 ? W : fr + 1;
  for (int j = threadIdx.x; j < W; j += blockDim.x) {
    const int slot = (abs0 + j) % W;
    const int v = j < nc ? __ldcg(P.res_x + static_cast<size_t>(b) * W + slot) : -1;
    P.committed[static_cast<size_t>(b) * W + j] = v;
    if (out_committed) out_committed[static_cast<size_t>(b) * W + j] = v;
  }
  if (threadIdx.x == 0) {
    P.first_rej[b] = fr;
    P.n_commit[b] = nc;
    if (out_ncommit) out_ncommit[b] = nc;
    if (out_firstrej) out_firstrej[b] = fr;
  }
  if (fused) {
    __syncthreads();
    batch_refresh(P, b, fr, nc, sc);
  }
  if (threadIdx.x == 0) {
    P.ticket[b] = 0;
    atomicAdd(&P.stats[3], b == 0 ? 1ull : 0ull);
  }
}

// The same S6 + S9 epilogue with every row result of the batch element read
// in one round (all rows' loads in flight together) and exchanged through
// `stage` (shared memory the row kernel no longer needs, stage_words 32-bit
// words); falls back to batch_epilogue when the stage is too small.
__device__ void batch_epilogue_staged(const DevParams& P, int b, bool fused, int32_t* out_committed,
                                      int32_t* out_ncommit, int32_t* out_firstrej, Scratch& sc, int32_t* stage,
                                      size_t stage_words) {
  const int W = P.W;
  const int Km1 = P.K > 1 ? P.K - 1 : 0;
  const size_t need = static_cast<size_t>(W) * (4 + 2 * Km1);
  if (need > stage_words) {
    batch_epilogue(P, b, fused, out_committed, out_ncommit, out_firstrej, sc);
    return;
  }
  int32_t* X = stage;                   // [W] result token of window row j
  int32_t* XF = X + W;                  // [W] vanilla-SJD tail draw
  int32_t* NA = XF + W;                 // [W] alternates drawn
  int32_t* NAF = NA + W;                // [W] alternates of the tail draw
  int32_t* AL = NAF + W;                // [W][Km1]
  int32_t* ALF = AL + static_cast<size_t>(W) * Km1;
  const int abs0 = P.abs_pos[b];
  const uint32_t t = P.step_t[b];
  uint32_t first = 0xFFFFFFFFu;
  for (int j = threadIdx.x; j < W; j += blockDim.x) {
    const size_t bsj = static_cast<size_t>(b) * W + (abs0 + j) % W;
    if (__ldcg(P.res_dev + bsj)) first = min(first, static_cast<uint32_t>(j));
    X[j] = __ldcg(P.res_x + bsj);
    NA[j] = Km1 ? __ldcg(P.res_altn + bsj) : 0;
    for (int k = 0; k < Km1; ++k) AL[static_cast<size_t>(j) * Km1 + k] = __ldcg(P.res_alt + bsj * Km1 + k);
    if (!P.ac) {
      XF[j] = __ldcg(P.res_xf + bsj);
      NAF[j] = Km1 ? __ldcg(P.res_altfn + bsj) : 0;
      for (int k = 0; k < Km1; ++k) ALF[static_cast<size_t>(j) * Km1 + k] = __ldcg(P.res_altf + bsj * Km1 + k);
    }
  }
  first = block_min_u32(first, sc);  // its barriers also publish the stage
  const int fr = first == 0xFFFFFFFFu ? -1 : static_cast<int>(first);
  const int nc = fr < 0 ? W : fr + 1;
  for (int j = threadIdx.x; j < W; j += blockDim.x) {
    const int v = j < nc ? X[j] : -1;
    P.committed[static_cast<size_t>(b) * W + j] = v;
    if (out_committed) out_committed[static_cast<size_t>(b) * W + j] = v;
  }
  if (threadIdx.x == 0) {
    P.first_rej[b] = fr;
    P.n_commit[b] = nc;
    if (out_ncommit) out_ncommit[b] = nc;
    if (out_firstrej) out_firstrej[b] = fr;
  }
  if (fused) {
    // S9 as batch_refresh, from the stage
    const int new_abs = abs0 + nc;
    for (int r = threadIdx.x; r < W; r += blockDim.x) {
      const size_t bs = static_cast<size_t>(b) * W + (new_abs + r) % W;
      int32_t* cg = P.cand + bs * P.K;
      int x;
      if (r < W - nc) {
        const int j = r + nc;
        const bool fresh_tail = !P.ac && fr >= 0 && j > fr;
        x = fresh_tail ? XF[j] : X[j];
        int g = 1;
        if (fr >= 0 && j <= fr + P.D && Km1 > 0) {
          const int na = fresh_tail ? NAF[j] : NA[j];
          const int32_t* src = (fresh_tail ? ALF : AL) + static_cast<size_t>(j) * Km1;
          for (int k = 0; k < na; ++k) cg[1 + k] = src[k];
          g = 1 + na;
        }
        cg[0] = x;
        P.gsize[bs] = g;
      } else {
        const uint32_t a = static_cast<uint32_t>(new_abs + r);
        const uint64_t r64 = rand64(P, a, t, static_cast<uint32_t>(b), kInit);
        x = P.lo + static_cast<int>(__umul64hi(r64, static_cast<unsigned long long>(P.veff)));
        cg[0] = x;
        P.gsize[bs] = 1;
        P.q_len[bs] = -1;
      }
      P.win_tok[static_cast<size_t>(b) * W + r] = x;
    }
    if (threadIdx.x == 0) {
      P.last_tok[b] = X[nc - 1];
      P.abs_pos[b] = new_abs;
      P.step_t[b] = t + 1;
    }
  }
  if (threadIdx.x == 0) {
    P.ticket[b] = 0;
    atomicAdd(&P.stats[3], b == 0 ? 1ull : 0ull);
  }
}


// ---------------------------------------------------------------------------
// S6 + S9 with the full proactive-drafting tree (fused step). Thread 0 walks
// the tree from the root: the result of the current node's row (the window
// row on the main path, the node's own row off it) moves the walk to the
// child carrying that token; the context breaks where no child does, or at
// the last tree row once the path has left the main path (the chain after
// it hangs off the main path), and at a chain row whose result is not its
// draft. Later rows keep adaptive continuation's results. Then the step's P
// rows move into their slots, the window shifts, and thread 0 writes the
// next tree over the rows after the break: group 0 of each depth is the
// row's token and alternates, group i >= 1 the row's drawn tree group i.
// res_xf (unused with adaptive continuation) holds the token of every row.
__device__ void batch_epilogue_tree(const DevParams& P, int b, int32_t* out_committed, int32_t* out_ncommit,
                                    int32_t* out_firstrej, Scratch& sc) {
  const int W = P.W, K = P.K;
  const int abs0 = P.abs_pos[b];
  const uint32_t t = P.step_t[b];
  int32_t* xs = P.res_xf + static_cast<size_t>(b) * W;
  int32_t* tt = P.tree_tok + static_cast<size_t>(b) * P.tree_n;
  if (threadIdx.x == 0) {
    const int Dt = P.tree_depth[b];
    int first = -1, node = 0, off = 0, kd = K;  // off: first slot of depth r + 1, kd = K^(r+1)
    bool on_main = true;
    int r = 0;
    for (; r < W; ++r) {
      const size_t bsr = static_cast<size_t>(b) * W + (abs0 + r) % W;
      int x;
      if (r < Dt && node != 0) {
        int e = node - 1;  // node row index: depths 1..r-1 first
        for (int d = 1, k2 = K; d < r; ++d, k2 *= K) e += k2 - 1;
        x = __ldcg(P.res_node + static_cast<size_t>(b) * P.X + SJD_IDX(e, P.X));
      } else {
        x = __ldcg(P.res_x + bsr);
      }
      xs[r] = x;
      if (r < Dt) {
        int kk = -1;
        for (int k = 0; k < K && kk < 0; ++k)
          if (tt[SJD_IDX(off + node * K + k, P.tree_n)] == x) kk = k;
        if (r < Dt - 1 || Dt == W) {
          if (kk < 0) {
            first = r;
            break;
          }
          node = node * K + kk;
          on_main = on_main && kk == 0;
        } else if (!(kk == 0 && on_main)) {
          first = r;
          break;
        }
        off += kd;
        kd *= K;
      } else if (x != __ldcg(P.cand + bsr * K)) {
        first = r;
        break;
      }
    }
    for (int r2 = first < 0 ? W : first + 1; r2 < W; ++r2)
      xs[r2] = __ldcg(P.res_x + static_cast<size_t>(b) * W + (abs0 + r2) % W);
    sc.bc_i[1] = first;
  }
  __syncthreads();
  const int fr = sc.bc_i[1];
  const int nc = fr < 0 ? W : fr + 1;
  for (int j = threadIdx.x; j < W; j += blockDim.x) {
    const int v = j < nc ? xs[j] : -1;
    P.committed[static_cast<size_t>(b) * W + j] = v;
    if (out_committed) out_committed[static_cast<size_t>(b) * W + j] = v;
  }
  if (threadIdx.x == 0) {
    P.first_rej[b] = fr;
    P.n_commit[b] = nc;
    if (out_ncommit) out_ncommit[b] = nc;
    if (out_firstrej) out_firstrej[b] = fr;
  }
  // the step's P rows into their slots (every row has read the old ones)
  const size_t S = static_cast<size_t>(P.S);
  for (size_t e = threadIdx.x; e < static_cast<size_t>(W) * S; e += blockDim.x) {
    const size_t bsr = static_cast<size_t>(b) * W + e / S, i = e % S;
    if (static_cast<int>(i) < __ldcg(P.tq_len + bsr)) {
      P.q_ids[bsr * S + i] = __ldcg(P.tq_ids + bsr * S + i);
      P.q_prob[bsr * S + i] = __ldcg(P.tq_prob + bsr * S + i);
    }
  }
  for (int j = threadIdx.x; j < W; j += blockDim.x)
    P.q_len[static_cast<size_t>(b) * W + j] = __ldcg(P.tq_len + static_cast<size_t>(b) * W + j);
  __syncthreads();
  // window refill (the ring keeps a carried row's P row in its slot)
  const int new_abs = abs0 + nc;
  const int Km1 = K - 1;
  for (int r = threadIdx.x; r < W; r += blockDim.x) {
    const size_t bs = static_cast<size_t>(b) * W + (new_abs + r) % W;
    int32_t* cg = P.cand + bs * K;
    int x;
    if (r < W - nc) {
      const int j = r + nc;
      x = xs[j];
      int g = 1;
      if (fr >= 0 && j <= fr + P.D) {
        const int na = __ldcg(P.res_altn + bs);
        for (int k = 0; k < na; ++k) cg[1 + k] = __ldcg(P.res_alt + bs * Km1 + k);
        g = 1 + na;
      }
      cg[0] = x;
      P.gsize[bs] = g;
    } else {
      const uint64_t r64 = rand64(P, static_cast<uint32_t>(new_abs + r), t, static_cast<uint32_t>(b), kInit);
      x = P.lo + static_cast<int>(__umul64hi(r64, static_cast<unsigned long long>(P.veff)));
      cg[0] = x;
      P.gsize[bs] = 1;
      P.q_len[bs] = -1;
    }
    P.win_tok[static_cast<size_t>(b) * W + r] = x;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    P.last_tok[b] = xs[nc - 1];
    P.abs_pos[b] = new_abs;
    P.step_t[b] = t + 1;
    // the next tree, over the old rows fr + 1 .. fr + depth
    for (int i = 0; i < P.tree_n; ++i) tt[i] = -1;
    const int depth = fr < 0 ? 0 : min(P.D, W - 1 - fr);
    int off_up = 0, off = 0, kd = 1;  // kd = K^(dl-1) parents, off_up: their first slot
    for (int dl = 1; dl <= depth; ++dl) {
      const int j = fr + dl;
      const size_t sj = static_cast<size_t>(b) * W + (abs0 + j) % W;
      for (int i = 0; i < kd; ++i) {
        const bool parent = dl == 1 ? i == 0 : tt[SJD_IDX(off_up + i, P.tree_n)] >= 0;
        if (!parent) continue;
        if (i == 0) {
          tt[SJD_IDX(off, P.tree_n)] = xs[j];
          const int na = __ldcg(P.res_altn + sj);
          for (int k = 0; k < na; ++k) tt[SJD_IDX(off + 1 + k, P.tree_n)] = __ldcg(P.res_alt + sj * Km1 + k);
        } else {
          const int32_t* src = P.res_tree + sj * static_cast<size_t>(P.tree_g) * K +
                               static_cast<size_t>(SJD_IDX(i - 1, P.tree_g)) * K;
          for (int k = 0; k < K; ++k) tt[SJD_IDX(off + i * K + k, P.tree_n)] = __ldcg(src + k);
        }
      }
      off_up = off;
      off += kd * K;
      kd *= K;
    }
    P.tree_depth[b] = depth;
    P.ticket[b] = 0;
    atomicAdd(&P.stats[3], b == 0 ? 1ull : 0ull);
  }
}

}  // namespace
}  // namespace sjd
