"""CPU oracle of one SJD-PAC Jacobi step (verify + adaptive continuation +
proactive drafting + window refill) and of the decode loop around it.

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference leg may import, call or run anything in oracle/.
The product (the CUDA library and its Python binding) never does, and
shares no code, header, table or constant generator with this file.

Method: Kang et al., "SJD-PAC: Accelerating Speculative Jacobi Decoding via
Proactive Drafting and Adaptive Continuation" (CVPR 2026). Citations name the
paper's sections, equations, algorithm and theorems:
  Sec. 3.2   rejection sampling: accept x ~ q iff u < p(x)/q(x), else draw
             from max(p - q, 0) renormalised (Eq. 1, the Rejection Sampling
             Lemma of Appendix A.1).
  Sec. 3.3   SJD: window of L tokens, one forward gives P^t, verify
             sequentially, append as many fresh tokens as were committed.
  Sec. 4.1   Proactive Drafting: after the first rejection at i, K candidates
             without replacement from p(.|X^{t-1}_{<j}) for j = i+1..i+D.
  Sec. 4.2   Adaptive Continuation: no break; every later position is tested
             against its stale (p_j, q_j), accepted tokens kept, rejected ones
             redrawn from the residual.
  Alg. 1     the full step; returns X^t and P^t (P^t becomes the next q).
  Thm. 1/2   (Appendix A) losslessness of AC and of sequential verification
             of K without-replacement candidates with adjusted q^(k) and
             residual p^(k+1).

Arithmetic. The paper fixes no precision. This file is the kernel-precision
specification: it writes out, operation by operation, the arithmetic the
GPU kernels perform, so that they can be compared with it bit for bit. (The
plain real-number definition, in float64, is oracle/sjd_fp64.py; tests
compare the kernels with it at the tolerance of near-ties.) Two stages:

Stage 1 (the cuts; IEEE fp32, round to nearest after every operation, a
fused multiply-add FMA(a, b, c) = a*b + c rounded once):
  logits   l_v = FMA(s, fl(C_v - U_v), U_v)  (s == 1 or no uncond: l = C),
           then l_v = fl(l_v / T) when T != 1, over the allowed ids [lo, hi).
  order    v before w iff l_v > l_w, or l_v == l_w and v < w.
  top-k    the first min(k, V_eff) ids in that order (k <= 0: all).
  weights  m = largest l; e_v = EXP(fl(l_v - m)) with the EXP below;
           E1_v = rint(e_v * 2^47) as an integer; Z1 = sum E1_v (exact).
  top-p    (tau < 1) the shortest prefix, in the order above, whose integer
           weight sum satisfies W >= tau * Z1 (tau as its exact fp32 value).
Stage 2 (the kept ids; every decision):
  kept     the ids inside both cuts whose precise weight E_v below is > 0.
  E_v      round(2^47 exp(t_v)) with t_v = (U + s (C - U)) / T - m taken
           exactly from the inputs in double-float arithmetic (each value
           an unevaluated sum of two fp32) and exp to about 1e-12 relative:
           see precise_weights(). Z = sum E_v over the kept ids (exact).
  probs    p_v = fl(fl(E_v) * 2^-47 / Wz), Wz = fl32(fl64(Z) * 2^-47).
  accept   candidate k (weights W of p^(k), sum Wsum; W = E at k = 1)
           with uniform u = (2m+1)/2^24 is accepted iff
           fl64(fl64(u q(c)) fl64(Wsum)) < fl64(W_c) d, where d = 1 -
           (fp64 sum of q over the rejected candidates), so d = 1 at k = 1.
  residual k = 1: R_v = max(0, E_v - ceil(q_v Z)) (exact integers);
           k > 1: R_v = max(0, W_v - ceil(q_v A)) with A = fl64(fl64(Wsum)
           / d) (one division per level; the ceiling exact) for ids not yet
           rejected, R_v = W_v for the rejected ones.
  draw     with integer weights w over ascending ids and u = (2m+1)/2^24:
           the first id whose inclusive prefix sum exceeds floor(u * sum w).
  relaxed  (optional, lossy; off by default) with token groups given, W_c in
           the acceptance test is the weight of c's whole group among the
           kept ids; a kept token may then lie outside its next draft row,
           and q(c) = 0 is no error there (the test accepts iff W_c > 0);
           everything else is unchanged.

EXP (stage 1) is written from the mathematics (base-2 range reduction after
Cody & Waite, "Software Manual for the Elementary Functions", 1980, with the
Taylor series of 2^f): a = fl(t * log2e), n = rint(a), f = fl(a - n)
(exact, |f| <= 1/2), 2^f by Horner on the Taylor coefficients (ln 2)^k / k!,
k = 1..7, each step FMA(y, f, c); result 2^n * poly (exact scaling). For
a < -64 the result is 0 (it would quantise to E = 0 anyway).
"""

import math
from dataclasses import dataclass, field
from fractions import Fraction

import numpy as np

from . import philox as px

FIX_BITS = 47                       # weights are integers in units of 2^-47
_FIX_SCALE = float(1 << FIX_BITS)
_FIX_INV = 1.0 / _FIX_SCALE

_LOG2E = np.float32(1.4426950408889634)
_TAYLOR = [np.float32(math.log(2.0) ** k / math.factorial(k)) for k in range(1, 8)]


def fma32(a, b, c):
    """FMA(a, b, c): a*b + c of fp32 values rounded once to fp32 (elementwise).

    a*b is exact in fp64 (two 24-bit significands). The fp64 sum s is made
    round-to-odd (Boldo & Melquiond, "Emulation of FMA and correctly rounded
    sums: proved algorithms using rounding to odd", IEEE TC 2008): Knuth's
    TwoSum gives the exact error e of s, and an inexact s with an even last
    bit moves one fp64 step toward e. Rounding that value to fp32 (53 >= 24 + 2
    bits) is the correctly rounded a*b + c.
    """
    a64 = np.asarray(a, dtype=np.float32).astype(np.float64)
    b64 = np.asarray(b, dtype=np.float32).astype(np.float64)
    c64 = np.asarray(c, dtype=np.float32).astype(np.float64)
    p = a64 * b64
    with np.errstate(invalid="ignore", over="ignore"):
        s = p + c64
        bv = s - p
        av = s - bv
        e = (p - av) + (c64 - bv)
        odd = (np.asarray(s).view(np.int64) & 1) == 1
        fix = np.isfinite(s) & np.isfinite(e) & (e != 0) & ~odd
        s = np.where(fix, np.nextafter(s, np.where(e > 0, np.inf, -np.inf)), s)
    return np.asarray(s).astype(np.float32)


# ---------------------------------------------------------------------------
# Stage 2: the precise weights. Constants are computed here from series in
# exact integer arithmetic (units of 2^-256) and rounded to fp32 exactly.

_FP = 256


def _nearest_f32(x):
    """The fp32 value (as a float) nearest to the rational x, half to even
    (x zero or in the fp32 normal range)."""
    x = Fraction(x)
    if x == 0:
        return 0.0
    a = abs(x)
    e = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** e > a:
        e -= 1
    if Fraction(2) ** (e + 1) <= a:
        e += 1
    ulp = Fraction(2) ** (e - 23)
    q, r = divmod(a / ulp, 1)
    q = int(q)
    if r > Fraction(1, 2) or (r == Fraction(1, 2) and q % 2 == 1):
        q += 1
    return float((1 if x > 0 else -1) * q * ulp)


def _split_f32(x):
    """(hi, lo): fp32 nearest to x, and fp32 nearest to x - hi."""
    hi = _nearest_f32(x)
    return np.float32(hi), np.float32(_nearest_f32(Fraction(x) - Fraction(hi)))


def _ln2_units():
    """ln 2 = sum over k >= 1 of 1 / (k 2^k), in units of 2^-_FP."""
    one = 1 << _FP
    return sum(one // (k << k) for k in range(1, _FP + 16))


def _exp_units(x):
    """e^x for |x| <= 1/2 given in units of 2^-_FP, by its Taylor series."""
    one = 1 << _FP
    term, total = one, one
    for n in range(1, 120):
        term = (term * x) // (one * n)
        total += term
    return total


_LN2_U = _ln2_units()
_LN2_HI, _LN2_LO = _split_f32(Fraction(_LN2_U, 1 << _FP))
_LOG2E_HI, _LOG2E_LO = _split_f32(Fraction(1 << _FP, _LN2_U))
_EXP2_HI, _EXP2_LO = (np.array(v, np.float32) for v in zip(
    *[_split_f32(Fraction(_exp_units(j * _LN2_U // 64), 1 << _FP)) for j in range(-32, 33)]))
_INV6, _INV24, _INV120 = (np.float32(_nearest_f32(Fraction(1, d))) for d in (6, 24, 120))
_MAGIC = np.float32(1.5 * 2 ** 23)
_MAGIC_BITS = int(np.array([_MAGIC]).view(np.uint32)[0])


def _f32(x):
    return np.asarray(x, dtype=np.float32)


def two_sum(a, b):
    """Knuth's TwoSum in fp32: a + b = s + e exactly (elementwise)."""
    a, b = _f32(a), _f32(b)
    with np.errstate(invalid="ignore"):         # infinite inputs give NaN errors
        s = a + b
        ap = s - b
        bp = s - ap
        return s, (a - ap) + (b - bp)


def _fix_mag(x, k):
    """|x| 2^k truncated toward zero for normal or zero fp32 x, uint64."""
    b = _f32(x).view(np.uint32).astype(np.int64)
    ex = (b >> 23) & 0xFF
    mnt = ((b & 0x7FFFFF) | 0x800000).astype(np.uint64)
    sh = ex - 150 + np.asarray(k, np.int64)
    up = np.where(sh >= 0, sh, 0).astype(np.uint64)
    dn = np.where((sh < 0) & (sh > -32), -sh, 0).astype(np.uint64)
    v = np.where(sh >= 0, mnt << up, np.where(sh > -32, mnt >> dn, np.uint64(0)))
    return np.where(ex == 0, np.uint64(0), v).astype(np.uint64)


def exp_weight_df(th, tl):
    """round(2^47 exp(th + tl)) as uint64 (0 below t = -44): x = t log2(e)
    = n + j/64 + g (|g| <= 1/128) in double-float, e^(g ln 2) by its Taylor
    series to the fifth power, times 2^(j/64) from the double-float table,
    then (rh + rl) 2^(47 + n) rounded with 16 fractional bits."""
    th, tl = _f32(th), _f32(tl)
    xh = th * _LOG2E_HI
    xe = fma32(th, _LOG2E_HI, -xh)
    xl = fma32(th, _LOG2E_LO, fma32(tl, _LOG2E_HI, xe))
    dead = ~(xh >= np.float32(-64.0))
    xh = np.where(dead, np.float32(0.0), xh).astype(np.float32)
    xl = np.where(dead, np.float32(0.0), xl).astype(np.float32)
    rn = xh + _MAGIC
    n = rn - _MAGIC
    ni = rn.view(np.uint32).astype(np.int64) - _MAGIC_BITS
    fh = xh - n
    rj = fh * np.float32(64.0) + _MAGIC
    jf = rj - _MAGIC
    ji = rj.view(np.uint32).astype(np.int64) - _MAGIC_BITS
    gh = fma32(jf, np.float32(-2.0 ** -6), fh)
    yh = gh * _LN2_HI
    ye = fma32(gh, _LN2_HI, -yh)
    yl = fma32(gh, _LN2_LO, fma32(xl, _LN2_HI, ye))
    y1 = yh + yl                                  # the polynomial's argument
    pp = fma32(y1, _INV120, _INV24)
    pp = fma32(pp, y1, _INV6)
    pp = fma32(pp, y1, np.float32(0.5))
    q = (y1 * y1) * pp
    sh = np.float32(1.0) + yh
    se = yh - (sh - np.float32(1.0))
    sl = se + (yl + q)
    Th, Tl = _EXP2_HI[ji + 32], _EXP2_LO[ji + 32]
    rh = Th * sh
    re = fma32(Th, sh, -rh)
    rl = fma32(Th, sl, fma32(Tl, sh, re))
    k = 47 + ni + 16
    a = _fix_mag(rh, k)
    lo = _fix_mag(rl, k)
    neg = (_f32(rl).view(np.uint32) >> 31) == 1
    f = np.where(neg, a - lo, a + lo)
    E = (f + np.uint64(0x8000)) >> np.uint64(16)
    return np.where(dead, np.uint64(0), E).astype(np.uint64)


def precise_weights(c, u, s, T, m, cfg, temp):
    """Stage-2 weights of ids with raw inputs c (cond) and u (uncond):
    t = (u + s (c - u)) / T - m in double-float (c alone without guidance,
    no division when T == 1), then exp_weight_df(t)."""
    c = _f32(c)
    if cfg:
        u, s = _f32(u), np.float32(s)
        dh, dl = two_sum(c, -u)
        ph = s * dh
        pe = fma32(s, dh, -ph)
        pe = fma32(s, dl, pe)
        lh, le = two_sum(u, ph)
        ll = le + pe
    else:
        lh, ll = c, np.zeros_like(c)
    if temp:
        T = np.float32(T)
        qh = lh / T
        r = fma32(-qh, T, lh)
        ll = (r + ll) / T
        lh = qh
    th, te = two_sum(lh, -np.float32(m))
    return exp_weight_df(th, te + ll)


class OracleError(Exception):
    """A condition the GPU path reports through its status word."""


class NonFiniteLogits(OracleError):
    pass


class InvalidDraft(OracleError):
    pass


@dataclass
class Params:
    """Problem statement of one decode (Sec. 3.3 and 4; defaults of Sec. 5.1)."""
    batch: int
    window: int                 # L of the paper (W here)
    vocab: int
    lo: int = 0                 # allowed (image-token) ids [lo, hi)
    hi: int = -1
    cfg_scale: float = 3.0
    temperature: float = 1.0
    top_k: int = 2000
    top_p: float = 1.0
    pd_k: int = 4               # K
    pd_depth: int = 3           # D
    ac: int = 1                 # 1: adaptive continuation, 0: vanilla SJD
    seed: int = 0
    tree: int = 0               # 1: the full K-ary proactive-drafting tree

    def __post_init__(self):
        if self.hi < 0:
            self.hi = self.vocab

    @property
    def v_eff(self):
        return self.hi - self.lo


# ---------------------------------------------------------------------------
# S1-S4: processed target distribution of one row (Sec. 5.1: CFG weight,
# temperature, top-k logit sampler; top-p and the id mask are workload
# parameters). The result is the sparse row p (ascending id).

def combine_logits(cond, uncond, cfg_scale, temperature):
    """Classifier-free-guidance combine in logit space, then temperature.

    cond/uncond: fp32 arrays over the allowed ids (exact values of the
    fp32 or bf16 inputs). uncond None means no guidance (l = cond).
    """
    c = np.asarray(cond, dtype=np.float32)
    s = np.float32(cfg_scale)
    if uncond is None or s == np.float32(1.0):
        l = c.copy()
    else:
        u = np.asarray(uncond, dtype=np.float32)
        l = fma32(s, (c - u).astype(np.float32), u)   # fl(c - u), then one FMA
    T = np.float32(temperature)
    if T != np.float32(1.0):
        l = l / T
    return l


def exp_neg(t):
    """EXP of the definition above for fp32 arguments t <= 0 (fp32 result)."""
    t = np.asarray(t, dtype=np.float32)
    a = t * _LOG2E
    tiny = ~(a >= np.float32(-64.0))          # also catches -inf
    a = np.where(tiny, np.float32(0.0), a).astype(np.float32)
    n = np.rint(a)
    f = (a - n).astype(np.float32)
    y = np.full_like(f, _TAYLOR[6])
    for c in reversed(_TAYLOR[:6]):
        y = fma32(y, f, c)
    y = fma32(y, f, np.float32(1.0))
    e = np.ldexp(y, n.astype(np.int32)).astype(np.float32)
    e[tiny] = np.float32(0.0)
    return e


def quantize(x32):
    """rint(x * 2^47) of non-negative fp32 values, as uint64 (half to even)."""
    return np.rint(np.asarray(x32, dtype=np.float32).astype(np.float64) * _FIX_SCALE).astype(np.uint64)


def dequantize(w):
    """w * 2^-47 as fp32; exact for every weight made by quantize()."""
    return (np.asarray(w, dtype=np.uint64).astype(np.float64) * _FIX_INV).astype(np.float32)


def fix_to_f32(total):
    """fl32(fl64(total) * 2^-47) of an exact integer sum."""
    return np.float32(float(int(total)) * _FIX_INV)


@dataclass
class Row:
    """Sparse processed distribution p of one row, ascending ids."""
    ids: np.ndarray        # int64
    E: np.ndarray          # uint64 integer weights
    p: np.ndarray          # fp32 probabilities
    Z: int                 # sum of E
    p64: np.ndarray = None  # fp64 softmax over the same ids (ideal values)


@dataclass
class UniformQ:
    """Draft distribution of a freshly appended position (uniform on [lo,hi))."""
    lo: int
    hi: int


def process_row(l, lo, top_k, top_p, raw=None):
    """Row l (stage-1 fp32 logits over ids lo..lo+len-1) -> Row.

    raw = (C, U, s, T): the row's raw inputs over the same ids (U None
    without guidance) from which the kept ids' precise weights are taken;
    None means that l itself holds the exact logits (no guidance, T = 1).
    """
    l = np.asarray(l, dtype=np.float32)
    n = l.shape[0]
    if np.isnan(l).any() or np.isposinf(l).any():
        raise NonFiniteLogits("NaN or +inf logit in the allowed range")
    ids = np.arange(lo, lo + n, dtype=np.int64)
    order = np.lexsort((ids, -l.astype(np.float64)))     # l desc, id asc
    kk = n if top_k <= 0 else min(int(top_k), n)
    sel = order[:kk]
    m = l[sel[0]]
    if not np.isfinite(m):
        raise NonFiniteLogits("no finite logit in the allowed range")
    # stage 1: the cuts
    tau = np.float32(top_p)
    if tau < np.float32(1.0):
        E1 = quantize(exp_neg((l[sel] - m).astype(np.float32)))
        Z1 = int(E1.sum(dtype=np.uint64))
        target = math.ceil(Fraction(float(tau)) * Z1)
        cum = np.cumsum(E1, dtype=np.uint64)
        cut = int(np.searchsorted(cum, np.uint64(target), side="left"))
        sel = sel[:cut + 1]
    # stage 2: precise weights of the kept ids
    if raw is None:
        E = precise_weights(l[sel], None, 1.0, 1.0, m, False, False)
    else:
        C, U, s, T = raw
        cfg = U is not None and np.float32(s) != np.float32(1.0)
        E = precise_weights(np.asarray(C, np.float32)[sel], None if not cfg else np.asarray(U, np.float32)[sel],
                            s, T, m, cfg, np.float32(T) != np.float32(1.0))
    live = E > 0                    # zero-weight ids have p = 0: not stored
    sel, E = sel[live], E[live]
    Z = int(E.sum(dtype=np.uint64))
    Wz = fix_to_f32(Z)
    e32 = (E.astype(np.float64).astype(np.float32) * np.float32(2.0 ** -47)).astype(np.float32)
    p = (e32 / Wz).astype(np.float32)
    by_id = np.argsort(ids[sel], kind="stable")
    sel, E, p = sel[by_id], E[by_id], p[by_id]
    l64 = l[sel].astype(np.float64)
    w64 = np.exp(l64 - l64.max())
    return Row(ids=ids[sel], E=E, p=p, Z=Z, p64=w64 / w64.sum())


def uniform_q_value(lo, hi):
    return np.float32(1.0) / np.float32(hi - lo)


def q_at(q, v):
    """q(v) (fp32) of a stored draft distribution."""
    if isinstance(q, UniformQ):
        return uniform_q_value(q.lo, q.hi) if q.lo <= v < q.hi else np.float32(0.0)
    i = int(np.searchsorted(q.ids, v))
    if i < q.ids.shape[0] and int(q.ids[i]) == int(v):
        return q.p[i]
    return np.float32(0.0)


def q_on(q, ids):
    """q(v) (fp32) for every v in ids."""
    ids = np.asarray(ids, dtype=np.int64)
    if isinstance(q, UniformQ):
        inside = (ids >= q.lo) & (ids < q.hi)
        return np.where(inside, uniform_q_value(q.lo, q.hi), np.float32(0.0)).astype(np.float32)
    if q.ids.shape[0] == 0:
        return np.zeros(ids.shape, dtype=np.float32)
    i = np.minimum(np.searchsorted(q.ids, ids), q.ids.shape[0] - 1)
    return np.where(q.ids[i] == ids, q.p[i], np.float32(0.0)).astype(np.float32)


# ---------------------------------------------------------------------------
# S5/S7: acceptance test, residual resample (Sec. 3.2, Eq. 1, Thm. 1) and
# sequential verification of K without-replacement candidates (Thm. 2).

def inv_cdf(weights, total, odd24):
    """Index of the first entry whose inclusive prefix sum exceeds
    floor(u * total), u = odd24 / 2^24, over integer weights in id order."""
    T = (int(odd24) * int(total)) >> 24
    cum = np.cumsum(np.asarray(weights, dtype=np.uint64), dtype=np.uint64)
    return int(np.searchsorted(cum, np.uint64(T), side="right"))


def accept_exact(odd24, q_c, Wsum, Wc, d):
    """u < p^(k)(c) / q^(k)(c) with p^(k)(c) = Wc / Wsum and q^(k)(c) =
    q_c / d, as fl64(fl64(u q_c) fl64(Wsum)) < fl64(Wc) d (Alg. 1, Thm. 2);
    u q_c is exact, and at the first level d = 1."""
    u = int(odd24) / float(1 << 24)
    return (u * float(q_c)) * float(int(Wsum)) < float(int(Wc)) * d


def _ceil_q_times(q, total):
    """ceil(q * total) exactly, q an fp32 value in [0, 1]."""
    fr = Fraction(float(q))
    return -((-fr.numerator * int(total)) // fr.denominator)


def residual_first(E, q, Z):
    """max(0, E - ceil(q Z)): weight of p - q at the first level."""
    c = _ceil_q_times(q, Z)
    return int(E) - c if int(E) > c else 0


def level_scale(Wsum, d):
    """A = fl64(fl64(Wsum) / d) of a later level, as (A_fix, G) with
    A = A_fix 2^-G exactly and A_fix in [2^62, 2^63)."""
    A = float(int(Wsum)) / d
    G = 62 - (math.frexp(A)[1] - 1)
    return int(math.ldexp(A, G)), G


def residual_level(W, q, A_fix, G):
    """max(0, W - ceil(q A)) with A = A_fix 2^-G: weight of p^(k) - q^(k) at
    a later level (q^(k) = q / d, so q^(k) Wsum = q A)."""
    fr = Fraction(float(q))
    if fr == 0:
        return int(W)
    c = -((-fr.numerator * A_fix) // (fr.denominator << G) if G >= 0 else
          (-fr.numerator * A_fix << -G) // fr.denominator)
    return int(W) - c if c < int(W) else 0


def verify_group(prow, q, cands, odd_acc, odd_res, groups=None):
    """Verify candidates c_1..c_g of one row against target prow (Thm. 2;
    g = 1 is the single-draft test of Sec. 3.2 / Alg. 1).

    q is the row's stored draft distribution P^{t-1}_j; the candidates were
    drawn from it without replacement. p^(k) is held as integer weights W
    (W = E at k = 1). Returns (token, k) with k the 1-based index of the
    accepted candidate, or 0 when the token was drawn from the final
    residual p^(g+1). groups (optional, lossy): token groups over the
    vocabulary; the test then takes W_c as the weight of c's whole group
    among the kept ids (the relaxed acceptance).
    """
    ids = prow.ids
    pos = {int(v): i for i, v in enumerate(ids)}
    qP = q_on(q, ids)                           # q over the support of p
    W = [int(e) for e in prow.E]
    Wsum = int(prow.Z)
    removed = [False] * ids.shape[0]
    S = 0.0                                     # q mass of the rejected candidates (fp64)
    g = len(cands)
    R, Rsum = W, Wsum
    for k in range(1, g + 1):
        c = int(cands[k - 1])
        q_c = q_at(q, c)
        if q_c == np.float32(0.0) and groups is None:
            raise InvalidDraft("draft token has zero draft probability")
        d = 1.0 - S
        i = pos.get(c)
        if groups is None:
            Wc = W[i] if i is not None else 0
        else:
            gc = groups[c]
            Wc = sum(W[v] for v in range(len(W)) if groups[int(ids[v])] == gc)
        if accept_exact(odd_acc[k - 1], q_c, Wsum, Wc, d):
            return c, k
        # rejected: residual p^(k+1) proportional to max(0, p^(k) - q^(k))
        if k == 1:
            R = [residual_first(W[v], qP[v], Wsum) for v in range(len(W))]
        else:
            A_fix, G = level_scale(Wsum, d)
            R = [W[v] if removed[v] else residual_level(W[v], qP[v], A_fix, G) for v in range(len(W))]
        Rsum = sum(R)
        if Rsum == 0:                  # only reachable through rounding
            R, Rsum = W, Wsum
        if k == g:
            break
        # adjusted draft q^(k+1): c_1..c_k removed, renormalised
        S = S + float(q_c)
        if i is not None:
            removed[i] = True
        if not 1.0 - S > 0.0:
            break                      # no draft mass left for more candidates
        W, Wsum = R, Rsum
    return int(ids[inv_cdf(np.array(R, dtype=np.uint64), Rsum, odd_res)]), 0


def sample_row(prow, odd24):
    """One draw from p itself (integer weights E)."""
    return int(prow.ids[inv_cdf(prow.E, prow.Z, odd24)])


def draw_alternates(prow, first, odds):
    """Proactive drafting (Sec. 4.1): candidates c_2.. drawn without
    replacement from p, c_1 = first excluded. Stops when no mass is left."""
    w = prow.E.copy()
    pos = np.searchsorted(prow.ids, first)
    if pos < w.shape[0] and int(prow.ids[pos]) == int(first):
        w[pos] = np.uint64(0)
    out = []
    for odd in odds:
        tot = int(w.sum(dtype=np.uint64))
        if tot == 0:
            break
        i = inv_cdf(w, tot, odd)
        out.append(int(prow.ids[i]))
        w[i] = np.uint64(0)
    return out


# ---------------------------------------------------------------------------
# Decode state, the step (S1-S9) and the loop (Sec. 3.3, Alg. 1).

@dataclass
class BatchState:
    abs_pos: int                        # absolute position of window row 0
    cands: list                         # per row: [c_1 (the draft), c_2, ...]
    q: list                             # per row: Row or UniformQ (P^{t-1}_j)
    last_token: int = 0                 # token before row 0 (0 at the start)
    batch_index: int = 0                # b of the Philox counters
    tree: list = field(default_factory=list)   # full tree: tree[r][i] = children of node i at depth r


def fresh_draft(params, b, abs_pos, step):
    """Draft of a newly appended position: uniform on [lo, hi) (Sec. 3.3)."""
    r = px.raw64(params.seed, abs_pos, step, b, px.INIT)
    return params.lo + ((r * params.v_eff) >> 64)


def init_state(params, step=0, batch_ids=None):
    """Window of W fresh positions 0..W-1 with uniform draft distributions,
    for batch elements batch_ids (default: all)."""
    out = []
    for b in (range(params.batch) if batch_ids is None else batch_ids):
        cands = [[fresh_draft(params, b, j, step)] for j in range(params.window)]
        q = [UniformQ(params.lo, params.hi) for _ in range(params.window)]
        out.append(BatchState(abs_pos=0, cands=cands, q=q, last_token=0, batch_index=b))
    return out


def _restrict(x, params):
    return np.asarray(x, dtype=np.float32)[..., params.lo:params.hi]


def draft_from_logits(params, states, step, qcond, quncond=None):
    """Set every row's draft distribution from draft logits and sample its
    draft from it (purpose SYNTH). quncond None: no guidance."""
    for i, st in enumerate(states):
        b = st.batch_index
        for j in range(params.window):
            qc = _restrict(qcond[i, j], params)
            qu = None if quncond is None else _restrict(quncond[i, j], params)
            s = params.cfg_scale if quncond is not None else 1.0
            l = combine_logits(qc, qu, s, params.temperature)
            row = process_row(l, params.lo, params.top_k, params.top_p, (qc, qu, s, params.temperature))
            odd, _ = px.uniform(params.seed, st.abs_pos + j, step, b, px.SYNTH, 0)
            st.q[j] = row
            st.cands[j] = [sample_row(row, odd)]
    return states


@dataclass
class BatchResult:
    x: list                 # x_j^t of every row (after AC / vanilla tail)
    dev: list               # x_j^t != c_1(j)
    first_dev: int          # first_rej_idx of Alg. 1 (0-based; -1 = none)
    n_commit: int
    committed: list
    rows: list              # processed p rows (P^t)
    accepted_k: list        # per row: accepted candidate index or 0


def step(params, states, step_idx, cond, uncond, groups=None):
    """One Jacobi iteration of Alg. 1 on every batch element.

    cond/uncond: arrays [len(states), W, V] holding the exact fp32 values of
    the logits P^t = M(X^{t-1}) (uncond may be None when cfg_scale == 1).
    Mutates `states` into the next window and returns per-batch results.
    """
    seed, W, K, D = params.seed, params.window, params.pd_k, params.pd_depth
    results = []
    for i, st in enumerate(states):
        b = st.batch_index
        xs, devs, rows, ks, alts, xf, altsf = [], [], [], [], [], [], []
        for j in range(W):
            a = st.abs_pos + j
            cj = _restrict(cond[i, j], params)
            uj = None if uncond is None else _restrict(uncond[i, j], params)
            l = combine_logits(cj, uj, params.cfg_scale, params.temperature)
            prow = process_row(l, params.lo, params.top_k, params.top_p,
                               (cj, uj, params.cfg_scale, params.temperature))
            cands = st.cands[j]
            odd_acc = [px.uniform(seed, a, step_idx, b, px.ACCEPT, k)[0] for k in range(len(cands))]
            odd_res = px.uniform(seed, a, step_idx, b, px.RESIDUAL, 0)[0]
            x, k = verify_group(prow, st.q[j], cands, odd_acc, odd_res, groups)
            odd_pd = [px.uniform(seed, a, step_idx, b, px.PD, kk)[0] for kk in range(1, K)]
            xs.append(x)
            ks.append(k)
            devs.append(x != cands[0])
            rows.append(prow)
            alts.append(draw_alternates(prow, x, odd_pd))
            if not params.ac:
                f = sample_row(prow, odd_res)      # vanilla SJD tail: fresh draw from p_j
                xf.append(f)
                altsf.append(draw_alternates(prow, f, odd_pd))
        first_dev = next((j for j in range(W) if devs[j]), -1)
        if not params.ac and first_dev >= 0:
            for j in range(first_dev + 1, W):
                xs[j], alts[j], ks[j] = xf[j], altsf[j], 0
        n_commit = W if first_dev < 0 else first_dev + 1
        committed = xs[:n_commit]
        # window refill (Sec. 3.3) with PD groups on the first D rows (Sec. 4.1)
        new_cands, new_q = [], []
        for r in range(W - n_commit):
            j = r + n_commit
            group = [xs[j]]
            if first_dev >= 0 and j <= first_dev + D:
                group += alts[j]
            new_cands.append(group)
            new_q.append(rows[j])
        new_pos = st.abs_pos + n_commit
        for r in range(W - n_commit, W):
            new_cands.append([fresh_draft(params, b, new_pos + r, step_idx)])
            new_q.append(UniformQ(params.lo, params.hi))
        results.append(BatchResult(x=xs, dev=devs, first_dev=first_dev, n_commit=n_commit,
                                   committed=committed, rows=rows, accepted_k=ks))
        st.abs_pos = new_pos
        st.cands, st.q = new_cands, new_q
        st.last_token = committed[-1]
    return results


def window_tokens(states):
    """Main-path tokens of every window, [B][W] (the forward's input)."""
    return [[c[0] for c in st.cands] for st in states]


def decode(params, n_tokens, forward, max_steps, start_step=0, states=None):
    """Jacobi decode until every batch element has n_tokens committed.

    forward(window [B][W], prev [B], abs_pos [B]) -> (cond, uncond) arrays
    [B, W, V] is the model (out of scope here: a stand-in supplied by the
    caller). Returns (grid [B][n_tokens], accept_len [steps][B], steps).
    """
    if states is None:
        states = init_state(params, start_step)
    grid = [[-1] * n_tokens for _ in range(params.batch)]
    accept_len = []
    t = start_step
    nsteps = 0
    while any(st.abs_pos < n_tokens for st in states):
        if nsteps >= max_steps:
            raise OracleError("step limit")
        prev = [st.last_token for st in states]
        pos = [st.abs_pos for st in states]
        cond, uncond = forward(window_tokens(states), prev, pos)
        res = step(params, states, t, cond, uncond)
        lens = []
        for b, r in enumerate(res):
            base = pos[b]
            take = max(0, min(r.n_commit, n_tokens - base))
            for i in range(take):
                grid[b][base + i] = r.committed[i]
            lens.append(take)
        accept_len.append(lens)
        t += 1
        nsteps += 1
    return grid, accept_len, nsteps


# ---------------------------------------------------------------------------
# The full K-ary proactive-drafting tree (Sec. 4.1): after a first rejection
# at f, node i at depth d (window row d - 1 of the next step) has the
# children i K .. i K + K - 1 at depth d + 1; group 0 of each depth is the
# main path's (adaptive continuation's token and its K - 1 alternates), any
# other group K draws without replacement from the position's target with
# purpose TREE, lane i K + k. Nodes off the main path at depths 1..D-1 get
# logit rows after the W window rows: node i at depth d is row
# W + extra_row(K, d, i).

def n_extra(K, D):
    return sum(K ** d - 1 for d in range(1, D))


def extra_row(K, d, i):
    return sum(K ** e - 1 for e in range(1, d)) + (i - 1)


def tree_group(prow, odds):
    """K draws without replacement from p (integer weights E)."""
    w = prow.E.copy()
    out = []
    for odd in odds:
        tot = int(w.sum(dtype=np.uint64))
        if tot == 0:
            break
        i = inv_cdf(w, tot, odd)
        out.append(int(prow.ids[i]))
        w[i] = np.uint64(0)
    return out


def step_tree(params, states, step_idx, cond, uncond):
    """One Jacobi iteration with the full tree (adaptive continuation on) on
    every batch element; cond / uncond are [len(states), W + n_extra, V].
    The traversal starts at the root; at row r the current node's children
    are verified against the node's own target (Thm. 2) and the traversal
    moves to the child whose token is the result. The context breaks where
    no child carries it, or at the last tree row when the path has left the
    main path; later rows keep adaptive continuation's main-path result."""
    seed, W, K, D = params.seed, params.window, params.pd_k, params.pd_depth
    results = []
    for bi, st in enumerate(states):
        b = st.batch_index

        def prow_of(r):
            cj = _restrict(cond[bi, r], params)
            uj = None if uncond is None else _restrict(uncond[bi, r], params)
            l = combine_logits(cj, uj, params.cfg_scale, params.temperature)
            return process_row(l, params.lo, params.top_k, params.top_p, (cj, uj, params.cfg_scale, params.temperature))

        def verify_at(r, prow, group):
            a = st.abs_pos + r
            odd_acc = [px.uniform(seed, a, step_idx, b, px.ACCEPT, k)[0] for k in range(len(group))]
            odd_res = px.uniform(seed, a, step_idx, b, px.RESIDUAL, 0)[0]
            return verify_group(prow, st.q[r], group, odd_acc, odd_res)

        rows = [prow_of(j) for j in range(W)]
        main = [verify_at(j, rows[j], st.cands[j]) for j in range(W)]
        Dt = len(st.tree)
        xs, ks = [], []
        first, node, on_main, r = -1, 0, True, 0
        while r < W:
            if r < Dt and node != 0:
                x, k = verify_at(r, prow_of(W + extra_row(K, r, node)), st.tree[r][node])
            else:
                x, k = main[r]
            xs.append(x)
            ks.append(k)
            if r < Dt:
                group = st.tree[r][node]
                kk = group.index(x) if x in group else -1
                if r < Dt - 1 or Dt == W:
                    if kk < 0:
                        first = r
                        break
                    node, on_main = node * K + kk, on_main and kk == 0
                elif not (kk == 0 and on_main):
                    first = r
                    break
            elif x != st.cands[r][0]:
                first = r
                break
            r += 1
        n_commit = W if first < 0 else first + 1
        committed = xs[:n_commit]
        x_all = xs[:n_commit] + [main[j][0] for j in range(n_commit, W)]
        k_all = ks[:n_commit] + [main[j][1] for j in range(n_commit, W)]
        depth = 0 if first < 0 else min(D, W - 1 - first)
        new_tree, parents = [], [0]
        for dlt in range(1, depth + 1):
            j = first + dlt
            a = st.abs_pos + j
            groups = [[] for _ in range(K ** (dlt - 1))]
            for i in parents:
                if i == 0:
                    odd_pd = [px.uniform(seed, a, step_idx, b, px.PD, kk)[0] for kk in range(1, K)]
                    groups[0] = [x_all[j]] + draw_alternates(rows[j], x_all[j], odd_pd)
                else:
                    odds = [px.uniform(seed, a, step_idx, b, px.TREE, i * K + kk)[0] for kk in range(K)]
                    groups[i] = tree_group(rows[j], odds)
            new_tree.append(groups)
            parents = [i * K + kk for i in parents for kk in range(len(groups[i]))]
        new_cands, new_q = [], []
        for rr in range(W - n_commit):
            j = rr + n_commit
            new_cands.append(list(new_tree[j - first - 1][0]) if first >= 0 and j - first - 1 < depth else [x_all[j]])
            new_q.append(rows[j])
        new_pos = st.abs_pos + n_commit
        for rr in range(W - n_commit, W):
            new_cands.append([fresh_draft(params, b, new_pos + rr, step_idx)])
            new_q.append(UniformQ(params.lo, params.hi))
        results.append(BatchResult(x=x_all, dev=[x_all[j] != st.cands[j][0] for j in range(W)], first_dev=first,
                                   n_commit=n_commit, committed=committed, rows=rows, accepted_k=k_all))
        st.abs_pos = new_pos
        st.cands, st.q, st.tree = new_cands, new_q, new_tree
        st.last_token = committed[-1]
    return results


def decode_tree(params, n_tokens, forward, max_steps, start_step=0, states=None):
    """Jacobi decode with the full tree; forward(window [B][W], prev [B],
    abs_pos [B], trees [B]) -> (cond, uncond) [B, W + n_extra, V]."""
    if states is None:
        states = init_state(params, start_step)
    grid = [[-1] * n_tokens for _ in range(params.batch)]
    accept_len = []
    t = start_step
    while any(st.abs_pos < n_tokens for st in states):
        if len(accept_len) >= max_steps:
            raise OracleError("step limit")
        prev = [st.last_token for st in states]
        pos = [st.abs_pos for st in states]
        cond, uncond = forward(window_tokens(states), prev, pos, [st.tree for st in states])
        res = step_tree(params, states, t, cond, uncond)
        lens = []
        for b, r in enumerate(res):
            base = pos[b]
            take = max(0, min(r.n_commit, n_tokens - base))
            for i in range(take):
                grid[b][base + i] = r.committed[i]
            lens.append(take)
        accept_len.append(lens)
        t += 1
    return grid, accept_len, len(accept_len)
