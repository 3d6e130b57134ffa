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

Arithmetic. The paper fixes no precision. Every quantity that decides an
integer (top-k membership, the top-p cut, the acceptance test, every
inverse-CDF draw) is taken in the same precision as the GPU kernel: IEEE
fp32 with round-to-nearest-even after every operation, where a fused
multiply-add (FMA: a*b + c rounded once) counts as one operation, and
normalising sums taken exactly as integers. The definition is
written out step by step below; the GPU path implements the same definition
independently. The ideal fp64 softmax over the same kept set is also
returned (`p64`) so that the fp32 probabilities can be checked against it.

  logits   l_v = FMA(s, fl(C_v - U_v), U_v)  (s == 1 or no uncond: l = C),
           then l_v = fl(l_v / T) when T != 1, over the allowed ids [lo, hi).
  order    v before w iff l_v > l_w, or l_v == l_w and v < w.
  top-k    the first min(k, V_eff) ids in that order (k <= 0: all).
  weights  m = largest l; e_v = EXP(fl(l_v - m)) with the EXP below;
           E_v = rint(e_v * 2^47) as an integer; Z = sum E_v (exact).
  top-p    (tau < 1) the shortest prefix, in the order above, whose integer
           weight sum W satisfies W >= tau * Z (tau as its exact fp32 value).
  probs    p_v = fl(fl(E_v * 2^-47) / Wz), Wz = fl32(fl64(Z') * 2^-47); the
           stored row holds the kept ids with E_v > 0 (the others have p = 0).
  accept   candidate c with uniform u = (2m+1)/2^24 is accepted iff
           u * q(c) < p(c), evaluated exactly (the fp64 product of two fp32
           values is exact).
  residual r_v = max(0, fl(p_v - q_v)); R_v = rint(r_v * 2^47); R = sum R_v.
  draw     with integer weights w over ascending ids and u = (2m+1)/2^24:
           the first id whose inclusive prefix sum exceeds floor(u * sum w).

EXP is written from the mathematics (base-2 range reduction after Cody &
Waite, "Software Manual for the Elementary Functions", 1980, with the Taylor
series of 2^f): a = fl(t * log2e), n = rint(a), f = fl(a - n) (exact,
|f| <= 1/2), 2^f by Horner on the Taylor coefficients (ln 2)^k / k!,
k = 1..7, each step FMA(y, f, c); result 2^n * poly (exact scaling).
For a < -64 the result is 0 (it would quantise to E = 0 anyway).
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


def process_row(l, lo, top_k, top_p):
    """Row l (fp32 over ids lo..lo+len-1) -> Row, following the definition."""
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
    e = exp_neg((l[sel] - m).astype(np.float32))
    E = quantize(e)
    Z = int(E.sum(dtype=np.uint64))
    tau = np.float32(top_p)
    if tau < np.float32(1.0):
        target = math.ceil(Fraction(float(tau)) * Z)
        cum = np.cumsum(E, dtype=np.uint64)
        cut = int(np.searchsorted(cum, np.uint64(target), side="left"))
        sel, E = sel[:cut + 1], E[:cut + 1]
        Z = int(cum[cut])
    live = E > 0                    # zero-weight ids have p = 0: not stored
    sel, E = sel[live], E[live]
    Wz = fix_to_f32(Z)
    p = (dequantize(E) / Wz).astype(np.float32)
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


def accept(odd24, q_c, p_c):
    """u < p(c)/q(c) as the exact comparison u * q(c) < p(c) (Alg. 1)."""
    u = int(odd24) / float(1 << 24)
    return u * float(q_c) < float(p_c)


def verify_group(prow, q, cands, odd_acc, odd_res):
    """Verify candidates c_1..c_g of one row against target prow (Thm. 2;
    g = 1 is the single-draft test of Sec. 3.2 / Alg. 1).

    q is the row's stored draft distribution P^{t-1}_j; the candidates were
    drawn from it without replacement. Returns (token, k) with k the 1-based
    index of the accepted candidate, or 0 when the token was drawn from the
    final residual p^(g+1).
    """
    ids, cur = prow.ids, prow.p.copy()          # cur = p^(k), k = 1
    pos = {int(v): i for i, v in enumerate(ids)}
    qP = q_on(q, ids)                           # q over the support of p
    qc = [q_at(q, c) for c in cands]
    removed = np.zeros(ids.shape[0], dtype=bool)
    S = np.float32(0.0)
    d = np.float32(1.0)
    g = len(cands)
    R = None
    Rsum = 0
    for k in range(1, g + 1):
        c = int(cands[k - 1])
        q_c = qc[k - 1] if k == 1 else np.float32(qc[k - 1] / d)
        if q_c == np.float32(0.0):
            raise InvalidDraft("draft token has zero draft probability")
        p_c = cur[pos[c]] if c in pos else np.float32(0.0)
        if accept(odd_acc[k - 1], q_c, p_c):
            return c, k
        # rejected: residual p^(k+1) proportional to max(0, p^(k) - q^(k))
        qk = qP if k == 1 else np.where(removed, np.float32(0.0), qP / d).astype(np.float32)
        r = np.maximum(np.float32(0.0), (cur - qk).astype(np.float32))
        R = quantize(r)
        Rsum = int(R.sum(dtype=np.uint64))
        if Rsum == 0:                  # only reachable through rounding
            R = quantize(cur)
            Rsum = int(R.sum(dtype=np.uint64))
        if k == g:
            break
        # adjusted draft q^(k+1): c_1..c_k removed, renormalised
        S = np.float32(S + qc[k - 1])
        if c in pos:
            removed[pos[c]] = True
        d_next = np.float32(np.float32(1.0) - S)
        if not d_next > np.float32(0.0):
            break                      # no draft mass left for more candidates
        d = d_next
        cur = (dequantize(R) / fix_to_f32(Rsum)).astype(np.float32)
    return int(ids[inv_cdf(R, Rsum, odd_res)]), 0


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
            l = combine_logits(_restrict(qcond[i, j], params),
                               None if quncond is None else _restrict(quncond[i, j], params),
                               params.cfg_scale if quncond is not None else 1.0,
                               params.temperature)
            row = process_row(l, params.lo, params.top_k, params.top_p)
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


def step(params, states, step_idx, cond, uncond):
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
            l = combine_logits(_restrict(cond[i, j], params),
                               None if uncond is None else _restrict(uncond[i, j], params),
                               params.cfg_scale, params.temperature)
            prow = process_row(l, params.lo, params.top_k, params.top_p)
            cands = st.cands[j]
            odd_acc = [px.uniform(seed, a, step_idx, b, px.ACCEPT, k)[0] for k in range(len(cands))]
            odd_res = px.uniform(seed, a, step_idx, b, px.RESIDUAL, 0)[0]
            x, k = verify_group(prow, st.q[j], cands, odd_acc, odd_res)
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
