"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test checks an oracle function against something other than itself:
published known-answer vectors (Philox), closed forms (softmax, the inverse
CDF), brute force (top-k ranks), the paper's theorems restated with exact
fractions in tests/exact_enum.py (Thm. 1, Thm. 2, losslessness of the whole
decode), and statistical identities (acceptance rate 1 - d_TV, Sec. 4.2).
"""

import math
import os
from fractions import Fraction as Fr

import numpy as np
import pytest
from scipy import special, stats

import exact_enum as ee
from oracle import philox as px
from oracle import sjd_oracle as so

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
ODD_MAX = (1 << 24) - 1


def fr(x):
    return Fr(float(x))


# --------------------------------------------------------------------------
# Philox-4x32-10 (SC'11 definition) against the published known answers.

def test_philox_known_answers():
    n = 0
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            w = [int(x, 16) for x in line.split()]
            assert px.philox4x32_10(w[0:4], w[4:6]) == tuple(w[6:10])
            n += 1
    assert n == 3


def test_uniform_mapping_is_open_interval_and_exact():
    assert px.uniform_odd24(0) == 1
    assert px.uniform_odd24(0xFFFFFFFF) == ODD_MAX
    # u = odd / 2^24 is exact in fp32
    for r in (0, 1 << 9, 0x12345678, 0xFFFFFFFF):
        o = px.uniform_odd24(r)
        assert float(np.float32(o / 2.0 ** 24)) == o / 2.0 ** 24
    # lanes 0..3 share one block, lane 4 moves to the next counter word
    assert px.counter(1, 2, 3, px.PD, 3) == (1, 2, 3, px.PD)
    assert px.counter(1, 2, 3, px.PD, 4) == (1, 2, 3, px.PD + 8)


# --------------------------------------------------------------------------
# EXP against the fp64 exponential (error bound derived from the rounding of
# a = t*log2e, |t| * 2^-23 relative, plus the polynomial's few ulps).

def test_exp_error_bound_and_special_values():
    t = -np.linspace(0.0, 44.36, 200001).astype(np.float32)
    e = so.exp_neg(t)
    ref = np.exp(t.astype(np.float64))
    rel = np.abs(e.astype(np.float64) - ref) / ref
    bound = 2.0 ** -22 + np.abs(t.astype(np.float64)) * 1.5 * 2.0 ** -23
    assert np.all(rel <= bound)
    assert so.exp_neg(np.float32([0.0]))[0] == np.float32(1.0)
    # below the cut-off (a < -64) the value is 0; it would quantise to 0 anyway
    tiny = so.exp_neg(np.float32([-44.4, -100.0, -np.inf]))
    assert np.all(tiny == 0)
    assert math.exp(-44.36) * 2 ** 47 < 0.5


def _f32_nearest(x):
    """fp32 nearest to an exact rational (half to even), fp32 normal range."""
    if x == 0:
        return 0.0
    sg = -1 if x < 0 else 1
    x = abs(x)
    e = x.numerator.bit_length() - x.denominator.bit_length()
    while Fr(2) ** e > x:
        e -= 1
    while Fr(2) ** (e + 1) <= x:
        e += 1
    unit = Fr(2) ** (max(e, -126) - 23)
    m = x / unit
    q, r = divmod(m.numerator, m.denominator)
    if 2 * r > m.denominator or (2 * r == m.denominator and q % 2 == 1):
        q += 1
    return sg * float(q * unit)


def test_fma32_rounds_once():
    """FMA(a, b, c) equals a*b + c in exact rationals rounded once to fp32,
    on random operands and on sums placed next to an fp32 rounding midpoint,
    where rounding to fp64 first and then to fp32 goes wrong."""
    rng = np.random.default_rng(7)
    n = 3000
    def rnd(k):
        m = rng.integers(1 << 23, 1 << 24, size=k)
        ex = rng.integers(-30, 30, size=k)
        sg = rng.choice([-1.0, 1.0], size=k)
        return np.float32(sg * np.ldexp(m.astype(np.float64), ex - 23))
    a, b = rnd(n), rnd(n)
    c = np.where(rng.random(n) < 0.5, rnd(n), np.float32(-a.astype(np.float64) * b.astype(np.float64) * 0.75))
    c = c.astype(np.float32)
    # a*b exactly on an fp32 rounding midpoint, c a power of two far below
    # it: the exact sum lies a hair above or below the midpoint, which fp64
    # cannot hold (a = 1 + m1 2^-12, b = 1 + m2 2^-12 with m1 m2 odd)
    m1 = 2 * rng.integers(0, 1024, size=n) + 1
    m2 = 2 * rng.integers(0, 1024, size=n) + 1
    sc = rng.integers(-20, 20, size=n)
    a2 = np.float32(np.ldexp(1.0 + m1 * 2.0 ** -12, sc))
    b2 = np.float32(np.ldexp(1.0 + m2 * 2.0 ** -12, -sc))
    c2 = np.float32(rng.choice([-1.0, 1.0], size=n) * np.ldexp(1.0, -rng.integers(54, 80, size=n)))
    A = np.concatenate([a, a2]); B = np.concatenate([b, b2]); C = np.concatenate([c, c2])
    got = so.fma32(A, B, C)
    want = np.float32([_f32_nearest(fr(x) * fr(y) + fr(z)) for x, y, z in zip(A, B, C)])
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
    naive = (A.astype(np.float64) * B.astype(np.float64) + C.astype(np.float64)).astype(np.float32)
    assert np.sum(naive.view(np.uint32) != want.view(np.uint32)) > 0   # the cases do bite
    assert so.fma32(np.float32(3.0), np.float32(-1.0), np.float32(3.0)) == np.float32(0.0)


def test_small_weights_never_decrease_with_t():
    """rint(2^47 EXP(t)) is non-decreasing over every fp32 t in [-34, -25].

    There the weights run from 0 to 1955. Ordering candidates by logit then
    orders their small weights, so a top-k cut whose weight lies below 1024
    follows from per-weight counts alone. Weight 1024 is first reached at
    t = -25.6469 (e^t 2^47 = 1023.5 at t = -25.64697 in exact arithmetic).
    """
    lo = np.array([-34.0], np.float32).view(np.uint32)[0]
    hi = np.array([-25.0], np.float32).view(np.uint32)[0]
    t = np.arange(hi, lo + 1, dtype=np.uint64).astype(np.uint32)[::-1].view(np.float32)
    assert np.all(np.diff(t.astype(np.float64)) > 0)
    E = so.quantize(so.exp_neg(t)).astype(np.int64)
    assert np.all(np.diff(E) >= 0)
    first = t[np.argmax(E >= 1024)]
    assert abs(float(first) - (math.log(1023.5) - 47 * math.log(2))) < 1e-4


# --------------------------------------------------------------------------
# Processed distribution (S1-S4).

def test_cfg_and_temperature_closed_form():
    c = np.float32([1.0, 2.0, -0.5])
    u = np.float32([0.5, 3.0, 0.25])
    l = so.combine_logits(c, u, 3.0, 1.0)
    assert l.tolist() == [2.0, 0.0, -2.0]          # u + 3 (c - u), exact here
    l2 = so.combine_logits(c, u, 3.0, 2.0)
    assert l2.tolist() == [1.0, 0.0, -1.0]
    assert so.combine_logits(c, None, 3.0, 1.0).tolist() == c.tolist()


def test_softmax_matches_library_without_cuts():
    g = np.random.default_rng(5)
    for n, sig in ((7, 1.0), (300, 3.0), (4096, 8.0)):
        l = (g.standard_normal(n) * sig).astype(np.float32)
        row = so.process_row(l, 10, 0, 1.0)
        ref = special.softmax(l.astype(np.float64))
        stored = row.ids - 10
        assert np.all(np.diff(row.ids) > 0)
        assert np.all(np.abs(row.p - ref[stored]) <= 1e-5 * ref[stored] + 4e-15)
        # ids left out carry less than the 2^-47 weight resolution
        missing = np.setdiff1d(np.arange(n), stored)
        assert np.all(ref[missing] < 4e-15)
        assert int(row.E.sum(dtype=np.uint64)) == row.Z


def test_hand_worked_distribution():
    l = np.log(np.float64([1.0, 2.0, 3.0])).astype(np.float32)
    row = so.process_row(l, 0, 0, 1.0)
    assert np.allclose(row.p, [1 / 6, 2 / 6, 3 / 6], rtol=1e-6, atol=0)


def test_topk_membership_by_brute_force_ranks():
    g = np.random.default_rng(11)
    n, k = 257, 60
    # bf16-like values so that exact ties occur
    l = np.round(g.standard_normal(n) * 4, 1).astype(np.float32)
    l[[3, 40, 41, 200]] = l[17]                      # planted ties
    row = so.process_row(l, 1000, k, 1.0)
    ids = np.arange(1000, 1000 + n)
    rank = np.zeros(n, int)
    for v in range(n):
        for w in range(n):
            if l[w] > l[v] or (l[w] == l[v] and w < v):
                rank[v] += 1
    want = sorted(ids[rank < k].tolist())
    assert row.ids.tolist() == want
    assert len(want) == k


def test_topp_cut_worked_example():
    l = np.log(np.float64([5.0, 3.0, 2.0])).astype(np.float32)
    # probabilities 0.5, 0.3, 0.2 in order; cut = shortest prefix with mass >= tau
    assert so.process_row(l, 0, 0, 0.45).ids.tolist() == [0]
    assert so.process_row(l, 0, 0, 0.75).ids.tolist() == [0, 1]
    assert so.process_row(l, 0, 0, 0.85).ids.tolist() == [0, 1, 2]
    r = so.process_row(l, 0, 0, 0.75)
    assert np.allclose(r.p, [5 / 8, 3 / 8], rtol=1e-6)
    # top-k applies before top-p
    assert so.process_row(l, 0, 2, 0.85).ids.tolist() == [0, 1]


def test_masked_and_nonfinite_logits():
    l = np.float32([0.0, -np.inf, 1.0, -np.inf, -50.0])
    row = so.process_row(l, 0, 0, 1.0)
    # ids of zero weight (masked, or below the 2^-47 resolution) are not stored
    assert row.ids.tolist() == [0, 2]
    assert np.allclose(row.p, [1 / (1 + math.e), math.e / (1 + math.e)], rtol=1e-6)
    with pytest.raises(so.NonFiniteLogits):
        so.process_row(np.float32([0.0, np.nan]), 0, 0, 1.0)
    with pytest.raises(so.NonFiniteLogits):
        so.process_row(np.float32([0.0, np.inf]), 0, 0, 1.0)
    with pytest.raises(so.NonFiniteLogits):
        so.process_row(np.float32([-np.inf, -np.inf]), 0, 0, 1.0)


def test_inverse_cdf_closed_form():
    w = np.uint64([1, 2, 3])            # CDF 1/6, 3/6, 6/6
    for odd in range(1, ODD_MAX + 1, 99991):
        u = Fr(odd, 1 << 24)
        want = 0 if u < Fr(1, 6) else (1 if u < Fr(3, 6) else 2)
        assert so.inv_cdf(w, 6, odd) == want
    assert so.inv_cdf(np.uint64([0, 5, 0, 5]), 10, 1) == 1
    assert so.inv_cdf(np.uint64([0, 5, 0, 5]), 10, ODD_MAX) == 3


# --------------------------------------------------------------------------
# Acceptance test and residual (Sec. 3.2, Alg. 1, Thm. 1) and sequential
# verification of without-replacement candidates (Thm. 2).

def _row_from_probs(probs, lo=0):
    l = np.log(np.asarray(probs, np.float64)).astype(np.float32)
    return so.process_row(l, lo, 0, 1.0)


def _dist(row):
    return {int(v): fr(p) for v, p in zip(row.ids, row.p)}


def _accept_threshold(fn):
    """Smallest odd uniform numerator at which fn(odd) is False (fn monotone)."""
    lo, hi = 0, (ODD_MAX + 1) // 2            # m in [0, 2^23]
    if not fn(1):
        return 1
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if fn(2 * mid + 1):
            lo = mid
        else:
            hi = mid
    return 2 * hi + 1


def _residual_breaks(fn, tokens):
    """For a monotone step function odd -> token over ascending tokens, the
    fraction of uniforms mapped to each token."""
    out = {}
    prev = Fr(0)
    for t in tokens[:-1]:
        edge = _accept_threshold(lambda o: fn(o) <= t)
        cut = Fr(edge - 1, 1 << 24)
        out[t] = cut - prev
        prev = cut
    out[tokens[-1]] = 1 - prev
    return out


def _oracle_group_distribution(prow, qrow, cands):
    """Output distribution of oracle.verify_group for fixed candidates,
    measured by locating its decision thresholds in the uniforms."""
    g = len(cands)
    out = {int(v): Fr(0) for v in prow.ids}
    reach = Fr(1)
    for k in range(1, g + 1):
        def acc(o, k=k):
            odd = [ODD_MAX] * (k - 1) + [o] + [ODD_MAX] * (g - k)
            return so.verify_group(prow, qrow, cands, odd, 1)[1] == k
        thr = _accept_threshold(acc)
        a = Fr(thr - 1, 1 << 24)
        out[cands[k - 1]] = out.get(cands[k - 1], Fr(0)) + reach * a
        reach *= 1 - a
    toks = [int(v) for v in prow.ids]
    res = _residual_breaks(lambda o: so.verify_group(prow, qrow, cands, [ODD_MAX] * g, o)[0], toks)
    for t, pr in res.items():
        out[t] = out.get(t, Fr(0)) + reach * pr
    return out


def _close(d1, d2, tol):
    keys = set(d1) | set(d2)
    return max(abs(float(d1.get(k, 0)) - float(d2.get(k, 0))) for k in keys) <= tol


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_single_draft_verification_is_exact(seed):
    g = np.random.default_rng(seed)
    p = g.dirichlet(np.ones(5) * 0.7)
    q = g.dirichlet(np.ones(5) * 0.7)
    prow, qrow = _row_from_probs(p), _row_from_probs(q)
    P, Q = _dist(prow), _dist(qrow)
    mix = {v: Fr(0) for v in P}
    for c in range(5):
        want = min(Fr(1), P[c] / Q[c])
        dist_c = _oracle_group_distribution(prow, qrow, [c])
        exact_c = ee.rs_output(P, Q, [c])
        assert _close(dist_c, exact_c, 2e-6)
        wc = Fr(int(qrow.E[c]), qrow.Z)
        for v in mix:
            mix[v] += wc * dist_c.get(v, 0)
        # the decision threshold in u sits at min(1, p/q) (Alg. 1)
        thr = _accept_threshold(lambda o: so.verify_group(prow, qrow, [c], [o], 1)[1] == 1)
        assert abs(float(Fr(thr - 1, 1 << 24) - want)) <= 2 ** -23
    # Rejection Sampling Lemma / Thm. 1: the output is distributed as p
    assert _close(mix, P, 3e-6)


@pytest.mark.parametrize("K", [2, 3])
def test_without_replacement_group_verification_is_exact(K):
    g = np.random.default_rng(100 + K)
    p = g.dirichlet(np.ones(4))
    q = g.dirichlet(np.ones(4))
    prow, qrow = _row_from_probs(p), _row_from_probs(q)
    P, Q = _dist(prow), _dist(qrow)
    qs = {int(v): Fr(int(e), qrow.Z) for v, e in zip(qrow.ids, qrow.E)}
    mix = {v: Fr(0) for v in P}
    for tup, pt in ee.wor_tuples(qs, K).items():
        dist_t = _oracle_group_distribution(prow, qrow, list(tup))
        assert _close(dist_t, ee.rs_output(P, Q, list(tup)), 5e-6)
        for v in mix:
            mix[v] += pt * dist_t.get(v, 0)
    # Thm. 2: K candidates without replacement + final residual recover p
    assert _close(mix, P, 1e-5)


def test_equal_distributions_always_accept():
    row = _row_from_probs([0.1, 0.2, 0.3, 0.4])
    for c in range(4):
        assert so.verify_group(row, row, [c], [ODD_MAX], 1) == (c, 1)


def test_disjoint_supports_always_reject_to_p():
    prow = so.process_row(np.log(np.float64([0.2, 0.3, 0.5])).astype(np.float32), 0, 0, 1.0)
    qrow = so.process_row(np.float32([0.0, 0.0]), 3, 0, 1.0)
    for c in (3, 4):
        res = _residual_breaks(lambda o: so.verify_group(prow, qrow, [c], [1], o)[0], [0, 1, 2])
        assert so.verify_group(prow, qrow, [c], [1], 1)[1] == 0
        assert _close(res, _dist(prow), 2e-6)


def test_acceptance_rate_is_one_minus_tv():
    """Sec. 4.2: the probability that a draft survives is 1 - d_TV(p, q)."""
    g = np.random.default_rng(7)
    l = (g.standard_normal(50) * 1.5).astype(np.float32)
    prow = so.process_row(l, 0, 0, 1.0)
    qrow = so.process_row((l + g.standard_normal(50).astype(np.float32)).astype(np.float32), 0, 0, 1.0)
    P, Q = prow.p.astype(np.float64), qrow.p.astype(np.float64)
    tv = 0.5 * np.abs(P - Q).sum()
    n, acc = 20000, 0
    for i in range(n):
        x = so.sample_row(qrow, px.uniform(9, i, 0, 0, px.SYNTH, 0)[0])
        odd = px.uniform(9, i, 0, 0, px.ACCEPT, 0)[0]
        acc += so.verify_group(prow, qrow, [x], [odd], 1)[1] == 1
    mu = 1 - tv
    assert abs(acc / n - mu) <= 5 * math.sqrt(mu * (1 - mu) / n)


def test_renyi_bound_of_independent_resampling():
    """Sec. 4.2: sum p q <= exp(-(H2(p) + H2(q)) / 2) (Cauchy-Schwarz)."""
    g = np.random.default_rng(3)
    for _ in range(200):
        p = g.dirichlet(np.ones(30) * 0.3)
        q = g.dirichlet(np.ones(30) * 0.3)
        h2 = lambda d: -math.log((d * d).sum())
        assert (p * q).sum() <= math.exp(-(h2(p) + h2(q)) / 2) * (1 + 1e-12)


def test_alternates_are_without_replacement_draws():
    row = _row_from_probs([0.4, 0.3, 0.2, 0.1])
    dist = {int(v): Fr(int(e), row.Z) for v, e in zip(row.ids, row.E)}
    exact = ee.wor_tuples(dist, 2, exclude=(1,))
    counts = {}
    n = 6000
    for i in range(n):
        odds = [px.uniform(4, i, 0, 0, px.PD, k)[0] for k in (1, 2)]
        t = tuple(so.draw_alternates(row, 1, odds))
        counts[t] = counts.get(t, 0) + 1
    keys = sorted(exact)
    obs = [counts.get(k, 0) for k in keys]
    exp = [float(exact[k]) * n for k in keys]
    assert sum(obs) == n
    assert stats.chisquare(obs, exp).pvalue > 1e-4


# --------------------------------------------------------------------------
# Whole-decode losslessness (Sec. 4.2 "rigorously lossless", Thm. 1-2) and
# the readings of the window refill / PD / draft carry.

T3 = ({0: Fr(1, 2), 1: Fr(1, 3), 2: Fr(1, 6)},
      {0: Fr(1, 5), 1: Fr(3, 5), 2: Fr(1, 5)},
      {0: Fr(1, 4), 1: Fr(1, 4), 2: Fr(1, 2)})


@pytest.mark.parametrize("W,K,D,ac", [(1, 1, 0, 1), (2, 1, 0, 1), (2, 1, 0, 0), (2, 2, 1, 1),
                                      (2, 2, 1, 0), (3, 3, 2, 1)])
def test_readings_are_exactly_lossless(W, K, D, ac):
    dist = ee.decode_dist(T3, 3, 3, W, K, D, ac)
    assert sum(dist.values()) == 1
    assert ee.grid_marginal(dist) == ee.ar_joint(T3, 3)


class MarkovForward:
    """Tiny Markov model as a forward: row j's logits are log T[prev_j]."""

    def __init__(self, T):
        self.L = np.array([[math.log(float(d[v])) for v in range(len(d))] for d in T], np.float64)

    def __call__(self, window, prev, pos):
        B, W = len(window), len(window[0])
        out = np.empty((B, W, self.L.shape[1]), np.float32)
        for b in range(B):
            for j in range(W):
                ctx = prev[b] if j == 0 else window[b][j - 1]
                out[b, j] = self.L[ctx]
        return out, None


def _oracle_decodes(W, K, D, ac, n_tokens, n_seeds, T=T3):
    fwd = MarkovForward(T)
    grids, commits = {}, {}
    for s in range(n_seeds):
        P = so.Params(batch=1, window=W, vocab=len(T), cfg_scale=1.0, top_k=0, top_p=1.0,
                      pd_k=K, pd_depth=D, ac=ac, seed=s)
        grid, acc, steps = so.decode(P, n_tokens, fwd, max_steps=10)
        g = tuple(grid[0])
        c = tuple(a[0] for a in acc)
        grids[g] = grids.get(g, 0) + 1
        commits[c] = commits.get(c, 0) + 1
    return grids, commits


def _chi2_ok(counts, exact, n):
    keys = sorted(exact)
    obs = [counts.get(k, 0) for k in keys]
    assert sum(obs) == n, "outcome outside the exact support"
    if len(keys) == 1:
        return 1.0
    exp = [float(exact[k]) * n for k in keys]
    return stats.chisquare(obs, exp).pvalue


@pytest.mark.parametrize("W,K,D,ac", [(1, 1, 0, 1), (2, 2, 1, 1), (2, 2, 1, 0)])
def test_oracle_decode_matches_exact_distribution(W, K, D, ac):
    n = 4000
    grids, commits = _oracle_decodes(W, K, D, ac, 3, n)
    dist = ee.decode_dist(T3, 3, 3, W, K, D, ac)
    assert _chi2_ok(grids, ee.ar_joint(T3, 3), n) > 1e-4
    exact_c = {}
    for (_, cs), p in dist.items():
        exact_c[cs] = exact_c.get(cs, Fr(0)) + p
    assert _chi2_ok(commits, exact_c, n) > 1e-4
    if W == 1:
        assert set(commits) == {(1, 1, 1)}       # plain AR: one token per step


def test_adaptive_continuation_never_hurts_on_tiny_model():
    with_ac = ee.decode_dist(T3, 3, 4, 3, 1, 0, 1)
    without = ee.decode_dist(T3, 3, 4, 3, 1, 0, 0)
    steps = lambda d: sum(p * len(cs) for (_, cs), p in d.items())
    assert steps(with_ac) <= steps(without)
