"""Pins of the plain fp64 oracle (oracle/sjd_fp64.py) against what the paper
and the mathematics fix, and of the kernel-precision specification
(oracle/sjd_oracle.py) against the fp64 oracle.

The fp64 oracle is checked against closed forms, scipy's softmax, brute-force
ranks, exact-rational enumeration of the rejection-sampling lemma and of
Thm. 2 (tests/exact_enum.py), losslessness of whole decodes, and hand-made
near-ties that must raise its flags. Planted mistakes must fail these pins.
"""

import math
import os
import re
from fractions import Fraction as Fr

import numpy as np
import pytest
from scipy import special, stats

import exact_enum as ee
from oracle import philox as px
from oracle import sjd_fp64 as f64
from oracle import sjd_oracle as so
from paper_2603_18599_gb300 import workloads as wlm

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ODD_MAX = (1 << 24) - 1


def dist_of(probs, lo=0):
    return f64.Dist(ids=np.arange(lo, lo + len(probs), dtype=np.int64), p=np.asarray(probs, np.float64))


# --------------------------------------------------------------------------
# S1-S4

def test_guidance_and_temperature_closed_form():
    c = np.float32([1.0, 2.0, -0.5])
    u = np.float32([0.5, 3.0, 0.25])
    assert f64.guided_logits(c, u, 3.0, 1.0).tolist() == [2.0, 0.0, -2.0]
    assert f64.guided_logits(c, u, 3.0, 2.0).tolist() == [1.0, 0.0, -1.0]
    assert f64.guided_logits(c, None, 3.0, 1.0).tolist() == c.tolist()
    assert f64.guided_logits(c, u, 1.0, 1.0).tolist() == c.tolist()


def test_softmax_matches_library_without_cuts():
    g = np.random.default_rng(5)
    for n, sig in ((7, 1.0), (300, 3.0), (4096, 8.0)):
        l = g.standard_normal(n) * sig
        row = f64.process_row(l, 10, 0, 1.0)
        assert row.ids.tolist() == list(range(10, 10 + n))
        assert np.allclose(row.p, special.softmax(l), rtol=1e-13, atol=0)


def test_hand_worked_rows_and_cuts():
    l = np.log([1.0, 2.0, 3.0])
    assert np.allclose(f64.process_row(l, 0, 0, 1.0).p, [1 / 6, 2 / 6, 3 / 6], rtol=1e-15)
    l = np.log([5.0, 3.0, 2.0])
    # cumulative 0.5, 0.8, 1.0 in (p desc) order: shortest prefix with mass >= tau
    assert f64.process_row(l, 0, 0, 0.45).ids.tolist() == [0]
    assert f64.process_row(l, 0, 0, 0.75).ids.tolist() == [0, 1]
    assert f64.process_row(l, 0, 0, 0.85).ids.tolist() == [0, 1, 2]
    assert np.allclose(f64.process_row(l, 0, 0, 0.75).p, [5 / 8, 3 / 8], rtol=1e-15)
    assert f64.process_row(l, 0, 2, 0.85).ids.tolist() == [0, 1]      # top-k before top-p


def test_topk_membership_by_brute_force_ranks():
    g = np.random.default_rng(11)
    n, k = 257, 60
    l = np.round(g.standard_normal(n) * 4, 1)
    l[[3, 40, 41, 200]] = l[17]                    # planted exact ties
    row = f64.process_row(l, 1000, k, 1.0)
    rank = np.array([sum(1 for w in range(n) if l[w] > l[v] or (l[w] == l[v] and w < v)) for v in range(n)])
    assert row.ids.tolist() == sorted((1000 + np.flatnonzero(rank < k)).tolist())


def test_masked_and_nonfinite_logits():
    row = f64.process_row(np.array([0.0, -np.inf, 1.0]), 0, 0, 1.0)
    assert np.allclose(row.p, [1 / (1 + math.e), 0.0, math.e / (1 + math.e)], rtol=1e-15)
    for bad in ([0.0, np.nan], [0.0, np.inf], [-np.inf, -np.inf]):
        with pytest.raises(f64.NonFiniteLogits):
            f64.process_row(np.array(bad), 0, 0, 1.0)


def test_inverse_cdf_closed_form():
    w = np.array([1.0, 2.0, 3.0])
    for m in range(0, 1 << 23, 99991):
        u = (2 * m + 1) / 2.0 ** 24
        want = 0 if u < 1 / 6 else (1 if u < 3 / 6 else 2)
        assert f64.inv_cdf(w, u, [], "x") == want
    assert f64.inv_cdf(np.array([0.0, 5.0, 0.0, 5.0]), 2.0 ** -24, [], "x") == 1
    assert f64.inv_cdf(np.array([0.0, 5.0, 0.0, 5.0]), 1 - 2.0 ** -24, [], "x") == 3


# --------------------------------------------------------------------------
# S5/S7: the lemma and Thm. 2, by locating the decision thresholds in u

def _threshold(fn):
    """Smallest odd numerator at which the monotone predicate fn(odd) fails."""
    lo, hi = 0, (ODD_MAX + 1) // 2
    if not fn(1):
        return 1
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if fn(2 * mid + 1):
            lo = mid
        else:
            hi = mid
    return 2 * hi + 1


def _u(odd):
    return odd / 2.0 ** 24


def _group_distribution(row, q, cands):
    g = len(cands)
    out = {int(v): Fr(0) for v in row.ids}
    reach = Fr(1)
    for k in range(1, g + 1):
        def acc(o, k=k):
            us = [1 - 2.0 ** -24] * (k - 1) + [_u(o)] + [1 - 2.0 ** -24] * (g - k)
            return f64.verify_group(row, q, cands, us, 0.5)[1] == k
        a = Fr(_threshold(acc) - 1, 1 << 24)
        out[cands[k - 1]] = out.get(cands[k - 1], Fr(0)) + reach * a
        reach *= 1 - a
    toks = [int(v) for v in row.ids]
    us_rej = [1 - 2.0 ** -24] * g
    prev = Fr(0)
    for t in toks[:-1]:
        edge = _threshold(lambda o: f64.verify_group(row, q, cands, us_rej, _u(o))[0] <= t)
        cut = Fr(edge - 1, 1 << 24)
        out[t] = out.get(t, Fr(0)) + reach * (cut - prev)
        prev = cut
    out[toks[-1]] = out.get(toks[-1], Fr(0)) + reach * (1 - prev)
    return out


def _close(d1, d2, tol):
    return max(abs(float(d1.get(k, 0)) - float(d2.get(k, 0))) for k in set(d1) | set(d2)) <= tol


def _fr(d):
    return {int(v): Fr(float(p)) for v, p in zip(d.ids, d.p)}


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_single_draft_verification_is_exact(seed):
    g = np.random.default_rng(seed)
    p, q = dist_of(g.dirichlet(np.ones(5) * 0.7)), dist_of(g.dirichlet(np.ones(5) * 0.7))
    P, Q = _fr(p), _fr(q)
    mix = {v: Fr(0) for v in P}
    for c in range(5):
        d = _group_distribution(p, q, [c])
        assert _close(d, ee.rs_output(P, Q, [c]), 2e-6)
        for v in mix:
            mix[v] += Q[c] * d.get(v, 0)
    assert _close(mix, P, 3e-6)          # the rejection-sampling lemma (Eq. 1)


@pytest.mark.parametrize("K", [2, 3])
def test_without_replacement_group_verification_is_exact(K):
    g = np.random.default_rng(100 + K)
    p, q = dist_of(g.dirichlet(np.ones(4))), dist_of(g.dirichlet(np.ones(4)))
    P, Q = _fr(p), _fr(q)
    mix = {v: Fr(0) for v in P}
    for tup, pt in ee.wor_tuples(Q, K).items():
        d = _group_distribution(p, q, list(tup))
        assert _close(d, ee.rs_output(P, Q, list(tup)), 5e-6)
        for v in mix:
            mix[v] += pt * d.get(v, 0)
    assert _close(mix, P, 1e-5)           # Thm. 2


def test_special_cases():
    p = dist_of([0.1, 0.2, 0.3, 0.4])
    for c in range(4):
        assert f64.verify_group(p, p, [c], [1 - 2.0 ** -24], 0.5)[:2] == (c, 1)
    q = dist_of([0.5, 0.5], lo=3)
    p = dist_of([0.2, 0.3, 0.5])
    for c in (3, 4):
        x, k, _, _ = f64.verify_group(p, q, [c], [2.0 ** -24], 0.6)
        assert k == 0 and x == f64.inv_cdf(p.p, 0.6, [], "x")
    with pytest.raises(f64.InvalidDraft):
        f64.verify_group(p, q, [0], [0.5], 0.5)


def test_acceptance_rate_is_one_minus_tv():
    g = np.random.default_rng(7)
    l = g.standard_normal(50) * 1.5
    p = f64.process_row(l, 0, 0, 1.0)
    q = f64.process_row(l + g.standard_normal(50), 0, 0, 1.0)
    tv = 0.5 * np.abs(p.p - q.p).sum()
    n, acc = 20000, 0
    for i in range(n):
        x = f64.sample(q, px.uniform(9, i, 0, 0, px.SYNTH, 0)[1], [])
        acc += f64.verify_group(p, q, [x], [px.uniform(9, i, 0, 0, px.ACCEPT, 0)[1]], 0.5)[1] == 1
    assert abs(acc / n - (1 - tv)) <= 5 * math.sqrt(tv * (1 - tv) / n)


def test_alternates_are_without_replacement_draws():
    row = dist_of([0.4, 0.3, 0.2, 0.1])
    exact = ee.wor_tuples(_fr(row), 2, exclude=(1,))
    counts = {}
    n = 6000
    for i in range(n):
        us = [px.uniform(4, i, 0, 0, px.PD, k)[1] for k in (1, 2)]
        t = tuple(f64.alternates(row, 1, us, []))
        counts[t] = counts.get(t, 0) + 1
    keys = sorted(exact)
    assert sum(counts.get(k, 0) for k in keys) == n
    assert stats.chisquare([counts.get(k, 0) for k in keys], [float(exact[k]) * n for k in keys]).pvalue > 1e-4


# --------------------------------------------------------------------------
# Whole decodes: lossless (the output is plain autoregressive sampling)

T3 = ({0: Fr(1, 2), 1: Fr(1, 3), 2: Fr(1, 6)},
      {0: Fr(1, 5), 1: Fr(3, 5), 2: Fr(1, 5)},
      {0: Fr(1, 4), 1: Fr(1, 4), 2: Fr(1, 2)})


def _forward(T):
    L = np.array([[math.log(float(d[v])) for v in range(len(d))] for d in T])

    def fwd(window, prev, pos):
        out = np.empty((len(window), L.shape[1]))
        for j in range(len(window)):
            out[j] = L[prev if j == 0 else window[j - 1]]
        return out, None
    return fwd


@pytest.mark.parametrize("W,K,D,ac", [(1, 1, 0, 1), (2, 2, 1, 1), (3, 3, 2, 1), (2, 2, 1, 0)])
def test_decode_matches_exact_distribution(W, K, D, ac):
    n = 3000
    fwd = _forward(T3)
    grids, commits = {}, {}
    for s in range(n):
        P = f64.Params(batch=1, window=W, vocab=3, cfg_scale=1.0, top_k=0, top_p=1.0, pd_k=K,
                       pd_depth=D, ac=ac, seed=s)
        grid, lens = f64.decode(P, 3, fwd, 10)
        grids[tuple(grid)] = grids.get(tuple(grid), 0) + 1
        commits[tuple(lens)] = commits.get(tuple(lens), 0) + 1
    exact = ee.ar_joint(T3, 3)
    keys = sorted(exact)
    assert sum(grids.get(k, 0) for k in keys) == n
    assert stats.chisquare([grids.get(k, 0) for k in keys], [float(exact[k]) * n for k in keys]).pvalue > 1e-4
    dist = ee.decode_dist(T3, 3, 3, W, K, D, ac)
    exact_c = {}
    for (_, cs), p in dist.items():
        exact_c[cs] = exact_c.get(cs, Fr(0)) + p
    ck = sorted(exact_c)
    assert sum(commits.get(k, 0) for k in ck) == n
    if len(ck) > 1:
        assert stats.chisquare([commits.get(k, 0) for k in ck], [float(exact_c[k]) * n for k in ck]).pvalue > 1e-4
    if W == 1:
        assert set(commits) == {(1, 1, 1)}


# --------------------------------------------------------------------------
# Near-tie flags

def test_flags_fire_on_near_ties():
    p, q = dist_of([0.3, 0.7]), dist_of([0.6, 0.4])
    ratio = 0.3 / 0.6
    assert "accept1" in f64.verify_group(p, q, [0], [ratio + 4e-7], 0.5)[2]
    assert "accept1" not in f64.verify_group(p, q, [0], [ratio + 4e-6], 0.5)[2]
    fl = []
    f64.inv_cdf(np.array([1.0, 1.0]), 0.5 + 1e-6, fl, "sample")
    assert fl == ["sample"]
    l = np.array([3.0, 2.0, 2.0 - 1.5e-6, 0.0])
    assert "topk" in f64.process_row(l, 0, 2, 1.0).flags
    assert "topk" not in f64.process_row(l, 0, 3, 1.0).flags
    assert "topk" not in f64.process_row(np.array([3.0, 2.0, 2.0, 0.0]), 0, 2, 1.0).flags   # exact tie
    l = np.log([0.5, 0.3, 0.2])
    assert "topp" in f64.process_row(l, 0, 0, 0.8 + 5e-7).flags
    assert "topp" not in f64.process_row(l, 0, 0, 0.85).flags


# --------------------------------------------------------------------------
# Planted mistakes

def _lemma_holds():
    g = np.random.default_rng(0)
    p, q = dist_of(g.dirichlet(np.ones(5) * 0.7)), dist_of(g.dirichlet(np.ones(5) * 0.7))
    P, Q = _fr(p), _fr(q)
    mix = {v: Fr(0) for v in P}
    for c in range(5):
        d = _group_distribution(p, q, [c])
        for v in mix:
            mix[v] += Q[c] * d.get(v, 0)
    return _close(mix, P, 3e-6)


def test_planted_mistakes_fail_the_lemma(monkeypatch):
    assert _lemma_holds()
    real_max = np.maximum
    with monkeypatch.context() as m:   # residual max(0, q - p)
        m.setattr(f64.np, "maximum", lambda a, b: real_max(a, -b) if np.ndim(b) else real_max(a, b))
        assert not _lemma_holds()
    real_values = f64.values_on
    with monkeypatch.context() as m:   # the ratio taken against the wrong draft row (q shifted by one id)
        m.setattr(f64, "values_on", lambda d, ids: real_values(d, np.asarray(ids) + 1))
        assert not _lemma_holds()


# --------------------------------------------------------------------------
# The kernel-precision specification against the fp64 oracle

def _spec_window(st, t):
    q = [f64.Uniform(r.lo, r.hi) if isinstance(r, so.UniformQ) else
         f64.Dist(ids=r.ids.astype(np.int64), p=r.p.astype(np.float64)) for r in st.q]
    return f64.Window(abs_pos=st.abs_pos, step=t, batch_index=st.batch_index, cands=[list(c) for c in st.cands],
                      q=q, last_token=st.last_token)


@pytest.mark.parametrize("name,over,steps", [
    ("b1w16v8192_f32", dict(), 6),
    ("b8w32v16384_bf16_sigma1to5", dict(batch=2, window=8, sigmas_by_batch=(1, 5)), 3),
    ("b16w64v65536_bf16_mask8192_topp09", dict(batch=1, window=16), 3),
    ("b1w16v8192_f32", dict(batch=2, window=8, vocab=1003, lo=5, hi=998, top_k=100, temperature=0.7,
                            top_p=0.8, dtype="bf16"), 3),
])
def test_specification_agrees_with_fp64(name, over, steps):
    """Teacher-forced from the specification's state, the fp64 oracle gives
    the same tokens except at flagged near-ties, and the specification's
    probabilities lie within 2e-7 (relative) of the fp64 ones, above the
    2^-48 weight resolution."""
    w = wlm.workloads()[name].scaled(**over)
    kw = dict(batch=w.batch, window=w.window, vocab=w.vocab, lo=w.lo, hi=w.hi, cfg_scale=w.cfg_scale,
              temperature=w.temperature, top_k=w.top_k, top_p=w.top_p, pd_k=w.pd_k, pd_depth=w.pd_depth,
              ac=w.ac, seed=w.seed)
    P, P64 = so.Params(**kw), f64.Params(**kw)
    st = so.init_state(P)
    _, _, qc, qu = wlm.logits_step(w, 0)
    so.draft_from_logits(P, st, 0, qc, qu)
    worst = 0.0
    for t in range(steps):
        c, u, _, _ = wlm.logits_step(w, t + 1)
        wins = [_spec_window(s, t) for s in st]
        res = so.step(P, st, t, c, u)
        for i, win in enumerate(wins):
            r64 = f64.step(P64, win, c[i], u[i])
            for j in range(w.window):
                if res[i].x[j] != r64.x[j]:
                    assert r64.row_flags[j], (t, i, j)
                a, b = res[i].rows[j], r64.rows[j]
                common, ia, ib = np.intersect1d(a.ids, b.ids, return_indices=True)
                pa, pb = a.p[ia].astype(np.float64), b.p[ib]
                assert np.all(np.abs(pa - pb) <= 2e-7 * pb + 4e-15), (t, i, j)
                big = pb > 1e-6
                if big.any():
                    worst = max(worst, float(np.max(np.abs(pa[big] - pb[big]) / pb[big])))
    assert worst < 2e-7


def test_kernel_exp2_table_equals_the_mathematics():
    """The CUDA path's double-float constants (written by its own generator)
    equal the specification's, which are computed from series here."""
    txt = open(os.path.join(ROOT, "paper_2603_18599_gb300", "csrc", "sjd_exp2_table.h")).read()
    pairs = re.findall(r"\{(\S+)f, (\S+)f\},\s*// j = (-?\d+)", txt)
    assert len(pairs) == 65
    for hi, lo, j in pairs:
        assert float.fromhex(hi) == float(so._EXP2_HI[int(j) + 32])
        assert float.fromhex(lo) == float(so._EXP2_LO[int(j) + 32])
    consts = dict(re.findall(r"(k\w+) = (\S+)f", txt))
    assert float.fromhex(consts["kLog2eHi"]) == float(so._LOG2E_HI)
    assert float.fromhex(consts["kLog2eLo"]) == float(so._LOG2E_LO)
    assert float.fromhex(consts["kLn2Hi"]) == float(so._LN2_HI)
    assert float.fromhex(consts["kLn2Lo"]) == float(so._LN2_LO)
    for name, d in (("kInv6", 6), ("kInv24", 24), ("kInv120", 120)):
        assert float.fromhex(consts[name]) == float(np.float32(1.0 / d))


def test_precise_weights_within_their_error_bound():
    """round(2^47 exp(t)) of the specification against the fp64 exponential:
    within 1/2 unit plus 4e-12 relative, on guided bf16 and fp32 logits."""
    g = np.random.default_rng(1)
    for s, T, bf in ((3.0, 1.0, True), (3.0, 1.0, False), (7.3, 0.7, False), (1.0, 1.0, False)):
        c = (g.standard_normal(20000) * 3).astype(np.float32)
        u = (g.standard_normal(20000) * 3).astype(np.float32)
        if bf:
            c, u = wlm.bf16_round(c), wlm.bf16_round(u)
        cfg = s != 1.0
        m = so.combine_logits(c, u if cfg else None, s, T).max()
        E = so.precise_weights(c, u, s, T, m, cfg, T != 1.0).astype(np.float64)
        s32, T32 = float(np.float32(s)), float(np.float32(T))
        l = (u.astype(np.float64) + s32 * (c.astype(np.float64) - u)) if cfg else c.astype(np.float64)
        ref = np.exp(l / T32 - float(m)) * 2.0 ** 47
        assert np.all(np.abs(E - ref) <= 0.5 + 1e-4 + 4e-12 * ref)
