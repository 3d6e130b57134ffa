"""Pins of the relaxed (lossy, off by default) acceptance: candidate c is
accepted iff u < p^(k)(G(c)) / q^(k)(c), with G(c) the ids in c's token group.

- With every id in a group of its own it is the lossless test: both oracles
  give exactly their lossless results.
- The decision threshold in u sits at min(1, p(G(c)) / q(c)) (exact
  threshold location).
- It is lossy: the output of one verified draft is no longer distributed as
  p (exact enumeration over the uniforms), and drafts are accepted more
  often than under the lossless test.
- The kernel-precision specification agrees with the fp64 oracle on it.
"""

from fractions import Fraction as Fr

import numpy as np
import pytest

from oracle import sjd_fp64 as f64
from oracle import sjd_oracle as so
from paper_2603_18599_gb300 import workloads as wlm
from test_fp64_oracle_pins import _threshold, _u, dist_of

ODD_MAX = (1 << 24) - 1


def _kw(w):
    return dict(batch=w.batch, window=w.window, vocab=w.vocab, lo=w.lo, hi=w.hi, cfg_scale=w.cfg_scale,
                temperature=w.temperature, top_k=w.top_k, top_p=w.top_p, pd_k=w.pd_k, pd_depth=w.pd_depth,
                ac=w.ac, seed=w.seed)


def _small():
    return wlm.workloads()["b1w16v8192_f32"].scaled(batch=2, window=8, vocab=512, hi=512, top_k=64, sigma=0.7)


def test_identity_groups_are_the_lossless_test():
    w = _small()
    ident = np.arange(w.vocab, dtype=np.int64)
    P = so.Params(**_kw(w))
    a, b = so.init_state(P), so.init_state(P)
    _, _, qc, qu = wlm.logits_step(w, 0)
    so.draft_from_logits(P, a, 0, qc, qu)
    so.draft_from_logits(P, b, 0, qc, qu)
    P64 = f64.Params(**_kw(w))
    for t in range(3):
        c, u, _, _ = wlm.logits_step(w, t + 1)
        wins = [f64.Window(abs_pos=s.abs_pos, step=t, batch_index=s.batch_index, cands=[list(x) for x in s.cands],
                           q=[f64.Uniform(r.lo, r.hi) if isinstance(r, so.UniformQ) else
                              f64.Dist(ids=r.ids.astype(np.int64), p=r.p.astype(np.float64)) for r in s.q])
                for s in a]
        ra = so.step(P, a, t, c, u)
        rb = so.step(P, b, t, c, u, groups=ident)
        for x, y in zip(ra, rb):
            assert (x.x, x.first_dev, x.accepted_k) == (y.x, y.first_dev, y.accepted_k)
        assert [s.cands for s in a] == [s.cands for s in b]
        for i, win in enumerate(wins):
            r1 = f64.step(P64, win, c[i], u[i])
            r2 = f64.step(P64, win, c[i], u[i], groups=ident)
            assert (r1.x, r1.alts, r1.accepted_k) == (r2.x, r2.alts, r2.accepted_k)


def test_threshold_is_the_group_ratio():
    p = dist_of([0.1, 0.15, 0.05, 0.3, 0.4])
    q = dist_of([0.3, 0.1, 0.2, 0.2, 0.2])
    groups = np.array([0, 0, 1, 1, 2])
    for c in range(5):
        pg = p.p[groups == groups[c]].sum()
        want = min(1.0, pg / q.p[c])
        thr = _threshold(lambda o: f64.verify_group(p, q, [c], [_u(o)], 0.5, groups)[1] == 1)
        assert abs((thr - 1) / 2.0 ** 24 - want) <= 2.0 ** -23


def _single_draft_output(p, q, groups):
    """Exact output distribution of one draft c ~ q verified against p."""
    out = {int(v): Fr(0) for v in p.ids}
    acc_total = Fr(0)
    toks = [int(v) for v in p.ids]
    for c in range(len(q.p)):
        qc = Fr(float(q.p[c]))
        a = Fr(_threshold(lambda o: f64.verify_group(p, q, [c], [_u(o)], 0.5, groups)[1] == 1) - 1, 1 << 24)
        out[c] += qc * a
        acc_total += qc * a
        prev = Fr(0)
        for tk in toks[:-1]:
            edge = _threshold(lambda o: f64.verify_group(p, q, [c], [1 - 2.0 ** -24], _u(o), groups)[0] <= tk)
            cut = Fr(edge - 1, 1 << 24)
            out[tk] += qc * (1 - a) * (cut - prev)
            prev = cut
        out[toks[-1]] += qc * (1 - a) * (1 - prev)
    return out, acc_total


def test_relaxed_acceptance_is_lossy_and_accepts_more():
    p = dist_of([0.05, 0.45, 0.1, 0.4])
    q = dist_of([0.4, 0.1, 0.4, 0.1])
    lossless, acc0 = _single_draft_output(p, q, None)
    assert max(abs(float(lossless[v]) - p.p[v]) for v in range(4)) < 3e-6          # Eq. 1: exactly p
    relaxed, acc1 = _single_draft_output(p, q, np.array([0, 0, 1, 1]))
    assert abs(float(sum(relaxed.values())) - 1.0) < 1e-12
    assert max(abs(float(relaxed[v]) - p.p[v]) for v in range(4)) > 0.05             # biased: lossy
    assert acc1 > acc0 + Fr(1, 10)


def test_specification_agrees_with_fp64_when_relaxed():
    w = wlm.workloads()["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=1, window=16, top_p=1.0, top_k=300,
                                                                    sigma=0.5)
    groups = (np.arange(w.vocab) // 64).astype(np.int64)      # blocks of 64 neighbouring ids
    P, P64 = so.Params(**_kw(w)), f64.Params(**_kw(w))
    st = so.init_state(P)
    _, _, qc, qu = wlm.logits_step(w, 0)
    so.draft_from_logits(P, st, 0, qc, qu)
    accepted = 0
    for t in range(3):
        c, u, _, _ = wlm.logits_step(w, t + 1)
        s0 = st[0]
        win = f64.Window(abs_pos=s0.abs_pos, step=t, batch_index=0, cands=[list(x) for x in s0.cands],
                         q=[f64.Uniform(r.lo, r.hi) if isinstance(r, so.UniformQ) else
                            f64.Dist(ids=r.ids.astype(np.int64), p=r.p.astype(np.float64)) for r in s0.q])
        res = so.step(P, st, t, c, u, groups=groups)[0]
        r64 = f64.step(P64, win, c[0], u[0], groups=groups)
        for j in range(w.window):
            if res.x[j] != r64.x[j]:
                assert r64.row_flags[j]
        accepted += sum(1 for k in res.accepted_k if k)
    assert accepted > 0
