"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in the oracle (monkeypatched, on the CPU only)
and checks that the pin meant to guard that part now fails.
"""

from fractions import Fraction as Fr

import numpy as np
import pytest

import exact_enum as ee
import test_oracle_pins as pins
from oracle import sjd_oracle as so


def _lemma_holds():
    g = np.random.default_rng(0)
    p = g.dirichlet(np.ones(5) * 0.7)
    q = g.dirichlet(np.ones(5) * 0.7)
    prow, qrow = pins._row_from_probs(p), pins._row_from_probs(q)
    P = pins._dist(prow)
    mix = {v: Fr(0) for v in P}
    for c in range(5):
        d = pins._oracle_group_distribution(prow, qrow, [c])
        for v in mix:
            mix[v] += Fr(int(qrow.E[c]), qrow.Z) * d.get(v, 0)
    return pins._close(mix, P, 3e-6)


def test_lemma_pin_holds_for_the_oracle():
    assert _lemma_holds()


def test_inverted_ratio_is_caught(monkeypatch):
    # u < q(c) / p(c) instead of u < p(c) / q(c)
    monkeypatch.setattr(so, "accept_exact",
                        lambda odd, q_c, Wsum, Wc, d: (odd / 2.0 ** 24) * float(int(Wc)) < float(q_c) * float(int(Wsum)) * d)
    assert not _lemma_holds()


def test_wrong_residual_sign_is_caught(monkeypatch):
    # max(0, q - p) instead of max(0, p - q)
    def wrong_residual(E, q, Z):
        c = so._ceil_q_times(q, Z)
        return c - int(E) if c > int(E) else 0

    monkeypatch.setattr(so, "residual_first", wrong_residual)
    assert not _lemma_holds()


def test_missing_draft_carry_is_caught(monkeypatch):
    """If the next step's q were left uniform instead of P^t (Alg. 1 returns
    P^t), drafts drawn from p would be tested against the wrong proposal and
    the decode would no longer be lossless."""
    real_step = so.step

    def step_without_carry(params, states, step_idx, cond, uncond):
        res = real_step(params, states, step_idx, cond, uncond)
        for st in states:
            st.q = [so.UniformQ(params.lo, params.hi) for _ in st.q]
        return res

    monkeypatch.setattr(so, "step", step_without_carry)
    sharp = ({0: Fr(4, 5), 1: Fr(3, 20), 2: Fr(1, 20)},
             {0: Fr(1, 10), 1: Fr(4, 5), 2: Fr(1, 10)},
             {0: Fr(1, 20), 1: Fr(3, 20), 2: Fr(4, 5)})
    n = 8000
    grids, _ = pins._oracle_decodes(3, 2, 1, 1, 3, n, T=sharp)
    # the pin accepts p-values above 1e-4
    assert pins._chi2_ok(grids, ee.ar_joint(sharp, 3), n) < 1e-6
