"""Pins of the full K-ary proactive-drafting tree (Sec. 4.1).

- Exact enumeration (tests/exact_enum.py, exact fractions) shows that whole
  decodes with the tree are lossless: the grid is distributed exactly as
  plain autoregressive sampling from the model.
- The fp64 oracle's tree decodes on a tiny Markov model match that exact
  distribution (chi-square over grids and per-step commit counts).
- A planted mistake (verifying off-path nodes against the main path's
  target) is caught.
"""

import math
from fractions import Fraction as Fr

import numpy as np
import pytest
from scipy import stats

import exact_enum as ee
from oracle import sjd_fp64 as f64

T3 = ({0: Fr(1, 2), 1: Fr(1, 3), 2: Fr(1, 6)},
      {0: Fr(1, 5), 1: Fr(3, 5), 2: Fr(1, 5)},
      {0: Fr(1, 4), 1: Fr(1, 4), 2: Fr(1, 2)})
SHARP = ({0: Fr(4, 5), 1: Fr(3, 20), 2: Fr(1, 20)},
         {0: Fr(1, 10), 1: Fr(4, 5), 2: Fr(1, 10)},
         {0: Fr(1, 20), 1: Fr(3, 20), 2: Fr(4, 5)})


@pytest.mark.parametrize("W,K,D", [(2, 2, 1), (3, 2, 2), (3, 3, 2)])
def test_tree_decode_is_exactly_lossless(W, K, D):
    dist = ee.decode_dist_tree(T3, 3, 3, W, K, D)
    assert sum(dist.values()) == 1
    assert ee.grid_marginal(dist) == ee.ar_joint(T3, 3)


def markov_tree_forward(T, K, D, stale_nodes=False):
    L = np.array([[math.log(float(d[v])) for v in range(len(d))] for d in T])

    def fwd(window, prev, pos, tree):
        W = len(window)
        out = np.empty((W + f64.n_extra(K, D), L.shape[1]))
        for j in range(W):
            out[j] = L[prev if j == 0 else window[j - 1]]
        for d in range(1, D):
            for i in range(1, K ** d):
                r = W + f64.extra_row(K, d, i)
                grp = tree[d - 1][i // K] if d - 1 < len(tree) and i // K < len(tree[d - 1]) else []
                tok = grp[i % K] if i % K < len(grp) else 0
                out[r] = out[d] if stale_nodes else L[tok]
        return out, None
    return fwd


def _decodes(T, W, K, D, n, stale_nodes=False):
    fwd = markov_tree_forward(T, K, D, stale_nodes)
    grids, commits = {}, {}
    for s in range(n):
        P = f64.Params(batch=1, window=W, vocab=len(T), cfg_scale=1.0, top_k=0, top_p=1.0, pd_k=K,
                       pd_depth=D, ac=1, seed=s, tree=1)
        g, lens = f64.decode_tree(P, 3, fwd, 10)
        grids[tuple(g)] = grids.get(tuple(g), 0) + 1
        commits[tuple(lens)] = commits.get(tuple(lens), 0) + 1
    return grids, commits


def _pvalue(counts, exact, n):
    keys = sorted(exact)
    assert sum(counts.get(k, 0) for k in keys) == n, "outcome outside the exact support"
    if len(keys) == 1:
        return 1.0
    return stats.chisquare([counts.get(k, 0) for k in keys], [float(exact[k]) * n for k in keys]).pvalue


@pytest.mark.parametrize("W,K,D", [(3, 2, 2), (3, 3, 2)])
def test_oracle_tree_decodes_match_the_exact_distribution(W, K, D):
    n = 3000
    grids, commits = _decodes(T3, W, K, D, n)
    dist = ee.decode_dist_tree(T3, 3, 3, W, K, D)
    assert _pvalue(grids, ee.ar_joint(T3, 3), n) > 1e-4
    exact_c = {}
    for (_, cs), p in dist.items():
        exact_c[cs] = exact_c.get(cs, Fr(0)) + p
    assert _pvalue(commits, exact_c, n) > 1e-4


def test_stale_node_targets_are_caught():
    """Verifying the nodes off the main path against the main path's target
    (as if they had no rows of their own) biases the decode."""
    n = 6000
    grids, _ = _decodes(SHARP, 3, 2, 2, n, stale_nodes=True)
    assert _pvalue(grids, ee.ar_joint(SHARP, 3), n) < 1e-6


def test_specification_tree_decodes_match_the_exact_distribution():
    """The kernel-precision specification's tree decode (the bit-exact
    reference of the kernels) on the same tiny model."""
    from oracle import sjd_oracle as so
    W, K, D, n = 3, 2, 2, 2000
    fwd = markov_tree_forward(T3, K, D)

    def fwd_b(window, prev, pos, trees):
        c, _ = fwd(window[0], prev[0], pos[0], trees[0])
        return c[None].astype(np.float32), None

    grids = {}
    for s in range(n):
        P = so.Params(batch=1, window=W, vocab=3, cfg_scale=1.0, top_k=0, top_p=1.0, pd_k=K, pd_depth=D, ac=1,
                      seed=s, tree=1)
        grid, _, _ = so.decode_tree(P, 3, fwd_b, 10)
        grids[tuple(grid[0])] = grids.get(tuple(grid[0]), 0) + 1
    assert _pvalue(grids, ee.ar_joint(T3, 3), n) > 1e-4
