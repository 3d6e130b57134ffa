"""Run the CUDA path and the CPU oracle side by side on the same seeded
inputs and compare everything a step produces."""

import numpy as np
import torch

from oracle import sjd_oracle as so
from paper_2603_18599_gb300 import sjd
from paper_2603_18599_gb300 import workloads as wlm

P_REL = 1e-5          # parity tolerance on probabilities (relative)
P_ABS = 4e-15         # floor: weights are quantised to 2^-47 (< 4e-15 in p)


def params_of(w, batch_ids=None):
    return so.Params(batch=w.batch, window=w.window, vocab=w.vocab, lo=w.lo, hi=w.hi,
                     cfg_scale=w.cfg_scale, temperature=w.temperature, top_k=w.top_k,
                     top_p=w.top_p, pd_k=w.pd_k, pd_depth=w.pd_depth, ac=w.ac, seed=w.seed)


def config_of(w, **over):
    kw = dict(batch=w.batch, window=w.window, vocab=w.vocab, allowed_lo=w.lo, allowed_hi=w.hi,
              cfg_scale=w.cfg_scale, temperature=w.temperature, top_k=w.top_k, top_p=w.top_p,
              pd_k=w.pd_k, pd_depth=w.pd_depth, adaptive_continuation=w.ac, seed=w.seed,
              logit_dtype=sjd.SJD_BF16 if w.dtype == "bf16" else sjd.SJD_F32)
    kw.update(over)
    return sjd.make_config(**kw)


def device_logits(w, arrays, dev):
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    return [torch.from_numpy(np.ascontiguousarray(a)).to(dev).to(dt) for a in arrays]


def compare_window(ctx, states, where=""):
    tok, cands, group, pos, prev = [t.cpu().numpy() for t in ctx.get_window()]
    for i, st in enumerate(states):
        b = st.batch_index
        assert int(pos[b]) == st.abs_pos, (where, b, "abs_pos", int(pos[b]), st.abs_pos)
        assert int(prev[b]) == st.last_token, (where, b, "prev", int(prev[b]), st.last_token)
        for r, g in enumerate(st.cands):
            assert int(group[b, r]) == len(g), (where, b, r, "group", int(group[b, r]), g)
            assert cands[b, r, :len(g)].tolist() == list(g), (where, b, r, cands[b, r].tolist(), g)
            assert int(tok[b, r]) == g[0]


def compare_rows(ctx, states, where="", check_p64=True):
    ids, probs, n = [t.cpu().numpy() for t in ctx.get_rows()]
    for st in states:
        b = st.batch_index
        for r, q in enumerate(st.q):
            k = int(n[b, r])
            if isinstance(q, so.UniformQ):
                assert k == -1, (where, b, r, "expected uniform row", k)
                continue
            assert k == q.ids.shape[0], (where, b, r, "row length", k, q.ids.shape[0])
            assert np.array_equal(ids[b, r, :k], q.ids), (where, b, r, "row ids")
            assert np.array_equal(probs[b, r, :k], q.p), (where, b, r, "row probs (bit-exact)")
            if check_p64:
                p = probs[b, r, :k].astype(np.float64)
                assert np.all(np.abs(p - q.p64) <= P_REL * q.p64 + P_ABS), (where, b, r, "p vs fp64")


def compare_results(committed, n_commit, first, res, states):
    committed, n_commit, first = committed.cpu().numpy(), n_commit.cpu().numpy(), first.cpu().numpy()
    for r, st in zip(res, states):
        b = st.batch_index
        assert int(first[b]) == r.first_dev, (b, "first_rej", int(first[b]), r.first_dev)
        assert int(n_commit[b]) == r.n_commit, (b, "n_commit", int(n_commit[b]), r.n_commit)
        assert committed[b, :r.n_commit].tolist() == r.committed, (b, "committed")
        assert np.all(committed[b, r.n_commit:] == -1)


class Lockstep:
    """The CUDA path for every batch element, the oracle for `check_batches`."""

    def __init__(self, w, dev="cuda", check_batches=None, fused=True, config_over=None, groups=None):
        self.w, self.dev, self.fused = w, torch.device(dev), fused
        self.P = params_of(w)
        self.ctx = sjd.SJD(config_of(w, **(config_over or {})), self.dev)
        self.groups = groups            # relaxed (lossy) acceptance's token groups, or None
        if groups is not None:
            self.ctx.set_relaxed_groups(torch.from_numpy(np.asarray(groups, np.int32)).to(self.dev))
        self.check = list(range(w.batch)) if check_batches is None else list(check_batches)
        self.states = so.init_state(self.P, 0, self.check)
        self.t = 0
        self.history = []

    def inputs(self, step):
        """(cond, uncond, qcond, quncond) for every batch element (fp32 host)."""
        return wlm.logits_step(self.w, step)

    def start_from_logits(self, arrays=None):
        c, u, qc, qu = arrays if arrays is not None else self.inputs(0)
        dq = device_logits(self.w, (qc, qu), self.dev)
        self.ctx.draft_from_logits(*dq)
        so.draft_from_logits(self.P, self.states, self.t, qc[self.check], qu[self.check])
        assert self.ctx.sync() == sjd.SJD_OK, self.ctx.last_error()
        compare_window(self.ctx, self.states, "after draft")
        compare_rows(self.ctx, self.states, "after draft")
        return c, u

    def step(self, c, u, check_rows=True):
        dc, du = device_logits(self.w, (c, u), self.dev)
        if self.fused:
            out = self.ctx.step(dc, du)
        else:
            out = self.ctx.verify_step(dc, du)
            self.ctx.draft_pd()
        res = so.step(self.P, self.states, self.t, c[self.check], u[self.check], self.groups)
        assert self.ctx.sync() == sjd.SJD_OK, self.ctx.last_error()
        compare_results(*out, res, self.states)
        compare_window(self.ctx, self.states, "step %d" % self.t)
        if check_rows:
            compare_rows(self.ctx, self.states, "step %d" % self.t)
        self.history.append([r.n_commit for r in res])
        self.t += 1
        return res


def tree_to_slots(tree, K, D):
    """An oracle tree (tree[r][i] = children of node i at depth r) as the
    library's token slots: depth d from slot sum_{e<d} K^e, node i at +i."""
    out = [-1] * sum(K ** d for d in range(1, D + 1))
    off = 0
    for r, groups in enumerate(tree):
        for i, grp in enumerate(groups):
            for k, v in enumerate(grp):
                out[off + i * K + k] = v
        off += K ** (r + 1)
    return out


def slots_to_tree(tok, depth, K):
    """The library's token slots as an oracle tree of the given depth."""
    tree, off = [], 0
    for r in range(depth):
        groups = []
        for i in range(K ** r):
            g = [int(v) for v in tok[off + i * K: off + i * K + K]]
            groups.append([v for v in g if v >= 0])
        tree.append(groups)
        off += K ** (r + 1)
    return tree


def tree_inputs(w, step):
    """(cond, uncond) [B, W + X, V] for the full tree: the window rows and the
    node rows, every row its own seeded draw."""
    X = so.n_extra(w.pd_k, w.pd_depth)
    rows = w.window + X
    c = np.empty((w.batch, rows, w.vocab), np.float32)
    u = np.empty_like(c)
    for b in range(w.batch):
        for j in range(rows):
            c[b, j], u[b, j], _, _ = wlm.logits_row(w, step, b, j)
    return c, u


class TreeLockstep(Lockstep):
    """Lockstep with the full proactive-drafting tree (general kernel)."""

    def __init__(self, w, dev="cuda"):
        super().__init__(w, dev, config_over=dict(pd_tree=1))
        self.P.tree = 1

    def step(self, c, u, check_rows=True):
        dc, du = device_logits(self.w, (c, u), self.dev)
        out = self.ctx.step(dc, du)
        res = so.step_tree(self.P, self.states, self.t, c[self.check], u[self.check])
        assert self.ctx.sync() == sjd.SJD_OK, self.ctx.last_error()
        compare_results(*out, res, self.states)
        compare_window(self.ctx, self.states, "step %d" % self.t)
        if check_rows:
            compare_rows(self.ctx, self.states, "step %d" % self.t)
        tok, depth = [x.cpu().numpy() for x in self.ctx.get_tree()]
        for st in self.states:
            b = st.batch_index
            assert int(depth[b]) == len(st.tree), ("tree depth", b, int(depth[b]), len(st.tree))
            assert tok[b].tolist() == tree_to_slots(st.tree, self.w.pd_k, self.w.pd_depth), ("tree", b)
        self.history.append([r.n_commit for r in res])
        self.t += 1
        return res
