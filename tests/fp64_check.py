"""Teacher-forced comparison of the CUDA path with the plain fp64 oracle
(oracle/sjd_fp64.py) under the method's parity rules.

At every step the fp64 oracle starts from the GPU's own pre-step state (the
window, each row's candidate group and stored draft row, the positions),
steps on the same logits, and everything the step produces is compared: the
token of every row, the proactive-drafting alternates, the first rejection,
the commit count, the fresh drafts and the stored probability rows. A row
whose token or alternates differ is allowed only where the fp64 oracle
flagged a near-tie behind it (sjd_fp64's header lists the flags); such rows
are counted, and their number must stay below 1e-6 of all draws.
Probabilities must lie within 1e-5 (relative) of the fp64 values.
"""

from dataclasses import dataclass, field

import numpy as np
import torch

from oracle import sjd_fp64 as f64
from paper_2603_18599_gb300 import sjd
from paper_2603_18599_gb300 import workloads as wlm

P_REL = 1e-5            # stored probabilities vs fp64, relative
P_FLOOR = 4e-15         # ids whose weight rounds to 0 (p < 2^-48) may be left out
MISMATCH_RATE = 1e-6    # flagged mismatches per draw, at most


def params64(w):
    return f64.Params(batch=w.batch, window=w.window, vocab=w.vocab, lo=w.lo, hi=w.hi,
                      cfg_scale=w.cfg_scale, temperature=w.temperature, top_k=w.top_k, top_p=w.top_p,
                      pd_k=w.pd_k, pd_depth=w.pd_depth, ac=w.ac, seed=w.seed)


@dataclass
class Tally:
    draws: int = 0
    rows: int = 0
    flagged_rows: int = 0
    mismatches: list = field(default_factory=list)
    p_checked: int = 0
    p_max_rel: float = 0.0

    def check(self):
        assert len(self.mismatches) <= MISMATCH_RATE * self.draws, (
            "%d flagged mismatches in %d draws: %s" % (len(self.mismatches), self.draws, self.mismatches[:5]))

    def summary(self):
        return ("draws %d, rows %d, rows with a flagged near-tie %d, flagged mismatches %d, "
                "probabilities checked %d, largest relative error %.3g"
                % (self.draws, self.rows, self.flagged_rows, len(self.mismatches), self.p_checked, self.p_max_rel))


def gpu_windows(ctx, params, step, batches):
    """The GPU's pre-step state of each batch element as an fp64-oracle Window."""
    tok, cands, group, pos, prev = [x.cpu().numpy() for x in ctx.get_window()]
    ids, probs, n = [x.cpu().numpy() for x in ctx.get_rows()]
    out = []
    for b in batches:
        cg, qs = [], []
        for r in range(params.window):
            cg.append([int(v) for v in cands[b, r, :int(group[b, r])]])
            k = int(n[b, r])
            if k < 0:
                qs.append(f64.Uniform(params.lo, params.hi))
            else:
                qs.append(f64.Dist(ids=ids[b, r, :k].astype(np.int64), p=probs[b, r, :k].astype(np.float64)))
        out.append(f64.Window(abs_pos=int(pos[b]), step=step, batch_index=b, cands=cg, q=qs,
                              last_token=int(prev[b])))
    return out


def compare_row(ids_g, p_g, row64, flagged, tally, where):
    """A stored GPU row against the fp64 row of the same logits."""
    ids64 = row64.ids
    if not flagged:
        extra = np.setdiff1d(ids_g, ids64)
        assert extra.size == 0, (where, "ids outside the fp64 support", extra[:5])
        missing = np.isin(ids64, ids_g, invert=True)
        assert np.all(row64.p[missing] < P_FLOOR), (where, "ids left out", ids64[missing][:5], row64.p[missing][:5])
    common, ig, i64 = np.intersect1d(ids_g, ids64, return_indices=True)
    pg, pr = p_g[ig].astype(np.float64), row64.p[i64]
    assert np.all(np.abs(pg - pr) <= P_REL * pr + P_FLOOR), (where, "probabilities", np.max(np.abs(pg - pr) / pr))
    big = pr > 1e-6            # above the 2^-47 weight quantisation
    tally.p_checked += int(big.sum())
    if big.any():
        tally.p_max_rel = max(tally.p_max_rel, float(np.max(np.abs(pg[big] - pr[big]) / pr[big])))


def compare_step(params, pre, res, out, post, rows_after, tally, where):
    """One batch element's step: GPU results against the fp64 oracle's."""
    committed, n_commit, first = out
    tok, cands, group = post
    ids, probs, nrow = rows_after
    b = pre.batch_index
    W, D = params.window, params.pd_depth
    nc = int(n_commit[b])
    fr = int(first[b])
    tally.draws += res.draws
    tally.rows += W
    tally.flagged_rows += sum(1 for f in res.row_flags if f)
    # the token of every row: committed rows, then the carried rows' drafts
    x_gpu = [int(v) for v in committed[b, :nc]] + [int(cands[b, r, 0]) for r in range(W - nc)]
    alt_gpu = {}
    for r in range(W - nc):
        j = r + nc
        if fr >= 0 and j <= fr + D:
            alt_gpu[j] = [int(v) for v in cands[b, r, 1:int(group[b, r])]]
    bad = []
    for j in range(W):
        if x_gpu[j] != res.x[j]:
            bad.append(j)
        elif j in alt_gpu and alt_gpu[j] != res.alts[j]:
            bad.append(j)
    for j in bad:
        assert res.row_flags[j], (where, b, j, "unflagged mismatch", x_gpu[j], res.x[j], alt_gpu.get(j),
                                  res.alts[j])
        tally.mismatches.append((where, b, j, tuple(res.row_flags[j])))
    if not bad:
        assert fr == res.first_dev and nc == res.n_commit, (where, b, fr, res.first_dev)
        # the fresh positions' drafts and the carried groups
        assert [[int(v) for v in cands[b, r, :int(group[b, r])]] for r in range(W)] == res.next.cands, (where, b)
    # stored rows: window row r holds P^t of old row r + nc
    for r in range(W - nc):
        k = int(nrow[b, r])
        assert k >= 0, (where, b, r, "carried row without a stored row")
        j = r + nc
        fl = any(f in ("topk", "topp") for f in res.rows[j].flags)
        compare_row(ids[b, r, :k], probs[b, r, :k], res.rows[j], fl, tally, (where, b, j))


class Fp64Check:
    """The CUDA path for every batch element; the fp64 oracle, teacher-forced
    from the GPU's state, for the batch elements in `check`."""

    def __init__(self, w, dev="cuda", check=None, config_over=None, groups=None):
        from lockstep import config_of
        self.w, self.dev = w, torch.device(dev)
        self.P = params64(w)
        self.ctx = sjd.SJD(config_of(w, **(config_over or {})), self.dev)
        self.groups = None if groups is None else np.asarray(groups, np.int64)
        if groups is not None:
            self.ctx.set_relaxed_groups(torch.from_numpy(np.asarray(groups, np.int32)).to(self.dev))
        self.check = list(range(w.batch)) if check is None else list(check)
        self.t = 0
        self.tally = Tally()

    def _dev(self, arrays):
        dt = torch.bfloat16 if self.w.dtype == "bf16" else torch.float32
        return [torch.from_numpy(np.ascontiguousarray(a)).to(self.dev).to(dt) for a in arrays]

    def start_from_logits(self, qc, qu):
        """Drafts from draft logits: the drawn drafts and the rows against fp64."""
        self.ctx.draft_from_logits(*self._dev((qc, qu)))
        assert self.ctx.sync() == sjd.SJD_OK, self.ctx.last_error()
        tok, cands, group, pos, prev = [x.cpu().numpy() for x in self.ctx.get_window()]
        ids, probs, n = [x.cpu().numpy() for x in self.ctx.get_rows()]
        for b in self.check:
            w0 = f64.init_window(self.P, b, self.t)
            d = f64.draft_from_logits(self.P, w0, qc[b], qu[b])
            for r in range(self.P.window):
                fl = []
                f64.sample(d.q[r], f64.u_of(self.P, w0, r, f64.px.SYNTH, 0), fl)
                self.tally.draws += 1
                if int(cands[b, r, 0]) != d.cands[r][0]:
                    assert fl, ("draft", b, r, int(cands[b, r, 0]), d.cands[r][0])
                    self.tally.mismatches.append(("draft", b, r, tuple(fl)))
                k = int(n[b, r])
                compare_row(ids[b, r, :k], probs[b, r, :k], d.q[r], any(f in ("topk", "topp") for f in d.q[r].flags),
                            self.tally, ("draft", b, r))

    def step(self, c, u):
        pre = gpu_windows(self.ctx, self.P, self.t, self.check)
        out = [x.cpu().numpy() for x in self.ctx.step(*self._dev((c, u)))]
        assert self.ctx.sync() == sjd.SJD_OK, self.ctx.last_error()
        tok, cands, group, pos, prev = [x.cpu().numpy() for x in self.ctx.get_window()]
        rows_after = [x.cpu().numpy() for x in self.ctx.get_rows()]
        for i, b in enumerate(self.check):
            res = f64.step(self.P, pre[i], c[b], None if u is None else u[b], self.groups)
            compare_step(self.P, pre[i], res, out, (tok, cands, group), rows_after, self.tally,
                         "step %d" % self.t)
        self.t += 1
        return out


def run_workload(w, steps, check=None, start=0, groups=None):
    """Drafts from the step-0 draft logits, then `steps` chained steps on the
    workload's logits (steps 1..); groups: the relaxed acceptance's token
    groups (None: the lossless test)."""
    fc = Fp64Check(w, check=check, groups=groups)
    _, _, qc, qu = wlm.logits_step(w, 0)
    fc.start_from_logits(qc, qu)
    for t in range(steps):
        c, u, _, _ = wlm.logits_step(w, start + t + 1)
        fc.step(c, u)
    fc.tally.check()
    return fc


def run_decode(w, model, n_tokens, max_steps):
    """A full decode driven step by step on the GPU, with the stand-in model
    as the forward (host side, from the GPU's window), each step checked
    against the fp64 oracle. Returns (checker, grid, accepted per step)."""
    fc = Fp64Check(w, check=[0], config_over=dict(max_steps=max_steps))
    w0 = f64.init_window(fc.P, 0, 0)
    tok = fc.ctx.get_window()[0].cpu().numpy()
    assert tok[0].tolist() == [c[0] for c in w0.cands]      # the initial uniform drafts
    grid, acc = [], []
    while len(grid) < n_tokens:
        assert len(acc) < max_steps
        tok, _, _, pos, prev = [x.cpu().numpy() for x in fc.ctx.get_window()]
        c, u = model.forward(tok.tolist(), prev.tolist(), pos.tolist())
        committed, n_commit, _ = fc.step(c, u)
        take = min(int(n_commit[0]), n_tokens - len(grid))
        grid += [int(v) for v in committed[0, :take]]
        acc.append(take)
    fc.tally.check()
    return fc, grid, acc


def run_tree_decode(w, model_forward, n_tokens):
    """A decode with the full tree, stepped on the GPU with the forward fed
    from the GPU's window and tree, each step checked against the fp64
    oracle's step_tree teacher-forced from the GPU's state."""
    from lockstep import slots_to_tree, tree_to_slots
    fc = Fp64Check(w, check=[0], config_over=dict(pd_tree=1))
    fc.P.tree = 1
    K, D = w.pd_k, w.pd_depth
    n, steps = 0, 0
    while n < n_tokens:
        pre = gpu_windows(fc.ctx, fc.P, fc.t, [0])[0]
        tok, depth = [x.cpu().numpy() for x in fc.ctx.get_tree()]
        pre.tree = slots_to_tree(tok[0], int(depth[0]), K)
        c, u = model_forward([[g[0] for g in pre.cands]], [pre.last_token], [pre.abs_pos], [pre.tree])
        out = [x.cpu().numpy() for x in fc.ctx.step(*fc._dev((c, u)))]
        assert fc.ctx.sync() == sjd.SJD_OK, fc.ctx.last_error()
        res = f64.step_tree(fc.P, pre, c[0], u[0])
        tok2, cands, group, _, _ = [x.cpu().numpy() for x in fc.ctx.get_window()]
        rows_after = [x.cpu().numpy() for x in fc.ctx.get_rows()]
        before = len(fc.tally.mismatches)
        compare_step(fc.P, pre, res, out, (tok2, cands, group), rows_after, fc.tally, "tree step %d" % fc.t)
        if len(fc.tally.mismatches) == before:
            t_after, d_after = [x.cpu().numpy() for x in fc.ctx.get_tree()]
            assert int(d_after[0]) == len(res.next.tree)
            assert t_after[0].tolist() == tree_to_slots(res.next.tree, K, D), ("tree", fc.t)
        fc.t += 1
        n += int(out[1][0])
        steps += 1
    fc.tally.check()
    return fc, steps
