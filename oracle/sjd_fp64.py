"""Plain double-precision CPU oracle of one SJD-PAC Jacobi step, with
near-tie flags.

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's
cpu_baseline / reference leg may import, call or run anything in oracle/.
The product (the CUDA library and its Python binding) never does, and
shares no code, header, table or constant generator with this file.

This file is the paper's definition written out in numpy float64 and
nothing else: the guided logits, the softmax (np.exp), the top-k and top-p
cuts, the acceptance ratio p/q, the adjusted distributions of Thm. 2 and
every inverse-CDF draw are float64 operations on the exact input values.
No GPU arithmetic is emulated. Apart from the Philox generator (the
published algorithm, pinned to its known-answer vectors), it shares nothing
with oracle/sjd_oracle.py, the kernel-precision specification.

Paper: Kang et al., "SJD-PAC: Accelerating Speculative Jacobi Decoding via
Proactive Drafting and Adaptive Continuation" (CVPR 2026).
  Sec. 3.2   rejection sampling: accept x ~ q iff u < p(x)/q(x) (Eq. 1),
             else draw from max(p - q, 0) renormalised.
  Sec. 3.3   Jacobi window: one forward gives P^t for every row; the
             committed prefix leaves the window and as many fresh positions
             are appended.
  Sec. 4.1   Proactive Drafting: after the first rejection, K candidates per
             position for the next D positions, drawn without replacement.
  Sec. 4.2   Adaptive Continuation: every later position is still verified
             against its own (p_j, q_j); the first rejection does not stop
             the pass.
  Alg. 1     the whole step; P^t becomes the next step's draft rows q.
  Thm. 2     (Appendix A) sequential verification of K without-replacement
             candidates: q^(k) is q with c_1..c_{k-1} removed and
             renormalised; p^(k+1) is max(0, p^(k) - q^(k)) renormalised.
  Sec. 5.1   sampler settings: CFG weight, temperature, top-k.

Readings where the paper is silent (the same readings the CUDA path takes):
  guidance   l = u + s (c - u) on logits, then l / T;     s, T, tau are the
             fp32 values of the configuration.
  order      ids by l descending, ties by id ascending; top-k keeps the
             first min(k, V_eff); top-p keeps the shortest prefix of that
             order whose probability sum is >= tau, then renormalises.
  draw       inverse CDF in ascending id order: the first id whose
             cumulative weight exceeds u * (total weight).
  uniforms   Philox-4x32-10 keyed by the seed, counter
             (absolute position, step, batch, purpose), u = (2m+1) / 2^24.
  residual   if max(0, p - q) has no mass, the draw falls back to p.
  q mass     if the group's draft mass is used up (1 - sum q(c_i) <= 0),
             the remaining candidates are not tested.
  fresh row  draft lo + floor(r64 * V_eff / 2^64), q uniform (1 / V_eff).
  next q     every carried row's q becomes this step's p for it.

Near-ties. A decision is flagged when rounding alone could send a
real-number sampler, or any other correct implementation, down the other
branch:
  accept   |u - p(c)/q(c)| < 1e-6;
  draw     |C - u Z| < 2e-6 Z for the cumulative sum C on either side of
           the chosen id (Z the total weight of the draw), or a draw over a
           total weight below 1e-12 (rounding alone decides whether there
           is anything left to draw);
  top-k    0 < l_k - l_{k+1} <= 1e-6 max(1, |l_k|) at the cut;
  top-p    the cumulative probability at the cut or just before it lies
           within 1e-6 of tau;
  residual the positive part of p - q sums to less than 1e-12.
Every row result carries the flags of the decisions that produced it.
"""

from dataclasses import dataclass, field

import numpy as np

from . import philox as px

NEAR_ACCEPT = 1e-6
NEAR_CDF = 2e-6
NEAR_TOPK = 1e-6
NEAR_TOPP = 1e-6
NEAR_MASS = 1e-12


class NonFiniteLogits(Exception):
    pass


class InvalidDraft(Exception):
    pass


@dataclass
class Params:
    """Problem statement of one decode (Sec. 3.3, 4, 5.1)."""
    batch: int
    window: int                 # L of the paper
    vocab: int
    lo: int = 0                 # allowed ids [lo, hi)
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
        # the configuration carries these as fp32 values
        self.cfg_scale = float(np.float32(self.cfg_scale))
        self.temperature = float(np.float32(self.temperature))
        self.top_p = float(np.float32(self.top_p))

    @property
    def v_eff(self):
        return self.hi - self.lo


@dataclass
class Dist:
    """A sparse distribution over ascending ids (a row p, or a stored q)."""
    ids: np.ndarray             # int64, ascending
    p: np.ndarray               # float64
    flags: list = field(default_factory=list)


@dataclass
class Uniform:
    """Draft distribution of a freshly appended position: uniform on [lo, hi)."""
    lo: int
    hi: int


# ---------------------------------------------------------------------------
# S1-S4: the processed target distribution of one row.

def guided_logits(cond, uncond, s, T):
    """l = u + s (c - u), then l / T (no uncond, or s == 1: l = c)."""
    c = np.asarray(cond, dtype=np.float64)
    if uncond is None or s == 1.0:
        l = c.copy()
    else:
        u = np.asarray(uncond, dtype=np.float64)
        with np.errstate(invalid="ignore"):
            l = u + s * (c - u)
    if T != 1.0:
        l = l / T
    return l


def process_row(l, lo, top_k, top_p):
    """Guided logits over ids lo.. -> Dist: top-k, softmax, top-p."""
    l = np.asarray(l, dtype=np.float64)
    n = l.shape[0]
    if np.isnan(l).any() or np.isposinf(l).any():
        raise NonFiniteLogits("NaN or +inf logit in the allowed range")
    ids = np.arange(lo, lo + n, dtype=np.int64)
    order = np.lexsort((ids, -l))                   # l descending, id ascending
    k = n if top_k <= 0 else min(int(top_k), n)
    flags = []
    if k < n:
        lk, lnext = l[order[k - 1]], l[order[k]]
        if 0.0 < lk - lnext <= NEAR_TOPK * max(1.0, abs(lk)):
            flags.append("topk")
    kept = order[:k]
    m = l[kept[0]]
    if not np.isfinite(m):
        raise NonFiniteLogits("no finite logit in the allowed range")
    w = np.exp(l[kept] - m)
    p = w / w.sum()
    if top_p < 1.0:
        cum = np.cumsum(p)
        cut = min(int(np.searchsorted(cum, top_p, side="left")), k - 1)
        if abs(cum[cut] - top_p) < NEAR_TOPP or (cut > 0 and abs(cum[cut - 1] - top_p) < NEAR_TOPP):
            flags.append("topp")
        kept, w = kept[:cut + 1], w[:cut + 1]
        p = w / w.sum()
    by_id = np.argsort(ids[kept])
    return Dist(ids=ids[kept][by_id], p=p[by_id], flags=flags)


def value_at(d, v):
    """d(v) for a Dist or a Uniform."""
    if isinstance(d, Uniform):
        return 1.0 / (d.hi - d.lo) if d.lo <= v < d.hi else 0.0
    i = int(np.searchsorted(d.ids, v))
    return float(d.p[i]) if i < d.ids.shape[0] and int(d.ids[i]) == int(v) else 0.0


def values_on(d, ids):
    """d(v) for every v in ids."""
    ids = np.asarray(ids, dtype=np.int64)
    if isinstance(d, Uniform):
        return np.where((ids >= d.lo) & (ids < d.hi), 1.0 / (d.hi - d.lo), 0.0)
    if d.ids.shape[0] == 0:
        return np.zeros(ids.shape[0], dtype=np.float64)
    i = np.minimum(np.searchsorted(d.ids, ids), d.ids.shape[0] - 1)
    return np.where(d.ids[i] == ids, d.p[i], 0.0)


# ---------------------------------------------------------------------------
# Draws and the acceptance test (Sec. 3.2, Alg. 1, Thm. 2).

def inv_cdf(w, u, flags, tag):
    """First index whose cumulative weight exceeds u * sum(w); flags a
    threshold within NEAR_CDF of either cumulative sum around it."""
    w = np.asarray(w, dtype=np.float64)
    Z = w.sum()
    C = np.cumsum(w)
    T = u * Z
    i = min(int(np.searchsorted(C, T, side="right")), w.shape[0] - 1)
    if abs(C[i] - T) < NEAR_CDF * Z or (i > 0 and abs(C[i - 1] - T) < NEAR_CDF * Z):
        flags.append(tag)
    if Z < NEAR_MASS:
        flags.append(tag + "_mass")
    return i


def verify_group(row, q, cands, u_acc, u_res, groups=None):
    """Verify candidates c_1..c_g of one row (Thm. 2; g = 1 is Eq. 1).

    row: target Dist p of the row; q: its draft distribution (Dist or
    Uniform) from which the candidates were drawn without replacement.
    groups (optional, lossy): an int array over the vocabulary; candidate c
    is then accepted iff u < p^(k)(G(c)) / q^(k)(c), G(c) the ids of c's
    group (the relaxed acceptance; with every id in a group of its own it
    is the lossless test).
    Returns (token, k, flags, tests): k is the 1-based index of the
    accepted candidate, 0 when the token is a draw from the final residual;
    tests is the number of acceptance tests made.
    """
    flags = []
    ids = row.ids
    pk = row.p.copy()                       # p^(k) over the row's ids
    q_on_ids = values_on(q, ids)
    removed = np.zeros(ids.shape[0], dtype=bool)
    used = 0.0                              # sum of q(c_i) over rejected candidates
    r = None
    g = len(cands)
    for k in range(1, g + 1):
        c = int(cands[k - 1])
        d = 1.0 - used
        q_c = value_at(q, c) / d            # q^(k)(c_k)
        if q_c == 0.0 and groups is None:
            raise InvalidDraft("draft token with zero draft probability")
        j = int(np.searchsorted(ids, c))
        if groups is None:
            p_c = pk[j] if j < ids.shape[0] and int(ids[j]) == c else 0.0
        else:
            p_c = pk[groups[ids] == groups[c]].sum()
        # (relaxed test only: a token it kept may lie outside its stored
        # draft row; q(c) = 0 then makes the ratio infinite)
        ratio = p_c / q_c if q_c > 0.0 else (np.inf if p_c > 0.0 else 0.0)
        if abs(u_acc[k - 1] - ratio) < NEAR_ACCEPT:
            flags.append("accept%d" % k)
        if u_acc[k - 1] < ratio:
            return c, k, flags, k
        qk = np.where(removed, 0.0, q_on_ids / d)     # q^(k) on the row's ids
        r = np.maximum(0.0, pk - qk)
        if r.sum() < NEAR_MASS:
            flags.append("residual_mass")
        if r.sum() == 0.0:
            r = pk.copy()
        used += value_at(q, c)
        if j < ids.shape[0] and int(ids[j]) == c:
            removed[j] = True
        if k == g or not 1.0 - used > 0.0:
            break
        pk = r / r.sum()                    # p^(k+1)
    i = inv_cdf(r, u_res, flags, "residual")
    return int(ids[i]), 0, flags, k


def sample(row, u, flags):
    """One draw from p itself."""
    return int(row.ids[inv_cdf(row.p, u, flags, "sample")])


def alternates(row, first, us, flags):
    """Proactive drafting (Sec. 4.1): draws without replacement from p with
    c_1 = first excluded; stops when nothing is left."""
    w = row.p.copy()
    j = int(np.searchsorted(row.ids, first))
    if j < w.shape[0] and int(row.ids[j]) == int(first):
        w[j] = 0.0
    out = []
    for u in us:
        if not w.sum() > 0.0:
            break
        i = inv_cdf(w, u, flags, "pd")
        out.append(int(row.ids[i]))
        w[i] = 0.0
    return out


# ---------------------------------------------------------------------------
# The step on one batch element (S1-S9, Alg. 1) and the decode loop.

@dataclass
class Window:
    """Decode state of one batch element before a step."""
    abs_pos: int                # absolute position of window row 0
    step: int                   # Jacobi iteration index t
    batch_index: int            # b of the Philox counters
    cands: list                 # per row: [c_1 (the draft), c_2, ...]
    q: list                     # per row: Dist or Uniform (P^{t-1}_j)
    last_token: int = 0
    tree: list = field(default_factory=list)   # full tree: tree[r][i] = children of node i at depth r


def u_of(params, w, j, purpose, lane):
    return px.uniform(params.seed, w.abs_pos + j, w.step, w.batch_index, purpose, lane)[1]


def fresh_draft(params, b, abs_pos, step):
    r = px.raw64(params.seed, abs_pos, step, b, px.INIT)
    return params.lo + ((r * params.v_eff) >> 64)


def init_window(params, b, step=0):
    cands = [[fresh_draft(params, b, j, step)] for j in range(params.window)]
    return Window(abs_pos=0, step=step, batch_index=b, cands=cands,
                  q=[Uniform(params.lo, params.hi) for _ in range(params.window)])


@dataclass
class StepResult:
    x: list                     # x_j^t of every row
    accepted_k: list            # accepted candidate index, 0 = residual draw
    alts: list                  # proactive-drafting alternates of every row
    first_dev: int              # first row with x_j != c_1(j) (-1: none)
    n_commit: int
    committed: list
    rows: list                  # P^t rows (Dist)
    row_flags: list             # near-tie flags behind x_j and alts_j
    draws: int                  # uniforms consumed by decisions
    next: Window


def step(params, w, cond, uncond, groups=None):
    """One Jacobi iteration of Alg. 1 on one batch element.

    cond / uncond: [W, V] arrays holding the exact input logit values
    (uncond None: no guidance); groups: the relaxed acceptance's token
    groups (None: the lossless test). Returns a StepResult with the next
    window.
    """
    W, K, D, lo, hi = params.window, params.pd_k, params.pd_depth, params.lo, params.hi
    xs, ks, alts, rows, flags = [], [], [], [], []
    xf, altf = [], []
    draws = 0
    for j in range(W):
        l = guided_logits(np.asarray(cond[j])[lo:hi],
                          None if uncond is None else np.asarray(uncond[j])[lo:hi],
                          params.cfg_scale, params.temperature)
        row = process_row(l, lo, params.top_k, params.top_p)
        fl = list(row.flags)
        cands = w.cands[j]
        u_acc = [u_of(params, w, j, px.ACCEPT, k) for k in range(len(cands))]
        u_res = u_of(params, w, j, px.RESIDUAL, 0)
        u_pd = [u_of(params, w, j, px.PD, k) for k in range(1, K)]
        x, k, vf, tests = verify_group(row, w.q[j], cands, u_acc, u_res, groups)
        fl += vf
        draws += tests + (0 if k else 1)
        a = alternates(row, x, u_pd, fl)
        draws += len(a)
        if not params.ac:
            ff = []
            f = sample(row, u_res, ff)
            af = alternates(row, f, u_pd, ff)
            xf.append((f, af, ff))
        xs.append(x)
        ks.append(k)
        alts.append(a)
        rows.append(row)
        flags.append(fl)
    first = next((j for j in range(W) if xs[j] != w.cands[j][0]), -1)
    if not params.ac and first >= 0:
        for j in range(first + 1, W):       # vanilla SJD: the tail is redrawn from p_j
            xs[j], alts[j], ks[j] = xf[j][0], xf[j][1], 0
            flags[j] = list(rows[j].flags) + xf[j][2]
            draws += 1 + len(xf[j][1])
    n_commit = W if first < 0 else first + 1
    committed = xs[:n_commit]
    cands, qs = [], []
    for r in range(W - n_commit):           # carried rows, PD groups on the first D
        j = r + n_commit
        group = [xs[j]]
        if first >= 0 and j <= first + D:
            group += alts[j]
        cands.append(group)
        qs.append(rows[j])
    new_pos = w.abs_pos + n_commit
    for r in range(W - n_commit, W):        # fresh positions
        cands.append([fresh_draft(params, w.batch_index, new_pos + r, w.step)])
        qs.append(Uniform(lo, hi))
    nxt = Window(abs_pos=new_pos, step=w.step + 1, batch_index=w.batch_index, cands=cands, q=qs,
                 last_token=committed[-1])
    return StepResult(x=xs, accepted_k=ks, alts=alts, first_dev=first, n_commit=n_commit,
                      committed=committed, rows=rows, row_flags=flags, draws=draws, next=nxt)


def draft_from_logits(params, w, qcond, quncond=None):
    """Draft rows from draft logits (each row's q, and a draft drawn from it
    with purpose SYNTH); quncond None: no guidance."""
    cands, qs = [], []
    for j in range(params.window):
        l = guided_logits(np.asarray(qcond[j])[params.lo:params.hi],
                          None if quncond is None else np.asarray(quncond[j])[params.lo:params.hi],
                          params.cfg_scale if quncond is not None else 1.0, params.temperature)
        row = process_row(l, params.lo, params.top_k, params.top_p)
        qs.append(row)
        cands.append([sample(row, u_of(params, w, j, px.SYNTH, 0), [])])
    return Window(abs_pos=w.abs_pos, step=w.step, batch_index=w.batch_index, cands=cands, q=qs,
                  last_token=w.last_token)


def decode(params, n_tokens, forward, max_steps, b=0):
    """Jacobi decode of one batch element until n_tokens are committed.

    forward(window [W], prev, abs_pos) -> (cond [W, V], uncond [W, V] or
    None) is the model, supplied by the caller. Returns (grid, accept_len).
    """
    w = init_window(params, b)
    grid, lens = [], []
    while len(grid) < n_tokens:
        if len(lens) >= max_steps:
            raise RuntimeError("step limit")
        cond, uncond = forward([c[0] for c in w.cands], w.last_token, w.abs_pos)
        res = step(params, w, cond, uncond)
        take = min(res.n_commit, n_tokens - len(grid))
        grid += res.committed[:take]
        lens.append(take)
        w = res.next
    return grid, lens


# ---------------------------------------------------------------------------
# The full K-ary proactive-drafting tree (Sec. 4.1; the alternative to the
# main-path groups): after a first rejection at f, the next D positions
# carry a tree. Node i at depth d (window row d - 1 of the next step) has the
# children i K .. i K + K - 1 at depth d + 1, each node's group K draws
# without replacement from that position's target (group 0, the main
# path's, is adaptive continuation's token and its K - 1 alternates). Every
# node off the main path at depths 1..D-1 gets a logit row of its own (the
# target conditioned on its path), after the W window rows.

def n_extra(K, D):
    """Logit rows of the nodes off the main path at depths 1..D-1."""
    return sum(K ** d - 1 for d in range(1, D))


def extra_row(K, d, i):
    """Index, after the W window rows, of node i >= 1 at depth d."""
    return sum(K ** e - 1 for e in range(1, d)) + (i - 1)


def tree_group(row, us, flags):
    """K draws without replacement from p (one tree group)."""
    w = row.p.copy()
    out = []
    for u in us:
        if not w.sum() > 0.0:
            break
        i = inv_cdf(w, u, flags, "tree")
        out.append(int(row.ids[i]))
        w[i] = 0.0
    return out


def step_tree(params, w, cond, uncond):
    """One Jacobi iteration with the full tree (adaptive continuation on).

    cond / uncond: [W + n_extra(K, D), V]: the window rows, then the rows of
    the nodes off the main path. The traversal starts at the root (the last
    committed token); at row r the current node's children are verified
    against the node's own target (Thm. 2, drafts from the row's stale q),
    and the traversal moves to the child whose token is the result. The
    context breaks where no child carries it, or at the last tree row when
    the path has left the main path (the chain hangs off the main path);
    every later row keeps adaptive continuation's result with its main-path
    target and group.
    """
    W, K, D, lo, hi = params.window, params.pd_k, params.pd_depth, params.lo, params.hi

    def prow_of(r):
        l = guided_logits(np.asarray(cond[r])[lo:hi], None if uncond is None else np.asarray(uncond[r])[lo:hi],
                          params.cfg_scale, params.temperature)
        return process_row(l, lo, params.top_k, params.top_p)

    rows = [prow_of(j) for j in range(W)]
    draws = 0

    def verify_at(r, prow, group):
        u_acc = [u_of(params, w, r, px.ACCEPT, k) for k in range(len(group))]
        u_res = u_of(params, w, r, px.RESIDUAL, 0)
        x, k, fl, tests = verify_group(prow, w.q[r], group, u_acc, u_res)
        return x, k, list(prow.flags) + fl, tests + (0 if k else 1)

    # adaptive continuation's result of every row (main-path target and group)
    main = []
    for j in range(W):
        x, k, fl, n = verify_at(j, rows[j], w.cands[j])
        main.append((x, k, fl))
        draws += n
    # the traversal
    Dt = len(w.tree)
    xs, flags, ks = [], [], []
    first, node, on_main, r = -1, 0, True, 0
    while r < W:
        if r < Dt and node != 0:
            x, k, fl, n = verify_at(r, prow_of(W + extra_row(K, r, node)), w.tree[r][node])
            draws += n
        else:
            x, k, fl = main[r]
        xs.append(x)
        flags.append(fl)
        ks.append(k)
        if r < Dt:
            group = w.tree[r][node]
            kk = group.index(x) if x in group else -1
            if r < Dt - 1 or Dt == W:
                if kk < 0:
                    first = r
                    break
                node, on_main = node * K + kk, on_main and kk == 0
            elif not (kk == 0 and on_main):
                first = r
                break
        elif x != w.cands[r][0]:
            first = r
            break
        r += 1
    n_commit = W if first < 0 else first + 1
    committed = xs[:n_commit]
    x_all = xs[:n_commit] + [main[j][0] for j in range(n_commit, W)]
    f_all = flags[:n_commit] + [list(main[j][2]) for j in range(n_commit, W)]
    k_all = ks[:n_commit] + [main[j][1] for j in range(n_commit, W)]
    # proactive drafting: the new tree over rows first+1 .. first+depth
    depth = 0 if first < 0 else min(D, W - 1 - first)
    new_tree, alts = [], [[] for _ in range(W)]
    parents = [0]                     # node ids at the depth above
    for dlt in range(1, depth + 1):
        j = first + dlt
        groups = [[] for _ in range(K ** (dlt - 1))]
        a = alternates(rows[j], x_all[j], [u_of(params, w, j, px.PD, k) for k in range(1, K)], f_all[j])
        alts[j] = a
        draws += len(a)
        for i in parents:
            if i == 0:
                groups[0] = [x_all[j]] + a
            else:
                groups[i] = tree_group(rows[j], [u_of(params, w, j, px.TREE, i * K + k) for k in range(K)], f_all[j])
                draws += len(groups[i])
        new_tree.append(groups)
        parents = [i * K + k for i in parents for k in range(len(groups[i]))]
    cands, qs = [], []
    for rr in range(W - n_commit):
        j = rr + n_commit
        cands.append(new_tree[j - first - 1][0] if first >= 0 and j - first - 1 < depth else [x_all[j]])
        qs.append(rows[j])
    new_pos = w.abs_pos + n_commit
    for rr in range(W - n_commit, W):
        cands.append([fresh_draft(params, w.batch_index, new_pos + rr, w.step)])
        qs.append(Uniform(lo, hi))
    nxt = Window(abs_pos=new_pos, step=w.step + 1, batch_index=w.batch_index, cands=cands, q=qs,
                 last_token=committed[-1], tree=new_tree)
    return StepResult(x=x_all, accepted_k=k_all, alts=alts, first_dev=first, n_commit=n_commit,
                      committed=committed, rows=rows, row_flags=f_all, draws=draws, next=nxt)


def decode_tree(params, n_tokens, forward, max_steps, b=0):
    """Jacobi decode with the full tree. forward(window [W], prev, abs_pos,
    tree) -> (cond, uncond) with W + n_extra(K, D) rows: row W + extra_row(K,
    d, i) is the target after node i at depth d (tree[d - 1] holds the
    groups whose children are the depth-d nodes). Returns (grid, accept_len)."""
    w = init_window(params, b)
    grid, lens = [], []
    while len(grid) < n_tokens:
        if len(lens) >= max_steps:
            raise RuntimeError("step limit")
        cond, uncond = forward([c[0] for c in w.cands], w.last_token, w.abs_pos, w.tree)
        res = step_tree(params, w, cond, uncond)
        take = min(res.n_commit, n_tokens - len(grid))
        grid += res.committed[:take]
        lens.append(take)
        w = res.next
    return grid, lens
