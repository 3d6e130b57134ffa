"""Exact-rational enumeration of SJD-PAC on tiny problems (Python fractions).

Independent of oracle/ (no shared code): it restates the paper's rules with
exact probabilities instead of random draws, so that the theorems and the
readings of under-specified points can be checked as exact equalities.

  rs_output      sequential verification of fixed candidates c_1..c_g
                 (Sec. 3.2 / Alg. 1 for g = 1; Thm. 2 for g > 1): exact
                 output distribution.
  wor_tuples     ordered candidate tuples drawn without replacement from a
                 distribution, with their probabilities (Thm. 2 setting).
  decode_dist    whole Jacobi decode on a first-order Markov model: exact
                 joint distribution of (generated grid, per-step commit
                 counts) under the step rules (AC, PD groups on the first D
                 rows after a rejection, window refill with uniform drafts).
"""

from fractions import Fraction as Fr
from functools import lru_cache


def _norm(d):
    s = sum(d.values())
    return {k: v / s for k, v in d.items()}


def rs_output(p, q, cands):
    """Exact distribution of the token chosen by verifying cands in order.

    p, q: dicts token -> Fraction (target, draft). The candidates are assumed
    to have been drawn without replacement from q, so q^(k) is q with
    c_1..c_{k-1} removed and renormalised, and p^(k+1) is the normalised
    positive part of p^(k) - q^(k) (Thm. 2 definitions).
    """
    toks = sorted(set(p) | set(q))
    out = {v: Fr(0) for v in toks}
    reach = Fr(1)
    pk = {v: p.get(v, Fr(0)) for v in toks}
    removed = set()
    qrem = Fr(0)
    for c in cands:
        qk = {v: (Fr(0) if v in removed else q.get(v, Fr(0)) / (1 - qrem)) for v in toks}
        acc = min(Fr(1), pk[c] / qk[c])
        out[c] += reach * acc
        reach *= (1 - acc)
        if reach == 0:
            return out
        r = {v: max(Fr(0), pk[v] - qk[v]) for v in toks}
        pk = _norm(r)
        removed.add(c)
        qrem += q.get(c, Fr(0))
    for v in toks:
        out[v] += reach * pk[v]
    return out


def wor_tuples(dist, k, exclude=()):
    """All ordered tuples of up to k distinct tokens drawn without
    replacement from dist (tokens in `exclude` removed first), with their
    probabilities. Drawing stops early when no mass is left."""
    base = {v: w for v, w in dist.items() if v not in exclude and w > 0}
    res = {}

    def rec(prefix, prob, avail):
        tot = sum(avail.values())
        if len(prefix) == k or tot == 0:
            res[tuple(prefix)] = res.get(tuple(prefix), Fr(0)) + prob
            return
        for v, w in avail.items():
            nxt = dict(avail)
            del nxt[v]
            rec(prefix + [v], prob * w / tot, nxt)

    rec([], Fr(1), base)
    return res


def ar_joint(T, n_tokens, first_prev=0):
    """Exact autoregressive joint distribution of n_tokens under T[prev]."""
    res = {(): Fr(1)}
    for _ in range(n_tokens):
        nxt = {}
        for seq, pr in res.items():
            prev = seq[-1] if seq else first_prev
            for v, w in T[prev].items():
                if w:
                    nxt[seq + (v,)] = nxt.get(seq + (v,), Fr(0)) + pr * w
        res = nxt
    return res


def decode_dist(T, V, n_tokens, W, K, D, ac=1):
    """Exact joint distribution of (grid, commit counts) of a whole decode.

    T: tuple of dicts, T[prev] = next-token distribution (the model).
    The row at window index j is conditioned on the main-path token at
    j-1 (the last committed token for j = 0); its draft distribution q is
    the target distribution it had one step earlier, or uniform on [0, V)
    for a freshly appended position.
    """
    U = "U"
    Tt = tuple(tuple(sorted(d.items())) for d in T)
    uniform = {v: Fr(1, V) for v in range(V)}

    def dist_of(key):
        return uniform if key == U else dict(key)

    @lru_cache(maxsize=None)
    def run(abs_pos, last, rows):
        if abs_pos >= n_tokens:
            return {((), ()): Fr(1)}
        # per-row outcome distributions: (x, alternates) -> prob
        per_row = []
        fresh_row = []
        ps = []
        for j, (cands, qkey) in enumerate(rows):
            ctx = last if j == 0 else rows[j - 1][0][0]
            p = dict(Tt[ctx])
            ps.append(p)
            outs = {}
            for x, px_ in rs_output(p, dist_of(qkey), list(cands)).items():
                if px_ == 0:
                    continue
                for alts, pa in wor_tuples(p, K - 1, exclude=(x,)).items():
                    outs[(x, alts)] = outs.get((x, alts), Fr(0)) + px_ * pa
            per_row.append(outs)
            if not ac:
                fo = {}
                for x, px_ in p.items():
                    if px_ == 0:
                        continue
                    for alts, pa in wor_tuples(p, K - 1, exclude=(x,)).items():
                        fo[(x, alts)] = fo.get((x, alts), Fr(0)) + px_ * pa
                fresh_row.append(fo)
        res = {}

        def combine(j, chosen, prob):
            if j == len(rows):
                finish(chosen, prob)
                return
            for o, po in per_row[j].items():
                combine(j + 1, chosen + [o], prob * po)

        def finish(chosen, prob):
            devs = [chosen[j][0] != rows[j][0][0] for j in range(W)]
            first = next((j for j in range(W) if devs[j]), -1)
            if not ac and first >= 0:
                # vanilla tail: rows after the first rejection are fresh draws from p_j
                tails = [{(): Fr(1)}]
                for j in range(first + 1, W):
                    nt = {}
                    for pre, pp in tails[-1].items():
                        for o, po in fresh_row[j].items():
                            nt[pre + (o,)] = nt.get(pre + (o,), Fr(0)) + pp * po
                    tails.append(nt)
                for tail, pt in tails[-1].items():
                    finish_one(chosen[:first + 1] + list(tail), first, prob * pt)
            else:
                finish_one(chosen, first, prob)

        def finish_one(chosen, first, prob):
            n_commit = W if first < 0 else first + 1
            committed = tuple(c[0] for c in chosen[:n_commit])
            kept = []
            for r in range(W - n_commit):
                j = r + n_commit
                group = (chosen[j][0],)
                if first >= 0 and j <= first + D:
                    group = group + tuple(chosen[j][1])
                kept.append((group, tuple(sorted(ps[j].items()))))
            n_fresh = n_commit
            # fresh rows: uniform drafts, uniform q

            def fresh(i, acc_rows, pr):
                if i == n_fresh:
                    sub = run(abs_pos + n_commit, committed[-1], tuple(kept + acc_rows))
                    take = max(0, min(n_commit, n_tokens - abs_pos))
                    for (g, cs), ps_ in sub.items():
                        key = (committed[:take] + g, (take,) + cs)
                        res[key] = res.get(key, Fr(0)) + pr * ps_
                    return
                for d in range(V):
                    fresh(i + 1, acc_rows + [((d,), U)], pr / V)

            fresh(0, [], prob)

        combine(0, [], Fr(1))
        return res

    start = {}

    def init(i, rows, pr):
        if i == W:
            for k, v in run(0, 0, tuple(rows)).items():
                start[k] = start.get(k, Fr(0)) + pr * v
            return
        for d in range(V):
            init(i + 1, rows + [((d,), U)], pr / V)

    init(0, [], Fr(1))
    return start


def grid_marginal(dist):
    out = {}
    for (g, _), p in dist.items():
        out[g] = out.get(g, Fr(0)) + p
    return out


def commits_marginal(dist, n_first):
    """Distribution of the first n_first commit counts (padded with 0)."""
    out = {}
    for (_, cs), p in dist.items():
        key = tuple(cs[:n_first]) + (0,) * max(0, n_first - len(cs))
        out[key] = out.get(key, Fr(0)) + p
    return out


def decode_dist_tree(T, V, n_tokens, W, K, D):
    """Exact joint distribution of (grid, commit counts) of a whole decode
    with the full K-ary proactive-drafting tree (Sec. 4.1) and adaptive
    continuation.

    After a first rejection at f, the next D positions carry a tree: node i
    at depth d (window row d-1 of the next step) has the children iK..iK+K-1
    at depth d+1, every group K draws without replacement from that
    position's stale target; group 0 of each depth is the main path's (its
    first token is adaptive continuation's, the rest are drawn excluding it).
    At the next step the traversal starts at the root (the last committed
    token): the current node's children are verified against the target
    conditioned on the node (Thm. 2, drafts drawn from the position's stale
    target); the result moves the traversal to the child with that token.
    The context breaks where no child carries the result, or at the last
    tree row when the path has left the main path (the chain beyond hangs
    off the main path); rows after the break are verified as adaptive
    continuation does, with their main-path target and draft group.
    """
    U = "U"
    Tt = tuple(tuple(sorted(d.items())) for d in T)
    uniform = {v: Fr(1, V) for v in range(V)}

    def dist_of(key):
        return uniform if key == U else dict(key)

    def outcome(p, qkey, group):
        return {x: px_ for x, px_ in rs_output(p, dist_of(qkey), list(group)).items() if px_ != 0}

    @lru_cache(maxsize=None)
    def run(abs_pos, last, rows, tree):
        if abs_pos >= n_tokens:
            return {((), ()): Fr(1)}
        Dt = len(tree)
        res = {}
        main_ctx = [last] + [rows[j][0][0] for j in range(W - 1)]
        ps = [dict(Tt[main_ctx[j]]) for j in range(W)]

        def node_token(r, i):
            # token of node i at depth r (r >= 1)
            return tree[r - 1][i // K][i % K]

        # phase A: the traversal, rows 0.. until the context breaks
        def walk(r, i, on_main, xs, prob):
            if r == W:
                after(W - 1 if False else -1, xs, prob)
                return
            ctx = last if r == 0 else (node_token(r, i) if r <= Dt and r >= 1 and r - 1 < Dt else xs[-1])
            group = tree[r][i] if r < Dt else rows[r][0]
            p = dict(Tt[ctx])
            for x, px_ in outcome(p, rows[r][1], group).items():
                if r < Dt:
                    k = group.index(x) if x in group else -1
                    if r < Dt - 1 or (r == Dt - 1 and Dt == W):
                        if k >= 0 and (r < Dt - 1):
                            walk(r + 1, i * K + k, on_main and k == 0, xs + [x], prob * px_)
                        elif k >= 0 and Dt == W and r == Dt - 1:
                            after(-1, xs + [x], prob * px_)
                        else:
                            after(r, xs + [x], prob * px_)
                    else:  # the last tree row with a chain after it
                        if k == 0 and on_main:
                            walk(r + 1, 0, True, xs + [x], prob * px_)
                        else:
                            after(r, xs + [x], prob * px_)
                else:       # chain row (context exact: the path is the main one)
                    if x == group[0]:
                        walk(r + 1, 0, True, xs + [x], prob * px_)
                    else:
                        after(r, xs + [x], prob * px_)

        # phase B: adaptive continuation after the break, then proactive drafting
        def after(first, xs, prob):
            n_commit = W if first < 0 else first + 1
            committed = tuple(xs[:n_commit])

            def tail(j, xs2, prob2):
                if j == W:
                    draft(first, n_commit, committed, xs2, prob2)
                    return
                for x, px_ in outcome(ps[j], rows[j][1], rows[j][0]).items():
                    tail(j + 1, xs2 + [x], prob2 * px_)

            tail(len(xs), list(xs), prob)

        def draft(first, n_commit, committed, xs, prob):
            # rows first+1 .. first+D of this window become the new tree
            depth = 0 if first < 0 else min(D, W - 1 - first)
            levels = []

            def build(d, groups_acc, prob3):
                if d == depth:
                    finish(first, n_commit, committed, xs, tuple(groups_acc), prob3)
                    return
                j = first + 1 + d
                p = ps[j]
                n_nodes = 1 if d == 0 else sum(len(g) for g in groups_acc[-1])
                # group 0: adaptive continuation's token and K-1 alternates
                opts0 = {(xs[j],) + alts: pa for alts, pa in wor_tuples(p, K - 1, exclude=(xs[j],)).items()}

                def rest(n, acc, pr):
                    if n == n_nodes:
                        build(d + 1, groups_acc + [tuple(acc)], pr)
                        return
                    for g, pg in wor_tuples(p, K).items():
                        rest(n + 1, acc + [g], pr * pg)

                for g0, pg0 in opts0.items():
                    rest(1, [g0], prob3 * pg0)

            build(0, [], prob)

        def finish(first, n_commit, committed, xs, new_tree, prob):
            kept = []
            for r in range(W - n_commit):
                j = r + n_commit
                group = (xs[j],)
                if first >= 0 and j - first - 1 < len(new_tree):
                    group = new_tree[j - first - 1][0]
                kept.append((group, tuple(sorted(ps[j].items()))))

            def fresh(i, acc_rows, pr):
                if i == n_commit:
                    sub = run(abs_pos + n_commit, committed[-1], tuple(kept + acc_rows), new_tree)
                    take = max(0, min(n_commit, n_tokens - abs_pos))
                    for (g, cs), ps_ in sub.items():
                        key = (committed[:take] + g, (take,) + cs)
                        res[key] = res.get(key, Fr(0)) + pr * ps_
                    return
                for d in range(V):
                    fresh(i + 1, acc_rows + [((d,), U)], pr / V)

            fresh(0, [], prob)

        walk(0, 0, True, [], Fr(1))
        return res

    start = {}

    def init(i, rows, pr):
        if i == W:
            for k, v in run(0, 0, tuple(rows), ()).items():
                start[k] = start.get(k, Fr(0)) + pr * v
            return
        for d in range(V):
            init(i + 1, rows + [((d,), U)], pr / V)

    init(0, [], Fr(1))
    return start
