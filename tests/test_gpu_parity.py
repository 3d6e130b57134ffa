"""CUDA path vs the CPU oracle, element by element, on seeded inputs.

Tokens, first rejections, committed counts, candidate groups and the
sparse rows (ids and fp32 probabilities) must be bit-identical; the
probabilities must also lie within 1e-5 (relative) of the fp64 softmax over
the same kept set. Sizes span many CTAs, ragged tails, unaligned allowed
ranges, ties, chained steps and both kernel paths (fused step and split
verify + draft).
"""

import numpy as np
import pytest
import torch

from lockstep import Lockstep, config_of, device_logits
from oracle import sjd_oracle as so
from paper_2603_18599_gb300 import sjd
from paper_2603_18599_gb300 import workloads as wlm

pytestmark = pytest.mark.gpu

WL = wlm.workloads()


@pytest.fixture(autouse=True, params=["fast", "general"])
def row_kernel(request, monkeypatch):
    """Every case runs on both row kernels (the fast register-resident one,
    where the configuration allows it, and the general one)."""
    if request.param == "general":
        monkeypatch.setenv("SJD_KERNEL", "general")
    else:
        monkeypatch.delenv("SJD_KERNEL", raising=False)
    return request.param


def test_fast_path_is_taken_where_it_applies(row_kernel):
    for name in ("b1w16v8192_f32", "b16w64v65536_bf16_mask8192_topp09", "b8w32v16384_bf16_sigma1to5",
                 "b4w32v32768_bf16_dominant_chain100"):
        w = WL[name].scaled(batch=1)
        ctx = sjd.SJD(config_of(w), "cuda")
        assert ctx.row_path() == (1 if row_kernel == "fast" else 0), name
    # rows whose byte length is not a multiple of 16 always take the general kernel
    w = WL["b1w16v8192_f32"].scaled(vocab=8191, hi=8191)
    assert sjd.SJD(config_of(w), "cuda").row_path() == 0


def run(w, steps, **kw):
    ls = Lockstep(w, **kw)
    c, u = ls.start_from_logits()
    ls.step(c, u)
    for t in range(1, steps):
        c, u, _, _ = ls.inputs(t)
        ls.step(c, u)
    return ls


def test_b1w16v8192_f32_single_step_and_chain():
    run(WL["b1w16v8192_f32"], 4)


def test_split_verify_then_draft_equals_fused_step():
    w = WL["b1w16v8192_f32"].scaled(batch=2)
    a = run(w, 3, fused=True)
    b = run(w, 3, fused=False)
    assert a.history == b.history


def test_b8w32v16384_entropy_sweep_reduced():
    w = WL["b8w32v16384_bf16_sigma1to5"].scaled(batch=5, sigmas_by_batch=(1, 2, 3, 4, 5))
    run(w, 2)


def test_b4w32v32768_dominant_rows_chain_reduced():
    w = WL["b4w32v32768_bf16_dominant_chain100"].scaled(batch=2, steps=4)
    run(w, 4)


def test_b16w64v65536_mask_topp_reduced():
    w = WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=2)
    run(w, 3)


def test_full_size_b8w32v16384_entropy_sweep_every_batch():
    """Full size, as the bench launches it (256 rows: wide CTAs in two
    waves): every batch element, sigma 1 to 5, checked against the oracle
    over three chained steps."""
    run(WL["b8w32v16384_bf16_sigma1to5"], 3)


def test_full_size_b4w32v32768_dominant_rows_every_batch():
    """Full size, as the bench launches it (128 rows, 10 % of them with one
    dominant logit): every batch element checked against the oracle over 25
    chained steps."""
    run(WL["b4w32v32768_bf16_dominant_chain100"], 25)


@pytest.mark.parametrize("top_k,top_p", [(24, 0.95), (300, 1.0), (3000, 0.9)])
def test_topk_cut_far_above_the_weight_floor(top_k, top_p):
    """Flat rows with thousands of candidates: the top-k cut lies far above
    t = -34 (ranked inside one bin of t), reaches into the ids near the
    maximum (small k), or keeps a long row without top-p; the candidate list
    spills past shared memory."""
    w = WL["b8w32v16384_bf16_sigma1to5"].scaled(batch=3, window=8, sigmas_by_batch=(2, 3, 4), top_k=top_k,
                                                 top_p=top_p)
    run(w, 2)


def test_id_ordered_trend_defeats_the_sampled_bound():
    """Logits that fall with the id: the first ids streamed overestimate the
    row's k-th largest logit, so the fast kernel must notice that its bound
    excluded candidates and stream the row again."""
    w = WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=2, window=8, ramp=20.0)
    run(w, 2)
    w2 = w.scaled(top_p=1.0, ramp=-20.0)
    run(w2, 2)


def test_no_guidance_at_scale_one():
    """CFG scale 1: the unconditional logits are not read (the kernels built
    without guidance); every allowed id is a candidate."""
    run(WL["b1w16v8192_f32"].scaled(batch=2, cfg_scale=1.0), 3)
    run(WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=2, window=8, cfg_scale=1.0), 2)


@pytest.mark.parametrize("name,over,pinned,stages", [
    ("b16w64v65536_bf16_mask8192_topp09", dict(batch=2, window=16), True, 2),
    ("b16w64v65536_bf16_mask8192_topp09", dict(batch=2, window=16), True, 1),
    ("b16w64v65536_bf16_mask8192_topp09", dict(batch=2, window=16), False, 2),
    ("b1w16v8192_f32", dict(batch=2), True, 2),
    ("b1w16v8192_f32", dict(batch=2, window=8, vocab=1003, lo=5, hi=998, top_k=100, dtype="bf16"), True, 2),
])
def test_host_input_step_equals_device_step(name, over, pinned, stages):
    """sjd_step_host gives the bits of sjd_step on the full rows, over
    chained steps: the allowed columns of pinned or pageable host rows
    (row pitches of 16 bytes and of 2006 bytes) copied into compact device
    rows, in two alternating stages on the copy stream or in one stage on
    the context's stream."""
    w = WL[name].scaled(**over)
    cfg = config_of(w)
    dev = torch.device("cuda", torch.cuda.current_device())
    a, b = sjd.SJD(cfg, dev), sjd.SJD(cfg, dev)
    _, _, qc, qu = wlm.logits_step(w, 0)
    dq = device_logits(w, (qc, qu), dev)
    a.draft_from_logits(*dq)
    b.draft_from_logits(*dq)
    stage = b.host_stage()
    if stages == 1:
        stage = stage[: stage.numel() // 2]
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    for t in range(4):
        c, u, _, _ = wlm.logits_step(w, t + 1)
        dc, du = device_logits(w, (c, u), dev)
        hc = torch.from_numpy(c).to(dt)
        hu = torch.from_numpy(u).to(dt)
        if pinned:
            hc, hu = hc.pin_memory(), hu.pin_memory()
        ra = a.step(dc, du)
        rb = b.step_host(hc, hu, stage)
        torch.cuda.synchronize()
        for x, y in zip(ra, rb):
            assert torch.equal(x, y), t
        for x, y in zip(a.get_window(), b.get_window()):
            assert torch.equal(x, y), t
        for x, y in zip(a.get_rows(), b.get_rows()):
            assert torch.equal(x, y), t
    assert a.sync() == sjd.SJD_OK and b.sync() == sjd.SJD_OK


def test_aligned_mask_range_and_vanilla_sjd():
    w = WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=2, window=16, lo=32768, hi=40960, ac=0)
    run(w, 3)


@pytest.mark.parametrize("K,D", [(1, 0), (2, 1), (5, 3), (8, 6)])
def test_pd_group_shapes(K, D):
    w = WL["b1w16v8192_f32"].scaled(batch=2, vocab=1024, hi=1024, top_k=300, pd_k=K, pd_depth=D,
                                    sigma=1.0, seed=K * 10 + D)
    run(w, 4)


def test_window_of_one_is_plain_sampling():
    w = WL["b1w16v8192_f32"].scaled(batch=3, window=1, vocab=512, hi=512, top_k=0)
    ls = run(w, 5)
    assert all(n == [1, 1, 1] for n in ls.history)


def test_ragged_vocab_scalar_path_and_temperature():
    # V not a multiple of 4/8 -> no 128-bit loads; unaligned range; T != 1
    w = WL["b1w16v8192_f32"].scaled(batch=2, window=8, vocab=1003, lo=5, hi=998, top_k=100,
                                    temperature=0.7, top_p=0.8, dtype="bf16")
    run(w, 3)


def test_no_topk_and_topk_at_least_vocab():
    w = WL["b1w16v8192_f32"].scaled(batch=1, window=8, vocab=700, hi=700, top_k=0, sigma=2.0)
    run(w, 2)
    w2 = w.scaled(top_k=5000)
    run(w2, 2)


def test_exact_ties_resolved_by_id():
    """Logits on a coarse grid: thousands of exact ties, including at the
    top-k and top-p boundaries and whole tied rows (> 1024 candidates)."""
    w = WL["b1w16v8192_f32"].scaled(batch=2, window=8, vocab=4096, hi=4096, top_k=1500, top_p=0.97,
                                    dtype="bf16", sigma=1.0)
    ls = Lockstep(w)
    rng = np.random.default_rng(3)
    def coarse(shape):
        return (np.round(rng.standard_normal(shape) * 2) / 2).astype(np.float32)
    B, W, V = w.batch, w.window, w.vocab
    c, u = coarse((B, W, V)), coarse((B, W, V))
    c[0, 2] = 1.0
    u[0, 2] = 1.0            # a fully tied row
    qc, qu = coarse((B, W, V)), coarse((B, W, V))
    ls.start_from_logits((c, u, qc, qu))
    ls.step(c, u)
    c2, u2 = coarse((B, W, V)), coarse((B, W, V))
    ls.step(c2, u2)


def test_neg_inf_logits_are_masked_not_errors():
    w = WL["b1w16v8192_f32"].scaled(batch=1, window=8, vocab=512, hi=512, top_k=0)
    ls = Lockstep(w)
    c, u, qc, qu = ls.inputs(0)
    # -inf in the conditional branch gives l = u + s(-inf - u) = -inf; -inf in
    # both branches would give -inf + inf = NaN under logit-space guidance.
    c[:, :, 100:400] = -np.inf
    qc[:, :, 300:350] = -np.inf
    ls.start_from_logits((c, u, qc, qu))
    ls.step(c, u)


def test_nonfinite_logits_set_the_status_word():
    w = WL["b1w16v8192_f32"].scaled(batch=1, window=4, vocab=256, hi=256, top_k=0)
    ctx = sjd.SJD(config_of(w), "cuda")
    c, u, qc, qu = wlm.logits_step(w, 0)
    c[0, 1, 7] = np.nan
    dc, du = device_logits(w, (c, u), torch.device("cuda"))
    ctx.step(dc, du)
    assert ctx.sync() == sjd.SJD_ERR_NONFINITE
    assert ctx.sync() == sjd.SJD_OK          # cleared by the read


def test_call_order_errors():
    w = WL["b1w16v8192_f32"].scaled(batch=1, window=4, vocab=256, hi=256, top_k=0)
    ctx = sjd.SJD(config_of(w), "cuda")
    c, u, _, _ = wlm.logits_step(w, 0)
    dc, du = device_logits(w, (c, u), torch.device("cuda"))
    with pytest.raises(sjd.SJDError) as e:
        ctx.draft_pd()
    assert e.value.code == sjd.SJD_ERR_STATE
    ctx.verify_step(dc, du)
    with pytest.raises(sjd.SJDError) as e:
        ctx.verify_step(dc, du)
    assert e.value.code == sjd.SJD_ERR_STATE
    with pytest.raises(sjd.SJDError) as e:
        ctx.step(dc, du)
    assert e.value.code == sjd.SJD_ERR_STATE
    ctx.draft_pd()
    ctx.step(dc, du)
    assert ctx.sync() == sjd.SJD_OK


def test_smaller_context_keeps_the_shared_memory_limit():
    """The kernels' dynamic shared-memory limit is a setting of the whole
    process: a context of a smaller configuration created later must not
    lower it below what an existing, larger context launches with."""
    dev = torch.device("cuda")
    big = WL["b4w32v32768_bf16_dominant_chain100"].scaled(batch=1, window=4)
    small = WL["b1w16v8192_f32"].scaled(batch=1, window=4, vocab=256, hi=256, top_k=0)
    a = sjd.SJD(config_of(big), dev)
    sjd.SJD(config_of(small), dev)
    c, u, qc, qu = wlm.logits_step(big, 0)
    a.draft_from_logits(*device_logits(big, (qc, qu), dev))
    a.step(*device_logits(big, (c, u), dev))
    assert a.sync() == sjd.SJD_OK


def test_checkpoint_resume_reproduces_bits():
    w = WL["b4w32v32768_bf16_dominant_chain100"].scaled(batch=2, window=16, vocab=4096, hi=4096)
    ctx = sjd.SJD(config_of(w), "cuda")
    dev = torch.device("cuda")
    c0, u0, qc, qu = wlm.logits_step(w, 0)
    ctx.draft_from_logits(*device_logits(w, (qc, qu), dev))
    ctx.step(*device_logits(w, (c0, u0), dev))
    blob = ctx.get_state()
    outs = []
    for t in (1, 2):
        c, u, _, _ = wlm.logits_step(w, t)
        outs.append([x.cpu() for x in ctx.step(*device_logits(w, (c, u), dev))])
    ctx.set_state(blob)
    for i, t in enumerate((1, 2)):
        c, u, _, _ = wlm.logits_step(w, t)
        again = [x.cpu() for x in ctx.step(*device_logits(w, (c, u), dev))]
        for a, b in zip(outs[i], again):
            assert torch.equal(a, b)
    assert ctx.sync() == sjd.SJD_OK


def test_full_decode_32x32_standin_identical_grid():
    """Full synthetic decode of a 32x32 grid with the stand-in model: the
    generated grid and the per-step acceptance lengths are identical."""
    w = WL["decode32x32_b1w16v8192_bf16"]
    model = wlm.StandInModel()
    memo = {}

    def forward(window, prev, pos):
        key = (tuple(map(tuple, window)), tuple(prev), tuple(pos))
        if key not in memo:
            memo[key] = model.forward(window, prev, pos)
        return memo[key]

    dev = torch.device("cuda")
    n_tokens = 1024
    P = so.Params(batch=1, window=16, vocab=8192, cfg_scale=3.0, top_k=2000, top_p=1.0, pd_k=4,
                  pd_depth=3, ac=1, seed=w.seed)
    grid_o, acc_o, steps_o = so.decode(P, n_tokens, forward, max_steps=2000)
    ctx = sjd.SJD(config_of(w, max_steps=2000), dev)
    cbuf = torch.empty((1, 16, 8192), dtype=torch.bfloat16, device=dev)
    ubuf = torch.empty_like(cbuf)

    def fwd(win, prev, pos, cond_out, uncond_out):
        c, u = forward(win.cpu().tolist(), prev.cpu().tolist(), pos.cpu().tolist())
        cond_out.copy_(torch.from_numpy(c).to(torch.bfloat16))
        uncond_out.copy_(torch.from_numpy(u).to(torch.bfloat16))

    grid, acc, steps = ctx.decode_loop(fwd, n_tokens, cbuf, ubuf)
    assert steps == steps_o
    assert grid.cpu().numpy()[0].tolist() == grid_o[0]
    assert acc.cpu().numpy()[:, 0].tolist() == [a[0] for a in acc_o]
    assert min(grid_o[0]) >= 0


def test_decode_90x90_v32768_standin_first_tokens_identical(row_kernel):
    """The larger full decode (90 x 90 grid, V = 32768, stand-in model): its
    first 2000 tokens (320 on the general kernel) and per-step acceptance
    lengths are identical."""
    w = WL["decode90x90_b1w16v32768_bf16"]
    model = wlm.StandInModel(vocab=w.vocab, n_pos=8192)
    memo = {}

    def forward(window, prev, pos):
        key = (tuple(map(tuple, window)), tuple(prev), tuple(pos))
        if key not in memo:
            memo[key] = model.forward(window, prev, pos)
        return memo[key]

    dev = torch.device("cuda")
    n_tokens = 2000 if row_kernel == "fast" else 320
    P = so.Params(batch=1, window=16, vocab=w.vocab, cfg_scale=3.0, top_k=2000, top_p=1.0, pd_k=4,
                  pd_depth=3, ac=1, seed=w.seed)
    grid_o, acc_o, steps_o = so.decode(P, n_tokens, forward, max_steps=n_tokens)
    ctx = sjd.SJD(config_of(w, max_steps=n_tokens), dev)
    cbuf = torch.empty((1, 16, w.vocab), dtype=torch.bfloat16, device=dev)
    ubuf = torch.empty_like(cbuf)

    def fwd(win, prev, pos, cond_out, uncond_out):
        c, u = forward(win.cpu().tolist(), prev.cpu().tolist(), pos.cpu().tolist())
        cond_out.copy_(torch.from_numpy(c).to(torch.bfloat16))
        uncond_out.copy_(torch.from_numpy(u).to(torch.bfloat16))

    grid, acc, steps = ctx.decode_loop(fwd, n_tokens, cbuf, ubuf)
    assert steps == steps_o
    assert grid.cpu().numpy()[0].tolist() == grid_o[0]
    assert acc.cpu().numpy()[:steps, 0].tolist() == [a[0] for a in acc_o]


@pytest.mark.parametrize("step_cfg,steps", [("fused", 10), ("split", 3)])
def test_full_size_b16w64v65536_every_batch(step_cfg, steps):
    """The bench's launch configuration at full size: all 16 batch elements
    checked in full against the oracle over chained steps (10 fused, 3 with
    the split verify + draft)."""
    w = WL["b16w64v65536_bf16_mask8192_topp09"]
    ls = Lockstep(w, fused=step_cfg == "fused")
    c, u = ls.start_from_logits()
    ls.step(c, u)
    for t in range(1, steps):
        c, u, _, _ = ls.inputs(t)
        ls.step(c, u)


def test_full_size_rows_streamed_twice(row_kernel):
    """At the bench's full size, logits that fall with the id (a trend of
    20 across the allowed range) make the sampled bound of the k-th largest
    logit too high, so the fast kernel must stream rows a second time; its
    counter shows it did, and every batch element matches the oracle."""
    w = WL["b16w64v65536_bf16_mask8192_topp09"].scaled(ramp=20.0)
    ls = run(w, 2)
    if row_kernel == "fast":
        assert ls.ctx.stats()[4] > 0


@pytest.mark.parametrize("gs", [1, 64])
def test_relaxed_acceptance_with_token_groups(gs):
    """The relaxed (lossy) acceptance with token groups of gs neighbouring
    ids, bit for bit against the specification over chained steps (gs = 1
    puts every id in a group of its own: the lossless test); a flat row mix
    so that groups matter, short and long kept rows, PD groups."""
    w = WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=2, window=16, top_p=1.0, top_k=300, sigma=0.5)
    groups = (np.arange(w.vocab) // gs).astype(np.int32)
    ls = Lockstep(w, groups=groups)
    c, u = ls.start_from_logits()
    ls.step(c, u)
    for t in (1, 2, 3):
        c, u, _, _ = ls.inputs(t)
        ls.step(c, u)
    w2 = WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=2, window=16, sigma=0.5)
    ls2 = Lockstep(w2, groups=groups)
    c, u = ls2.start_from_logits()
    ls2.step(c, u)
    c, u, _, _ = ls2.inputs(1)
    ls2.step(c, u)


@pytest.mark.parametrize("K,D,W", [(4, 3, 16), (2, 2, 8), (3, 2, 5)])
def test_full_tree_lockstep(K, D, W):
    """The full K-ary proactive-drafting tree (general kernel), bit for bit
    against the specification over chained steps: tokens, commit counts,
    windows, stored rows and the tree itself; node rows carry their own
    seeded logits. Flat rows (sigma 0.4) so that alternates are accepted and
    the walk leaves the main path."""
    w = WL["b1w16v8192_f32"].scaled(batch=3, window=W, vocab=1024, hi=1024, top_k=200, pd_k=K, pd_depth=D,
                                    sigma=0.4, dtype="bf16", seed=K * 100 + D)
    from lockstep import TreeLockstep, tree_inputs
    ls = TreeLockstep(w)
    ls.start_from_logits()
    for t in range(6):
        c, u = tree_inputs(w, t + 1)
        ls.step(c, u)


def standin_tree_forward(model, K, D):
    """The stand-in model as the forward of the full tree: window rows as in
    the plain decode; the row of node i at depth d is the target after that
    node's token at the node's children's position."""
    from oracle import sjd_oracle as so2
    X = so2.n_extra(K, D)

    def fwd(window, prev, pos, trees):
        cond, uncond = model.forward(window, prev, pos)
        B, W, V = cond.shape
        cx = np.empty((B, W + X, V), np.float32)
        ux = np.empty_like(cx)
        cx[:, :W], ux[:, :W] = cond, uncond
        for b in range(B):
            toks, at, rows = [], [], []
            for d in range(1, D):
                for i in range(1, K ** d):
                    tree = trees[b]
                    grp = tree[d - 1][i // K] if d - 1 < len(tree) and i // K < len(tree[d - 1]) else []
                    toks.append(grp[i % K] if i % K < len(grp) else 0)
                    at.append(pos[b] + d)
                    rows.append(W + so2.extra_row(K, d, i))
            if toks:
                c1, u1 = model.forward([[0]] * len(toks), toks, at)
                cx[b, rows], ux[b, rows] = c1[:, 0], u1[:, 0]
        return cx, ux
    return fwd


def test_full_tree_standin_decode_identical():
    """A decode of 256 tokens with the full tree (K = 4, D = 3, W = 16) on a
    sharper stand-in model (weights N(0, 0.3^2), V = 1024, top-k 200), so
    that the walk leaves the main path: every step bit for bit against the
    specification (tokens, windows, rows, the tree), the forward fed from
    the window and tree."""
    from lockstep import TreeLockstep
    w = WL["decode32x32_b1w16v8192_bf16"].scaled(vocab=1024, hi=1024, top_k=200)
    model = wlm.StandInModel(vocab=1024, std=0.3)
    fwd = standin_tree_forward(model, w.pd_k, w.pd_depth)
    ls = TreeLockstep(w)
    n, steps, deep = 0, 0, 0
    while n < 256:
        st = ls.states[0]
        c, u = fwd([[g[0] for g in st.cands]], [st.last_token], [st.abs_pos], [st.tree])
        res = ls.step(c, u)
        n += res[0].n_commit
        steps += 1
        deep += sum(1 for k in res[0].accepted_k[:res[0].n_commit] if k > 1)
    print("tree decode: %d tokens in %d steps (%.2f per step), %d off-main-path acceptances" % (n, steps, n / steps, deep))
    assert deep > 0


@pytest.mark.parametrize("name", ["b16w64v65536_bf16_mask8192_topp09", "b4w32v32768_bf16_dominant_chain100",
                                  "b1w16v8192_f32"])
def test_early_logits_steps_overlap_with_the_same_bits(name, row_kernel):
    """With the early-logits guarantee (resident inputs), consecutive fused
    steps run back to back, each streaming its logits while the one before
    finishes, and give the bits of steps that wait for each other: outputs,
    window and stored rows after every step, at full size (the 128-thread
    layout with short kept rows; the 512-thread layout with kept rows of
    2000 ids, bf16 and f32)."""
    w = WL[name]
    cfg = config_of(w)
    dev = torch.device("cuda", torch.cuda.current_device())
    steps = 6
    ins = [device_logits(w, wlm.logits_step(w, t + 1)[:2], dev) for t in range(steps)]
    dq = device_logits(w, wlm.logits_step(w, 0)[2:], dev)
    a, b = sjd.SJD(cfg, dev), sjd.SJD(cfg, dev)
    a.draft_from_logits(*dq)
    b.draft_from_logits(*dq)
    b.set_early_logits(True)
    torch.cuda.synchronize()
    ref = []
    for t in range(steps):
        ref.append([x.clone() for x in a.step(*ins[t])])
        torch.cuda.synchronize()
    got = [b.step(*ins[t]) for t in range(steps)]  # no synchronisation between the steps
    torch.cuda.synchronize()
    assert a.sync() == sjd.SJD_OK and b.sync() == sjd.SJD_OK, (a.last_error(), b.last_error())
    for t in range(steps):
        for x, y in zip(ref[t], got[t]):
            assert torch.equal(x, y), t
    for x, y in zip(a.get_window(), b.get_window()):
        assert torch.equal(x, y)
    for x, y in zip(a.get_rows(), b.get_rows()):
        assert torch.equal(x, y)
