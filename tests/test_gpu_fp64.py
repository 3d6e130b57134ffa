"""The CUDA path against the plain fp64 oracle (oracle/sjd_fp64.py), at the
full sizes of the five workloads and the two full decodes.

Each step is teacher-forced: the fp64 oracle starts from the GPU's pre-step
state and steps on the same logits (tests/fp64_check.py). Every token,
alternate, first rejection, commit count and fresh draft must be identical
except at rows behind which the oracle flagged a near-tie; those are
counted and must stay below 1e-6 of all draws. Stored probabilities must lie
within 1e-5 (relative) of the fp64 softmax.
"""

import pytest

from fp64_check import run_decode, run_workload
from paper_2603_18599_gb300 import workloads as wlm

pytestmark = pytest.mark.gpu

WL = wlm.workloads()


@pytest.fixture(params=["fast", "general"])
def row_kernel(request, monkeypatch):
    if request.param == "general":
        monkeypatch.setenv("SJD_KERNEL", "general")
    else:
        monkeypatch.delenv("SJD_KERNEL", raising=False)
    return request.param


def test_fp64_b1w16v8192_f32_chain(row_kernel):
    fc = run_workload(WL["b1w16v8192_f32"], 12)
    print(fc.tally.summary())


def test_fp64_b8w32v16384_entropy_sweep_every_batch():
    fc = run_workload(WL["b8w32v16384_bf16_sigma1to5"], 3)
    print(fc.tally.summary())


def test_fp64_b4w32v32768_dominant_rows_25_steps():
    fc = run_workload(WL["b4w32v32768_bf16_dominant_chain100"], 25)
    print(fc.tally.summary())


def test_fp64_b16w64v65536_mask_topp_every_batch_10_steps():
    fc = run_workload(WL["b16w64v65536_bf16_mask8192_topp09"], 10)
    print(fc.tally.summary())
    assert fc.tally.draws > 10000


def test_fp64_small_cases(row_kernel):
    """Temperature, an unaligned ragged range, vanilla SJD, wide groups."""
    w = WL["b1w16v8192_f32"]
    run_workload(w.scaled(batch=2, window=8, vocab=1003, lo=5, hi=998, top_k=100, temperature=0.7,
                          top_p=0.8, dtype="bf16"), 4)
    run_workload(WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=2, window=16, lo=32768, hi=40960,
                                                                 ac=0), 3)
    run_workload(w.scaled(batch=2, vocab=1024, hi=1024, top_k=300, pd_k=8, pd_depth=6, sigma=1.0, seed=86), 4)


def test_fp64_decode_32x32_standin_whole_grid():
    w = WL["decode32x32_b1w16v8192_bf16"]
    fc, grid, acc = run_decode(w, wlm.StandInModel(), 1024, 2000)
    print(fc.tally.summary(), "steps", len(acc))
    assert len(grid) == 1024 and min(grid) >= 0


def test_fp64_decode_90x90_v32768_standin_first_2000_tokens():
    w = WL["decode90x90_b1w16v32768_bf16"]
    fc, grid, acc = run_decode(w, wlm.StandInModel(vocab=w.vocab, n_pos=8192), 2000, 2000)
    print(fc.tally.summary(), "steps", len(acc))
    assert len(grid) == 2000


def test_fp64_relaxed_acceptance_with_token_groups(row_kernel):
    """The relaxed (lossy) acceptance against the fp64 oracle's relaxed test."""
    import numpy as np
    w = WL["b16w64v65536_bf16_mask8192_topp09"].scaled(batch=4, window=32, top_p=1.0, top_k=300, sigma=0.5)
    fc = run_workload(w, 4, groups=(np.arange(w.vocab) // 64))
    print(fc.tally.summary())


def test_fp64_full_tree_standin_decode():
    """The full tree (K = 4, D = 3) on the sharper stand-in model against the
    fp64 oracle's tree step, teacher-forced, 256 tokens."""
    import numpy as np
    from fp64_check import run_tree_decode
    from test_gpu_parity import standin_tree_forward
    w = WL["decode32x32_b1w16v8192_bf16"].scaled(vocab=1024, hi=1024, top_k=200)
    fwd = standin_tree_forward(wlm.StandInModel(vocab=1024, std=0.3), w.pd_k, w.pd_depth)
    fc, steps = run_tree_decode(w, fwd, 256)
    print(fc.tally.summary(), "steps", steps)
