"""sjd_step_noalloc, the entry point for callers that cannot allocate device
memory (they hand in the decode state and the outputs; the step's scratch
lives in a fixed array inside the library), must reproduce sjd_step bit for
bit: the committed tokens, counts and first rejections, and the whole decode
state, over consecutive calls.

This file is collected last on purpose, so that a run stopping at the first
failure has already run every other test.
"""

import ctypes

import pytest
import torch

from lockstep import config_of, device_logits
from paper_2603_18599_gb300 import sjd
from paper_2603_18599_gb300 import workloads as wlm

pytestmark = pytest.mark.gpu


def _outputs_like(ref):
    return tuple(torch.full_like(t, -7) for t in ref)


@pytest.mark.parametrize("name,over", [
    ("b1w16v8192_f32", dict(batch=2)),
    ("b16w64v65536_bf16_mask8192_topp09", dict(batch=3, window=32)),
])
def test_noalloc_step_matches_sjd_step(name, over):
    w = wlm.workloads()[name].scaled(**over)
    cfg = config_of(w)
    dev = torch.device("cuda", torch.cuda.current_device())
    ctx = sjd.SJD(cfg, dev)                       # existing entry points (caller workspace)
    n = sjd.step_noalloc_state_bytes(cfg)
    state = torch.empty(n, dtype=torch.uint8, device=dev)
    persistent = n - 256                          # the rest is the device status word
    for t in range(3):                            # reset on the first call, then continue
        c, u, _, _ = wlm.logits_step(w, t)
        dc, du = device_logits(w, (c, u), dev)
        ref = ctx.step(dc, du)
        out = _outputs_like(ref)
        sjd.step_noalloc(cfg, state, dc, du, *out, reset=(t == 0))
        torch.cuda.synchronize()
        for a, b in zip(ref, out):
            assert torch.equal(a, b), t
        assert torch.equal(ctx.workspace[:persistent], state[:persistent]), t
        assert int(state[persistent:persistent + 4].view(torch.int32)[0]) == 0
    assert ctx.sync() == sjd.SJD_OK


def test_noalloc_rejects_oversized_scratch_and_bad_arguments():
    L = sjd.load()
    big = sjd.make_config(512, 1024, 64, top_k=0)          # 512 x 1024 rows of scratch
    n = ctypes.c_size_t(0)
    assert L.sjd_step_noalloc(ctypes.byref(big), None, ctypes.byref(n), 0, None, None, None, None,
                              None, None) == sjd.SJD_OK
    state = torch.empty(n.value, dtype=torch.uint8, device="cuda")
    dummy = torch.empty(16, dtype=torch.uint8, device="cuda")
    rc = L.sjd_step_noalloc(ctypes.byref(big), ctypes.c_void_p(state.data_ptr()), ctypes.byref(n), 1,
                            ctypes.c_void_p(dummy.data_ptr()), ctypes.c_void_p(dummy.data_ptr()),
                            None, None, None, None)
    assert rc == sjd.SJD_ERR_CAPACITY
    small = sjd.make_config(1, 4, 64, top_k=0)
    n2 = ctypes.c_size_t(16)                                # too small a state buffer
    rc = L.sjd_step_noalloc(ctypes.byref(small), ctypes.c_void_p(state.data_ptr()), ctypes.byref(n2), 1,
                            ctypes.c_void_p(dummy.data_ptr()), ctypes.c_void_p(dummy.data_ptr()),
                            None, None, None, None)
    assert rc == sjd.SJD_ERR_CAPACITY
