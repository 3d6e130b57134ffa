"""Parity cases rerun on the bounds-checked build (libsjd_checked.so).

In that build every index a kernel takes from data (kept-row ranks, draw
positions, tree slots, node rows) is tested against its array's length;
one outside latches SJD_ERR_BOUNDS in the status word (the access is
clamped, the kernel never traps), which the parity tests' sjd_sync checks
then turn into a failure. The cases run in a child process, so that the
checked library is the one it loads.
"""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))

CASES = " or ".join([
    "test_b16w64v65536_mask_topp_reduced", "test_pd_group_shapes", "test_exact_ties_resolved_by_id",
    "test_topk_cut_far_above_the_weight_floor", "test_id_ordered_trend_defeats_the_sampled_bound",
    "test_full_tree_lockstep", "test_relaxed_acceptance_with_token_groups", "test_ragged_vocab_scalar_path",
    "test_early_logits_steps_overlap_with_the_same_bits",
])


def test_parity_cases_on_the_bounds_checked_build():
    env = dict(os.environ, SJD_LIBRARY="checked")
    r = subprocess.run([sys.executable, "-m", "pytest", os.path.join(HERE, "test_gpu_parity.py"), "-m", "gpu",
                        "-k", CASES, "-x", "-q", "-p", "no:cacheprovider"],
                       env=env, capture_output=True, text=True, timeout=1800)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-2000:]
    assert " passed" in r.stdout
