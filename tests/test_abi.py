"""The C-ABI library builds, loads and exports every entry point that
include/sjd.h declares; host-side argument checks (no GPU compute)."""

import ctypes
import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sjd.h")


@pytest.fixture(scope="session")
def libsjd():
    from paper_2603_18599_gb300 import _build, sjd
    if not os.path.exists(sjd.lib_path()):
        if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
            pytest.skip("nvcc not available to build libsjd.so")
        _build.build()
    return sjd.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = set(re.findall(r"\b(sjd_[a-z_]+)\s*\(", text))
    return sorted(n for n in names if n != "sjd_forward_fn")


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("sjd_init", "sjd_verify_step", "sjd_draft", "sjd_decode_loop", "sjd_step",
                     "sjd_workspace_size", "sjd_sync", "sjd_destroy"):
        assert required in names


def test_library_exports_every_declared_symbol(libsjd):
    from paper_2603_18599_gb300 import sjd
    names = declared_functions()
    for n in names:
        assert hasattr(libsjd, n), n
    nm = shutil.which("nm")
    if nm:
        out = subprocess.run([nm, "-D", "--defined-only", sjd.lib_path()], capture_output=True,
                             text=True).stdout
        exported = set(line.split()[-1] for line in out.splitlines() if line.strip())
        assert set(names) <= exported


def test_checked_build_exports_every_declared_symbol(libsjd):
    from paper_2603_18599_gb300 import _build
    if not os.path.exists(_build.LIB_CHECKED):
        pytest.skip("libsjd_checked.so not built")
    lib = ctypes.CDLL(_build.LIB_CHECKED)
    for n in declared_functions():
        assert hasattr(lib, n), n


def test_config_struct_matches_header(libsjd):
    from paper_2603_18599_gb300 import sjd
    # int32 x5, float x2, int32, float, int32 x3, pad, uint64, int32 x4
    assert ctypes.sizeof(sjd.sjd_config) == 72
    assert sjd.sjd_config.seed.offset == 48
    assert sjd.sjd_config.pd_tree.offset == 68


def test_workspace_size_validates_configs(libsjd):
    from paper_2603_18599_gb300 import sjd
    good = sjd.make_config(16, 64, 65536, 4, 8196, top_k=2000, top_p=0.9)
    n = sjd.workspace_size(good)
    assert n > 16 * 64 * 2000 * 8
    bad = [
        dict(batch=0), dict(window=0), dict(window=2000), dict(allowed_lo=9000),
        dict(top_p=0.0), dict(top_p=1.5), dict(pd_k=0), dict(pd_k=9), dict(temperature=0.0),
        dict(support_cap=10), dict(logit_dtype=7), dict(adaptive_continuation=2),
        dict(max_steps=0), dict(top_k=-1), dict(pd_tree=2),
        dict(pd_tree=1, adaptive_continuation=0), dict(pd_tree=1, pd_k=1), dict(pd_tree=1, pd_depth=0),
        dict(pd_tree=1, pd_k=8, pd_depth=3),
    ]
    for kw in bad:
        c = sjd.make_config(16, 64, 65536, 4, 8196, top_k=2000, top_p=0.9)
        for k, v in kw.items():
            setattr(c, k, v)
        assert sjd.workspace_size(c) == 0, kw


def test_init_rejects_bad_arguments_before_touching_the_device(libsjd):
    from paper_2603_18599_gb300 import sjd
    ctx = ctypes.c_void_p()
    bad = sjd.make_config(1, 4, 64, 0, 64, top_k=0)
    bad.batch = 0
    assert libsjd.sjd_init(ctypes.byref(bad), ctypes.c_void_p(256), 1 << 20, None,
                           ctypes.byref(ctx)) == sjd.SJD_ERR_ARG
    good = sjd.make_config(1, 4, 64, 0, 64, top_k=0)
    # NULL or misaligned workspace
    assert libsjd.sjd_init(ctypes.byref(good), None, 1 << 20, None, ctypes.byref(ctx)) == sjd.SJD_ERR_ARG
    assert libsjd.sjd_init(ctypes.byref(good), ctypes.c_void_p(8), 1 << 20, None,
                           ctypes.byref(ctx)) == sjd.SJD_ERR_ARG
    # NULL handle is reported, not dereferenced
    assert libsjd.sjd_sync(None) == sjd.SJD_ERR_ARG
    assert libsjd.sjd_step(None, None, None, None, None, None) == sjd.SJD_ERR_ARG
    assert libsjd.sjd_last_error(None) == b"no context"


def test_product_path_has_no_oracle_dependency():
    """The library and its binding never import, load or run the oracle."""
    pkg = os.path.join(ROOT, "paper_2603_18599_gb300")
    pat = re.compile(r"^\s*(from\s+oracle|import\s+oracle)|oracle[/\\]", re.M)
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".h", ".cuh")):
                assert not pat.search(open(os.path.join(dirpath, f)).read()), f
