"""Build libsjd.so (the CUDA library behind include/sjd.h) in-tree for sm_103a,
and libsjd_checked.so, the same library with its device-side bounds checks
on (SJD_CHECKS: an index outside its array latches SJD_ERR_BOUNDS and is
clamped, never trapping).

Every translation unit of both is compiled in parallel with nvcc, then
linked into paper_2603_18599_gb300/_build/ (git-ignored).
"""

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
OUT = os.path.join(PKG, "_build")
LIB = os.path.join(OUT, "libsjd.so")
LIB_CHECKED = os.path.join(OUT, "libsjd_checked.so")
SOURCES = ["sjd_kernels.cu", "sjd_fast.cu", "sjd_api.cu", "sjd_noalloc.cu"]
# the fast row kernels: sjd_fast_part.cu once per (dtype, mode) pair
FAST_PARTS = [(dt, mode) for dt in ("SJD_BF16", "SJD_F32") for mode in ("kModeVerify", "kModeStep", "kModeFromLogits")]
ARCH = "-gencode=arch=compute_103a,code=sm_103a"


def nvcc():
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libsjd.so")


def _flags():
    return [ARCH, "-lineinfo", "-O3", "-std=c++17", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
            "-I", os.path.join(ROOT, "include"), "-I", CSRC]


def build(verbose=False, extra_flags=()):
    """Compile and link libsjd.so and libsjd_checked.so; returns the first's path."""
    os.makedirs(os.path.join(OUT, "checked"), exist_ok=True)
    cc = nvcc()

    def one(job):
        src, sub, defs, name = job
        obj = os.path.join(OUT, sub, name + ".o")
        cmd = [cc, *_flags(), *defs, *extra_flags, "-c", os.path.join(CSRC, src), "-o", obj]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("nvcc failed for %s:\n%s\n%s" % (src, " ".join(cmd), r.stderr))
        if verbose and r.stderr:
            sys.stderr.write(r.stderr)
        return obj

    units = [(src, [], os.path.splitext(src)[0]) for src in SOURCES]
    units += [("sjd_fast_part.cu", ["-DSJD_FAST_DT=" + dt, "-DSJD_FAST_MODE=" + mode],
               "sjd_fast_%s_%s" % (dt[4:].lower(), mode[5:].lower())) for dt, mode in FAST_PARTS]
    jobs = [(src, "", defs, name) for src, defs, name in units]
    jobs += [(src, "checked", defs + ["-DSJD_CHECKS"], name) for src, defs, name in units]
    # the longest units first
    order = sorted(range(len(jobs)), key=lambda i: jobs[i][0] != "sjd_fast_part.cu")
    with ThreadPoolExecutor(min(len(jobs), max(4, os.cpu_count() or 4))) as ex:
        done = dict(zip(order, ex.map(one, [jobs[i] for i in order])))
    objs = [done[i] for i in range(len(jobs))]
    for lib, part in ((LIB, objs[:len(units)]), (LIB_CHECKED, objs[len(units):])):
        tmp = lib + ".tmp"
        cmd = [cc, ARCH, "-shared", "-o", tmp, *part]
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("link failed:\n%s\n%s" % (" ".join(cmd), r.stderr))
        os.replace(tmp, lib)
    return LIB


if __name__ == "__main__":
    print(build(verbose="-v" in sys.argv))
