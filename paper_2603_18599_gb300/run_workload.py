"""Runs one of the named synthetic workloads (workloads.workloads()) through
the library: a draft from step 0's draft logits, then chained fused steps on
the following steps' logits, each one timed with CUDA events on the
context's stream. Prints one line per step and the mean.

    python -m paper_2603_18599_gb300.run_workload b8w32v16384_bf16_sigma1to5 --steps 3
"""

import argparse

import torch

from . import sjd
from . import workloads as wlm


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("workload", choices=sorted(wlm.workloads()))
    ap.add_argument("--steps", type=int, default=3)
    args = ap.parse_args()
    w = wlm.workloads()[args.workload]
    dev = torch.device("cuda", torch.cuda.current_device())
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32

    def dev_logits(arrays):
        return [torch.from_numpy(a).to(dev).to(dt) for a in arrays]

    cfg = sjd.make_config(w.batch, w.window, w.vocab, w.lo, w.hi, w.cfg_scale, w.temperature, w.top_k, w.top_p,
                          w.pd_k, w.pd_depth, w.ac, w.seed, sjd.SJD_BF16 if w.dtype == "bf16" else sjd.SJD_F32)
    ctx = sjd.SJD(cfg, dev)
    ctx.draft_from_logits(*dev_logits(wlm.logits_step(w, 0)[2:]))
    times = []
    for t in range(1, args.steps + 1):
        c, u = dev_logits(wlm.logits_step(w, t)[:2])
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(ctx.stream):
            a.record(ctx.stream)
            ctx.step(c, u)
            b.record(ctx.stream)
        b.synchronize()
        times.append(a.elapsed_time(b) * 1e3)
        print("step %d: %.1f us" % (t, times[-1]))
    rc = ctx.sync()
    if rc != sjd.SJD_OK:
        raise SystemExit("status %d: %s" % (rc, ctx.last_error()))
    print("%s: %d steps, mean %.1f us per step (%s row kernel)" % (
        args.workload, len(times), sum(times) / len(times), "fast" if ctx.row_path() == 1 else "general"))


if __name__ == "__main__":
    main()
