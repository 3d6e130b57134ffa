"""Throughput of the fused SJD-PAC verify-and-draft step on GB300.

Workload (the largest of the five synthetic workloads): B=16 images, Jacobi
window W=64, vocabulary V=65536 bf16 logits N(0, 3^2), sampling restricted
to the 8192 image ids [4, 8196), CFG 3, temperature 1, top-k 2000, top-p 0.9,
K=4, D=3, Philox seed 1234, 50 chained steps on distinct logit buffers.

Prints one JSON line: verified draft positions per second (B*W per step),
with the roofline of the row kernel against the measured HBM bandwidth.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the CPU oracle (the reference arm of this build) on
bounded samples of the same workload.
"""

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "b16w64v65536_bf16_mask8192_topp09"
N_BUFFERS = 50
METRIC = "verified draft positions/sec"
KERNEL_SOURCES = ["sjd_fast.cuh", "sjd_device.cuh", "sjd_internal.h", "sjd_api.cu"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "stream_row_kernel_b16w64v65536_bf16.traffic.txt")


def code_without_comments(text):
    """C/C++/CUDA source with its comments and blank lines removed (string and
    character literals kept), so that a comment edit leaves the digest alone."""
    out, i, n = [], 0, len(text)
    while i < n:
        c = text[i]
        if c in "\"'":
            j = i + 1
            while j < n and text[j] != c:
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        elif text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
        else:
            out.append(c)
            i += 1
    lines = ("".join(out)).split("\n")
    return "\n".join(ln.rstrip() for ln in lines if ln.strip())


def kernel_source_digest():
    """sha256 over the code (comments removed) of the fast kernel's sources."""
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2603_18599_gb300", "csrc", f)) as fh:
            h.update(code_without_comments(fh.read()).encode())
    return h.hexdigest()


def measured_traffic():
    """DRAM bytes per launch of the fast row kernel from the committed ncu
    capture, or None when the kernel sources have changed since."""
    try:
        rec = {}
        with open(TRAFFIC_FILE) as fh:
            for ln in fh:
                if ln.startswith("#") or ":" not in ln:
                    continue
                k, v = ln.split(":", 1)
                rec[k.strip()] = v.strip()
        if rec.get("source_sha256") != kernel_source_digest():
            return None
        return int(rec["dram_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


def rank_seed(base_seed, rank):
    """Weak scaling: every rank decodes its own B images, with its own inputs
    and Philox key."""
    return base_seed + rank


def job_region_ms(local_ms, world, device=None):
    """Timed region of the whole job: the maximum over the ranks (every rank
    calls this; with one rank it is the local time)."""
    if world <= 1:
        return float(local_ms)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(local_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(world, batch, window, ms_per_step):
    """Whole-job verified draft positions per second: every rank verifies
    batch * window positions per step."""
    return world * batch * window / (ms_per_step * 1e-3)


def reports(rank):
    """Only rank 0 prints the JSON line (the other ranks exit 0 quietly)."""
    return rank == 0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--buffers", type=int, default=N_BUFFERS, help="distinct step inputs (>= 2)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the other four workloads")
    ap.add_argument("--no-graph", action="store_true", help="launch the timed steps one by one, not as a CUDA graph")
    ap.add_argument("--wait-logits", action="store_true",
                    help="every step waits for the one before it before reading its logits")
    return ap.parse_args()


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.2)
        self.proc.terminate()
        self.proc.wait()
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax = float(parts[2])
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


def make_config(wl, sjd, seed):
    return sjd.make_config(wl.batch, wl.window, wl.vocab, wl.lo, wl.hi, wl.cfg_scale, wl.temperature,
                           wl.top_k, wl.top_p, wl.pd_k, wl.pd_depth, wl.ac, seed, sjd.SJD_BF16)


def workload_config(wl):
    """The workload keys of the JSON line's config, the same on both arms."""
    return {"workload": wl.name, "batch": wl.batch, "window": wl.window, "vocab": wl.vocab,
            "allowed": [wl.lo, wl.hi], "top_k": wl.top_k, "top_p": wl.top_p, "cfg": wl.cfg_scale,
            "pd_k": wl.pd_k, "pd_depth": wl.pd_depth}


def algorithmic_bytes(wl, rows, nq, np_, steps):
    """Sum over rows of 2*V_eff*e (cond+uncond of the allowed range, e = 2
    for bf16, 4 for fp32) + 8 n_q (draft row read) + 8 n_p (target row
    written) + 12 (draft, token, flag), plus 4 (K-1) D B per step for the PD
    groups."""
    e = 2 if wl.dtype == "bf16" else 4
    return rows * (2 * wl.v_eff * e + 12) + 8 * (nq + np_) + 4 * (wl.pd_k - 1) * wl.pd_depth * wl.batch * steps


def cpu_baseline(wl, budget_s=12.0):
    """The oracle as it stands, one batch element's window per step, on the
    host cores (one thread), for about budget_s seconds."""
    from oracle import sjd_oracle as so
    from paper_2603_18599_gb300 import workloads as wlm
    P = so.Params(batch=wl.batch, window=wl.window, vocab=wl.vocab, lo=wl.lo, hi=wl.hi,
                  cfg_scale=wl.cfg_scale, temperature=wl.temperature, top_k=wl.top_k, top_p=wl.top_p,
                  pd_k=wl.pd_k, pd_depth=wl.pd_depth, ac=wl.ac, seed=wl.seed)
    st = so.init_state(P, 0, [0])
    c, u, qc, qu = wlm.logits_step(wl, 0, batches=[0])
    so.draft_from_logits(P, st, 0, qc, qu)
    steps, elapsed, t = 0, 0.0, 0
    while elapsed < budget_s:
        c, u, _, _ = wlm.logits_step(wl, t, batches=[0])
        t0 = time.perf_counter()
        so.step(P, st, t, c, u)
        elapsed += time.perf_counter() - t0
        steps += 1
        t += 1
    return {"value": steps * wl.window / elapsed, "unit": "positions/s", "cores": 1, "kind": "oracle",
            "sample": "%d chained steps of one batch element (%d rows x V_eff %d) of %s, %.1f s"
                      % (steps, wl.window, wl.v_eff, wl.name, elapsed)}


def _oracle_worker(job):
    """One host process of the all-cores oracle baseline: chained steps of one
    batch element for about budget_s seconds of oracle time."""
    name, b, budget_s = job
    from oracle import sjd_oracle as so
    from paper_2603_18599_gb300 import workloads as wlm
    wl = wlm.workloads()[name]
    P = so.Params(batch=wl.batch, window=wl.window, vocab=wl.vocab, lo=wl.lo, hi=wl.hi,
                  cfg_scale=wl.cfg_scale, temperature=wl.temperature, top_k=wl.top_k, top_p=wl.top_p,
                  pd_k=wl.pd_k, pd_depth=wl.pd_depth, ac=wl.ac, seed=wl.seed)
    st = so.init_state(P, 0, [b])
    _, _, qc, qu = wlm.logits_step(wl, 0, batches=[b])
    so.draft_from_logits(P, st, 0, qc, qu)
    steps, elapsed, t = 0, 0.0, 0
    while elapsed < budget_s:
        c, u, _, _ = wlm.logits_step(wl, t, batches=[b])
        t0 = time.perf_counter()
        so.step(P, st, t, c, u)
        elapsed += time.perf_counter() - t0
        steps += 1
        t += 1
    return steps, elapsed


def cpu_baseline_all_cores(wl, budget_s=12.0):
    """The same oracle on every host core at once: one single-threaded
    process per core (started with spawn), each on its own batch element
    (the batch elements are independent); the rates add up."""
    import multiprocessing as mp
    n = os.cpu_count() or 1
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    for k in saved:
        os.environ[k] = "1"
    try:
        with mp.get_context("spawn").Pool(n) as pool:
            res = pool.map(_oracle_worker, [(wl.name, i % wl.batch, budget_s) for i in range(n)])
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    rate = sum(st * wl.window / el for st, el in res)
    return {"value": rate, "unit": "positions/s", "cores": n, "kind": "oracle",
            "sample": "%d processes, each %d chained steps on average of one batch element (%d rows x V_eff %d) "
                      "of %s, %.1f s each" % (n, round(sum(r[0] for r in res) / n), wl.window, wl.v_eff, wl.name,
                                             budget_s)}


def run_reference(args):
    rank, _, world = dist_env()
    if not reports(rank):
        return
    from paper_2603_18599_gb300 import workloads as wlm
    wl = wlm.workloads()[WORKLOAD]
    t_total = 0.0
    from oracle import sjd_oracle as so
    P = so.Params(batch=wl.batch, window=wl.window, vocab=wl.vocab, lo=wl.lo, hi=wl.hi,
                  cfg_scale=wl.cfg_scale, temperature=wl.temperature, top_k=wl.top_k, top_p=wl.top_p,
                  pd_k=wl.pd_k, pd_depth=wl.pd_depth, ac=wl.ac, seed=wl.seed)
    st = so.init_state(P, 0, [0])
    c, u, qc, qu = wlm.logits_step(wl, 0, batches=[0])
    so.draft_from_logits(P, st, 0, qc, qu)
    for i in range(args.warmup + args.steps):
        c, u, _, _ = wlm.logits_step(wl, i, batches=[0])
        t0 = time.perf_counter()
        so.step(P, st, i, c, u)
        if i >= args.warmup:
            t_total += time.perf_counter() - t0
    value = args.steps * wl.window / t_total
    sample = ("each step: one batch element's window (%d rows x V_eff %d) of %s, chained"
              % (wl.window, wl.v_eff, wl.name))
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "positions/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t_total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32+int64",
        "data": "synthetic", "config": workload_config(wl),
        "cpu_baseline": {"value": value, "unit": "positions/s", "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "positions/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def device_logits(wl, g, dev, dominant=True):
    """Synthetic [B, W, V] bf16 cond/uncond of a workload drawn on the device
    (the recipe of workloads.logits_row: N(0, sigma_b^2), poison outside the
    allowed range, one +boost id on a fraction of the rows)."""
    import torch
    B, W, V = wl.batch, wl.window, wl.vocab
    sig = torch.tensor([wl.sigma_of(b) for b in range(B)], device=dev).view(B, 1, 1)
    out = []
    for _ in range(2):
        x = torch.randn((B, W, V), generator=g, device=dev) * sig
        x[:, :, :wl.lo] = 64.0
        x[:, :, wl.hi:] = 64.0
        out.append(x)
    if dominant and wl.dominant_frac > 0:
        n = int(round(wl.dominant_frac * B * W))
        rows = torch.randperm(B * W, generator=g, device=dev)[:n]
        ids = torch.randint(wl.lo, wl.hi, (n,), generator=g, device=dev)
        for x in out:
            x.view(B * W, V)[rows, ids] += wl.dominant_boost
    return [x.to(torch.bfloat16) if wl.dtype == "bf16" else x for x in out]


def other_configs(dev, early=True):
    """Fused-step throughput of the other synthetic workloads and the full
    32x32 decode with the seeded stand-in model (acceptance length per step)."""
    import torch
    from paper_2603_18599_gb300 import sjd
    from paper_2603_18599_gb300 import workloads as wlm
    W_ = wlm.workloads()
    res = {}
    for name, n_buf, steps in (("b1w16v8192_f32", 8, 200), ("b8w32v16384_bf16_sigma1to5", 8, 200),
                               ("b4w32v32768_bf16_dominant_chain100", 100, 100)):
        wl = W_[name]
        g = torch.Generator(device=dev)
        g.manual_seed(wl.seed)
        dt = sjd.SJD_BF16 if wl.dtype == "bf16" else sjd.SJD_F32
        bufs = []
        for _ in range(n_buf):
            bufs.append(tuple(device_logits(wl, g, dev)))
        cfg = sjd.make_config(wl.batch, wl.window, wl.vocab, wl.lo, wl.hi, wl.cfg_scale, wl.temperature,
                              wl.top_k, wl.top_p, wl.pd_k, wl.pd_depth, wl.ac, wl.seed, dt)
        ctx = sjd.SJD(cfg, dev)
        ctx.draft_from_logits(*bufs[0])
        if early:  # resident inputs: consecutive steps may overlap
            ctx.set_early_logits(True)
        for i in range(3):
            ctx.step_raw(bufs[i % n_buf][0].data_ptr(), bufs[i % n_buf][1].data_ptr())
        torch.cuda.synchronize()
        s0 = ctx.stats()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(ctx.stream):
            e0.record(ctx.stream)
            for i in range(steps):
                c, u = bufs[i % n_buf]
                ctx.step_raw(c.data_ptr(), u.data_ptr())
            e1.record(ctx.stream)
        torch.cuda.synchronize()
        assert ctx.sync() == 0, ctx.last_error()
        ms = e0.elapsed_time(e1) / steps
        s1 = ctx.stats()
        per_launch = algorithmic_bytes(wl, s1[0] - s0[0], s1[1] - s0[1], s1[2] - s0[2], steps) / steps
        peak, peak_kind = peaks()
        achieved = per_launch / (ms * 1e-3) / 1e9
        input_bytes = n_buf * 2 * wl.batch * wl.window * wl.v_eff * (2 if wl.dtype == "bf16" else 4)
        res[name] = {"positions_per_s": wl.batch * wl.window / (ms * 1e-3), "us_per_step": ms * 1e3,
                     "steps": steps, "distinct_inputs": n_buf, "steps_overlap": early,
                     "row_kernel": "fast" if ctx.row_path() == 1 else "general",
                     "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                                  "frac": achieved / peak, "peak_kind": peak_kind,
                                  "algorithmic_bytes_per_launch": per_launch,
                                  "inputs": "%d buffers, %.0f MB of allowed-range logits (%s the 129 MB L2)"
                                            % (n_buf, input_bytes / 1e6, "above" if input_bytes > 129e6 else "NOT above")}}
        ctx.close()
        del bufs
    # full decodes with the seeded stand-in model evaluated on the device
    def standin_forward(m, window):
        E_out = torch.tensor(m.E_out, dtype=torch.float32, device=dev)
        E_in = torch.tensor(m.E_in, dtype=torch.float32, device=dev)
        Pp = torch.tensor(m.P, dtype=torch.float32, device=dev)

        def fwd(win, prev, pos, cond_out, uncond_out):
            prev_tok = torch.cat([prev.view(1, 1), win[:, :-1]], dim=1).long()
            p = torch.clamp(pos.view(1, 1).long() + torch.arange(window, device=dev).view(1, -1), max=m.n_pos - 1)
            e = E_in[prev_tok]
            cond_out.copy_((torch.tanh(e + Pp[p]) @ E_out.T).to(torch.bfloat16))
            uncond_out.copy_((torch.tanh(e) @ E_out.T).to(torch.bfloat16))
        return fwd

    def decode(wl, fwd, n_tokens, k, d, ac, accept_len=False):
        cfg = sjd.make_config(1, wl.window, wl.vocab, wl.lo, wl.hi, wl.cfg_scale, wl.temperature, wl.top_k,
                              wl.top_p, k, d, ac, wl.seed, sjd.SJD_BF16, max_steps=n_tokens)
        c = sjd.SJD(cfg, dev)
        cbuf = torch.empty((1, wl.window, wl.vocab), dtype=torch.bfloat16, device=dev)
        ubuf = torch.empty_like(cbuf)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        grid, acc, steps = c.decode_loop(fwd, n_tokens, cbuf, ubuf, accept_len=accept_len)
        torch.cuda.synchronize()
        dt_s = time.perf_counter() - t0
        acc = acc[:steps, 0].cpu().tolist() if accept_len else None
        c.close()
        return steps, acc, dt_s

    wl = W_["decode32x32_b1w16v8192_bf16"]
    fwd = standin_forward(wlm.StandInModel(), wl.window)
    decode(wl, fwd, 1024, wl.pd_k, wl.pd_depth, wl.ac)  # untimed: first use of the forward's libraries
    steps, acc, dt_s = decode(wl, fwd, 1024, wl.pd_k, wl.pd_depth, wl.ac, accept_len=True)
    # the paper's component ablation on the stand-in: step compression of
    # vanilla SJD, +PD, +AC and SJD-PAC (same model, seed and grid)
    ablation = {}
    for label, ac, k, d in (("sjd", 0, 1, 0), ("sjd+pd", 0, wl.pd_k, wl.pd_depth), ("sjd+ac", 1, 1, 0),
                            ("sjd-pac", 1, wl.pd_k, wl.pd_depth)):
        n_st = decode(wl, fwd, 1024, k, d, ac)[0]
        ablation[label] = {"steps": n_st, "accepted_per_step": 1024 / n_st}
    # proactive-drafting factors: candidates per position K and positions D (AC on)
    sweep = {}
    for k in (2, 4, 8):
        for d in (1, 3, 5):
            n_st = decode(wl, fwd, 1024, k, d, 1)[0]
            sweep["K%d_D%d" % (k, d)] = {"steps": n_st, "accepted_per_step": 1024 / n_st}
    res[wl.name] = {"tokens": 1024, "steps": steps, "mean_accepted_per_step": 1024 / steps,
                    "ablation_W16": ablation, "pd_sweep_W16": sweep,
                    "max_accepted_per_step": max(acc), "tokens_per_s_with_standin_forward": 1024 / dt_s,
                    "ms_per_step_with_standin_forward": dt_s * 1e3 / steps,
                    "note": "stand-in forward in torch on the device and a host callback per step; the "
                            "positions are read back after ceil(remaining / W) steps"}
    # a larger grid and vocabulary: 90 x 90 tokens, V = 32768; acceptance-length
    # histograms of vanilla SJD and SJD-PAC
    wl = W_["decode90x90_b1w16v32768_bf16"]
    fwd = standin_forward(wlm.StandInModel(vocab=wl.vocab, n_pos=8192), wl.window)
    big = {"tokens": 8100}
    for label, ac, k, d in (("sjd", 0, 1, 0), ("sjd-pac", 1, wl.pd_k, wl.pd_depth)):
        n_st, acc, dt_s = decode(wl, fwd, 8100, k, d, ac, accept_len=True)
        hist = [0] * (wl.window + 1)
        for a in acc:
            hist[a] += 1
        big[label] = {"steps": n_st, "accepted_per_step": 8100 / n_st, "accept_len_hist": hist,
                      "tokens_per_s_with_standin_forward": 8100 / dt_s}
    res[wl.name] = big
    # the full K-ary proactive-drafting tree against the main-path groups, on
    # sharper stand-in models (weights N(0, 0.3^2)) whose targets depend on
    # the context, so that the tree's per-node targets matter; W = 16, K = 4,
    # D = 3: 32 x 32 tokens with V = 1024 (top-k 200), and the 90 x 90 grid
    # with V = 32768 (top-k 2000)
    def tree_vs_main_path(wl, m, n_tokens, label_model):
        E_out = torch.tensor(m.E_out, dtype=torch.float32, device=dev)
        E_in = torch.tensor(m.E_in, dtype=torch.float32, device=dev)
        Pp = torch.tensor(m.P, dtype=torch.float32, device=dev)
        K, D, W = wl.pd_k, wl.pd_depth, wl.window
        nd, ns = [], []  # depth and token slot of every node row
        for d in range(1, D):
            for i in range(1, K ** d):
                nd.append(d)
                ns.append(sum(K ** e for e in range(1, d)) + i)
        nd_t = torch.tensor(nd, dtype=torch.long, device=dev)
        ns_t = torch.tensor(ns, dtype=torch.long, device=dev)
        out = {"tokens": n_tokens, "model": label_model}
        for label, tree in (("main_path_groups", 0), ("full_tree", 1)):
            cfg = sjd.make_config(1, W, wl.vocab, wl.lo, wl.hi, wl.cfg_scale, wl.temperature, wl.top_k, wl.top_p,
                                  K, D, 1, wl.seed, sjd.SJD_BF16, max_steps=n_tokens, pd_tree=tree)
            c = sjd.SJD(cfg, dev)
            n = steps = 0
            hist = [0] * (W + 1)
            while n < n_tokens and steps < n_tokens:
                tok, _, _, pos, prev = c.get_window()
                rows_prev = torch.cat([prev.view(1), tok[0, :-1]]).long()
                rows_pos = torch.clamp(pos.long() + torch.arange(W, device=dev), max=m.n_pos - 1)
                if tree:
                    ttok, _ = c.get_tree()
                    rows_prev = torch.cat([rows_prev, torch.clamp(ttok[0, ns_t].long(), min=0)])
                    rows_pos = torch.cat([rows_pos, torch.clamp(pos.long() + nd_t, max=m.n_pos - 1)])
                e = E_in[rows_prev]
                cond = (torch.tanh(e + Pp[rows_pos]) @ E_out.T).to(torch.bfloat16).unsqueeze(0).contiguous()
                uncond = (torch.tanh(e) @ E_out.T).to(torch.bfloat16).unsqueeze(0).contiguous()
                _, nc, _ = c.step(cond, uncond)
                take = min(int(nc[0]), n_tokens - n)
                hist[take] += 1
                n += take
                steps += 1
            assert c.sync() == 0, c.last_error()
            out[label] = {"steps": steps, "accepted_per_step": n / steps, "accept_len_hist": hist}
            c.close()
        return out

    wl = W_["decode32x32_b1w16v8192_bf16"].scaled(vocab=1024, hi=1024, top_k=200)
    res["tree_vs_main_path_standin_sharp"] = tree_vs_main_path(
        wl, wlm.StandInModel(vocab=1024, std=0.3), 1024,
        "stand-in, weights N(0, 0.3^2), V 1024, top-k 200, W 16, K 4, D 3")
    wl = W_["decode90x90_b1w16v32768_bf16"]
    res["tree_vs_main_path_90x90_standin_sharp"] = tree_vs_main_path(
        wl, wlm.StandInModel(vocab=wl.vocab, n_pos=8192, std=0.3), 8100,
        "stand-in, weights N(0, 0.3^2), V 32768, top-k 2000, W 16, K 4, D 3, 90 x 90 tokens")
    return res


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2603_18599_gb300 import sjd
    from paper_2603_18599_gb300 import workloads as wlm

    rank, local, world = dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    wl = wlm.workloads()[WORKLOAD]
    seed = rank_seed(wl.seed, rank)  # weak scaling: every rank decodes its own B images
    B, W, V = wl.batch, wl.window, wl.vocab
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    # 50 distinct step inputs: cond and uncond N(0, 3^2), bf16, [B, W, V]
    conds, unconds = [], []
    for _ in range(args.buffers):
        conds.append((torch.randn((B, W, V), generator=g, device=dev) * wl.sigma).to(torch.bfloat16))
        unconds.append((torch.randn((B, W, V), generator=g, device=dev) * wl.sigma).to(torch.bfloat16))
    noise = torch.randn((B, W, V), generator=g, device=dev) * wl.q_noise
    qc = (conds[0].float() + noise).to(torch.bfloat16)
    qu = (unconds[0].float() + noise).to(torch.bfloat16)
    del noise
    torch.cuda.synchronize()  # inputs ready before the library's stream reads them
    stream = torch.cuda.Stream(dev)
    ctx = sjd.SJD(make_config(wl, sjd, seed), dev, stream=stream)
    ctx.draft_from_logits(qc, qu)
    # the step inputs are resident before the timed region: consecutive steps
    # may overlap (each streams its logits while the one before finishes)
    if not args.wait_logits:
        ctx.set_early_logits(True)
    cptr = [c.data_ptr() for c in conds]
    uptr = [u.data_ptr() for u in unconds]
    for i in range(args.warmup):
        rc = ctx.step_raw(cptr[i % args.buffers], uptr[i % args.buffers])
        assert rc == 0, ctx.last_error()
    torch.cuda.synchronize()
    assert ctx.sync() == 0, ctx.last_error()
    s0 = ctx.stats()
    # the timed steps: one launch each, captured once as a CUDA graph (the
    # launches themselves, as a decode loop would replay them)
    graph = None
    if not args.no_graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for i in range(args.steps):
                k = (args.warmup + i) % args.buffers
                ctx.step_raw(cptr[k], uptr[k])
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    clocks.start()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        t_start.record(stream)
        if graph is not None:
            graph.replay()
        else:
            for i in range(args.steps):
                k = (args.warmup + i) % args.buffers
                ctx.step_raw(cptr[k], uptr[k])
        t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    rc = ctx.sync()
    assert rc == 0, ctx.last_error()
    region_ms = t_start.elapsed_time(t_end)
    # every launch in the region is the step kernel, back to back: its mean
    # duration is the region over the launches (launch gaps included)
    kernel_ms = region_ms / args.steps
    s1 = ctx.stats()
    rows, nq, np_ = s1[0] - s0[0], s1[1] - s0[1], s1[2] - s0[2]
    region_ms = job_region_ms(region_ms, world, dev)
    ms_per_step = region_ms / args.steps
    value = job_value(world, B, W, ms_per_step)
    bytes_per_launch = algorithmic_bytes(wl, rows, nq, np_, args.steps) / args.steps
    fast = ctx.row_path() == 1
    traffic = measured_traffic() if fast else None
    peak, peak_kind = peaks()
    achieved = bytes_per_launch / (kernel_ms * 1e-3) / 1e9

    # end to end through the public API with host inputs: sjd_step_host takes
    # the pinned host logits and copies their allowed columns across the host
    # link into two alternating device stages (a step's copy overlapping the
    # step before); every step's committed tokens, commit count and first
    # rejection are copied back into a pinned ring, with no synchronisation
    # between steps
    e2e = None
    if not args.no_e2e:
        n_l = ((wl.hi + 7) // 8) * 8 - (wl.lo // 8) * 8  # allowed columns read per row
        step_bytes = 2 * B * W * n_l * 2
        # host buffers holding more than four times the L2 of allowed-range data
        nh = max(3, -(-4 * 129 * 10 ** 6 // step_bytes))
        host_c = [conds[i % args.buffers].cpu().pin_memory() for i in range(nh)]
        host_u = [unconds[i % args.buffers].cpu().pin_memory() for i in range(nh)]
        stage = ctx.host_stage()
        out_c = torch.empty((B, W), dtype=torch.int32, device=dev)
        out_n = torch.empty((B,), dtype=torch.int32, device=dev)
        out_f = torch.empty((B,), dtype=torch.int32, device=dev)
        e_steps = min(args.steps, 64)
        ring_c = torch.empty((e_steps, B, W), dtype=torch.int32).pin_memory()
        ring_n = torch.empty((e_steps, B), dtype=torch.int32).pin_memory()
        ring_f = torch.empty((e_steps, B), dtype=torch.int32).pin_memory()
        for i in range(2):  # untimed
            ctx.step_host(host_c[i % nh], host_u[i % nh], stage, out=(out_c, out_n, out_f))
        # the link's measured peak: one pinned host-to-device copy of 1 GiB
        big_h = torch.empty(1 << 30, dtype=torch.uint8).pin_memory()
        big_d = torch.empty(1 << 30, dtype=torch.uint8, device=dev)
        h2d_gbs = 0.0
        with torch.cuda.stream(stream):
            for _ in range(3):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                big_d.copy_(big_h, non_blocking=True)
                b.record(stream)
                b.synchronize()
                h2d_gbs = max(h2d_gbs, (1 << 30) / (a.elapsed_time(b) * 1e-3) / 1e9)
        del big_h, big_d
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        with torch.cuda.stream(stream):
            for i in range(e_steps):
                ctx.step_host(host_c[i % nh], host_u[i % nh], stage, out=(out_c, out_n, out_f))
                ring_c[i].copy_(out_c, non_blocking=True)
                ring_n[i].copy_(out_n, non_blocking=True)
                ring_f[i].copy_(out_f, non_blocking=True)
        stream.synchronize()
        e2e_s = time.perf_counter() - t0
        assert int(ring_n.min()) >= 1
        e2e = {"value": world * B * W * e_steps / e2e_s, "unit": "positions/s",
               "h2d_bytes_per_step": step_bytes, "d2h_bytes_per_step": B * (W + 2) * 4,
               "steps": e_steps, "host_buffers": nh,
               "host_data_gb": round(nh * step_bytes / 1e9, 3),
               "h2d_link_gbs": step_bytes * e_steps / e2e_s / 1e9,
               "h2d_peak_gbs_measured": h2d_gbs,
               "link_frac": (step_bytes * e_steps / e2e_s / 1e9) / h2d_gbs if h2d_gbs else None,
               "call": "sjd_step_host (allowed columns of pinned host rows copied into two alternating device "
                       "stages, each step's copy overlapping the step before); results copied to a pinned ring "
                       "every step, one synchronisation at the end"}
        assert ctx.sync() == 0, ctx.last_error()

    if not reports(rank):
        if world > 1:
            dist.destroy_process_group()
        return
    cpu = None if (args.no_cpu_baseline or world > 1) else cpu_baseline(wl)
    cpu_all = None if (args.no_cpu_baseline or world > 1) else cpu_baseline_all_cores(wl)
    others = None if (args.no_configs or world > 1) else other_configs(dev, early=not args.wait_logits)
    line = {
        "metric": METRIC, "value": value, "unit": "positions/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 in, f32 + int64 compute", "data": "synthetic",
        "config": {**workload_config(wl), "chained_steps_on_distinct_buffers": args.buffers,
                   "launch": "one CUDA graph of the timed steps" if graph is not None else "stream launches",
                   "steps_overlap": not args.wait_logits,
                   "l2": "inputs rotate over %d buffers (%.2f GB of allowed-range logits, %s the 129 MB L2)"
                         % (args.buffers, args.buffers * B * W * wl.v_eff * 4 / 1e9,
                            "above" if args.buffers * B * W * wl.v_eff * 4 > 129e6 else "NOT above")},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "peak_kind": peak_kind,
                     "kernel": "stream_row_kernel (fused step)" if fast else "row_kernel (fused step, general)",
                     "kernel_ms": kernel_ms,
                     "kernel_ms_is": "the timed region over the launches (consecutive launches overlap: "
                                     "each streams its logits while the one before finishes)"
                                     if not args.wait_logits else "the timed region over the launches",
                     "algorithmic_bytes_per_launch": bytes_per_launch},
        "cpu_baseline": cpu,
        "cpu_baseline_all_cores": cpu_all,
        "e2e": e2e,
        "gpu_launches": args.steps,
        "clocks": clk,
        "other_workloads": others,
    }
    print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
