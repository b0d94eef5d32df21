#!/usr/bin/env python
"""Benchmark of the ELSAA forward operator on GB300.

One step = one elsaa_forward over the whole workload (all B*H heads: sort
hash, stable sort, RACE summaries, block attention, RACE readout, fusion).
Default workload: B=2, H=16, N=16384, d_h=128, bf16, block b=128, RACE
r = 256 (L_s = 16, gamma = 4), non-causal. Prints ONE JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the CPU oracle (fp64, host cores) on bounded samples
of the same workload. Under torchrun (N > 1) every rank runs its own copy of
the workload on its own GPU (heads are independent: no collective on the
data path); rank 0 prints the aggregate.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2607_20214_gb300 import perfmodel  # noqa: E402
from paper_2607_20214_gb300.workloads import (WORKLOADS,  # noqa: E402
                                              make_gate_mlp, make_inputs)

METRIC = "ELSAA fwd tokens/s at N=16K bf16 on 1 GB300"
METRIC_BWD = "ELSAA bwd tokens/s (dQ, dK, dV fp32) on 1 GB300"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0,
                  "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def load_peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        d["source"] = "measured"
        return d
    except OSError:
        return dict(FALLBACK_PEAKS)


class ClockSampler:
    """nvidia-smi clocks / throttle reasons, sampled every 50 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,"
              "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.samples = []
        self.proc = None
        self.device_index = device_index

    def start(self):
        cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS,
               "--format=csv,noheader,nounits", "-lms", "50"]
        uuid = None
        try:
            uuid = str(torch.cuda.get_device_properties(
                self.device_index).uuid)
        except Exception:
            pass
        if uuid:
            cmd += ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        threading.Thread(target=self._read, daemon=True).start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float) -> dict:
        rows = []
        for t, line in self.samples:
            if t0 <= t <= t1:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [],
                    "samples": 0}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        for r in rows:
            for name, val in zip(names, r[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(rows)}


def dist_setup(gpus: int):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def ncu_traffic(kernel: str, workload: str):
    """Per-launch DRAM bytes from the committed ncu summary, if the kernel
    source is unchanged since the counters were taken."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        with open(path) as f:
            table = json.load(f)
    except OSError:
        return None
    ent = table.get("%s@%s" % (kernel, workload))
    if not ent or ent.get("workload") != workload:
        return None
    src = os.path.join(ROOT, ent["source"])
    try:
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    except OSError:
        return None
    if sha != ent.get("source_sha"):
        return None
    return ent.get("traffic_bytes_per_launch")


def cpu_oracle_time(wl, x_cpu, heads, threads):
    from oracle import oracle
    p = oracle.params_from_workload(wl)
    t0 = time.perf_counter()
    if wl.causal:
        # numpy fp64 (one head after another; its BLAS may use every core)
        from oracle import causal
        res = causal.forward(x_cpu, p, heads=heads)
    else:
        res = oracle.forward(x_cpu, p, heads=heads, threads=threads)
    return time.perf_counter() - t0, res


def heads_to_cpu(x, heads):
    """CPU copies of the listed (b, h) heads as a [1, n, N, d] batch."""
    out = {}
    for key in ("q", "k", "v"):
        out[key] = torch.stack([x[key][b, h] for b, h in heads])[None].cpu()
    out["w_sort"] = torch.stack([x["w_sort"][h] for _, h in heads]).cpu()
    out["w_race"] = torch.stack([x["w_race"][h] for _, h in heads]).cpu()
    return out


def run_reference(args, wl):
    """The CPU oracle as the reference arm: each step one bounded sample."""
    world, rank, _ = dist_setup(args.gpus)
    if rank != 0:
        return 0
    from oracle import oracle
    oracle.build()
    cores = os.cpu_count() or 1
    # the causal oracle runs one head at a time (numpy, about 3 s per c3
    # causal head): two heads per step
    per_step = 2 if wl.causal else max(1, min(wl.heads, cores))
    x = make_inputs(wl.with_(B=1, H=min(wl.H, per_step)))
    heads = [(0, h) for h in range(min(wl.H, per_step))]
    times = []
    for i in range(args.warmup + args.steps):
        t, _ = cpu_oracle_time(wl, x, heads, threads=per_step)
        if i >= args.warmup:
            times.append(t)
    t_step = statistics.mean(times)
    # the sample covers len(heads) of the workload's B*H heads
    value = wl.tokens * (len(heads) / wl.heads) / t_step
    sample = "%d of %d heads (N=%d, d_h=%d) per step, %d threads" % (
        len(heads), wl.heads, wl.N, wl.d_h, per_step)
    line = {
        "impl": "reference", "metric": METRIC, "value": value,
        "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_step * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic",
        "config": workload_config(wl),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def workload_config(wl):
    return {"workload": "%s: B=%d H=%d N=%d d_h=%d %s b=%d r=%d "
                        "(L_s=%d, gamma=%d) sort_bits=%d %s%s" % (
                            wl.name, wl.B, wl.H, wl.N, wl.d_h, wl.dtype,
                            wl.block, wl.r, wl.race_tables, wl.race_bits,
                            wl.sort_bits,
                            ("causal (C=%d, N_0=%d)" % (
                                wl.causal_chunk, wl.causal_base_len))
                            if wl.causal else "non-causal",
                            ((", %d neighbour blocks per side" %
                              wl.neighbor_blocks) if wl.neighbor_blocks
                             else "") +
                            ((", top-k selector: k=%d over %d candidate "
                              "blocks" % (wl.topk, wl.topk_blocks))
                             if wl.selector else "")),
            "B": wl.B, "H": wl.H, "N": wl.N, "d_h": wl.d_h,
            "block": wl.block, "r": wl.r, "global_batch": wl.B,
            "seq_len": wl.N,
            "l2": "no flush: Q+K+V = %.0f MB per step > 129 MB L2" % (
                3 * wl.heads * wl.N * wl.d_h * wl.elt / 1e6)}


def measure(step, steps, warmup, dev, stream):
    """Mean device milliseconds of one step over `steps` timed steps (CUDA
    events on the launching stream, after `warmup` untimed steps) and the
    library's per-kernel event times over the same region."""
    from paper_2607_20214_gb300 import elsaa
    for _ in range(warmup):
        step()
    torch.cuda.synchronize(dev)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    elsaa.elsaa_profile_start()
    ev0.record(stream)
    for _ in range(steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    prof = elsaa.elsaa_profile_stop()
    return ev0.elapsed_time(ev1) / steps, prof


def dominant_roofline(wl, prof, peaks, ms_step, steps):
    """Roofline of the kernel with the largest share of the device time."""
    dom = max(prof, key=lambda k: prof[k][1])
    n_dom, ms_dom = prof[dom]
    work = perfmodel.kernel_work(wl, dom)
    roof = perfmodel.roofline(work, ms_dom / n_dom / 1e3, peaks)
    roof["kernel"] = dom
    roof["share_of_step"] = ms_dom / steps / ms_step
    roof["peak_source"] = peaks.get("source", "measured")
    roof["traffic"] = ncu_traffic(dom, wl.name)
    roof["algorithmic"] = work["bytes"] if roof["bound"] == "hbm" else \
        work["flops"]
    return roof


def output_errors(got, ref):
    """max-abs, relative l2 (||got - ref|| / ||ref||) and max-abs over
    max |ref| of arrays of the same shape."""
    import numpy as np
    d = got - ref
    return {"max_abs": float(np.abs(d).max()),
            "rel_l2": float(np.linalg.norm(d) / np.linalg.norm(ref)),
            "max_abs_over_max_ref": float(np.abs(d).max() /
                                          np.abs(ref).max())}


def forward_errors(wl, x, o, heads, rows=None):
    """The oracle on the listed heads (rows: a sample of query rows, None =
    all) against the device output o; the errors over all of them."""
    import numpy as np
    from oracle import oracle as orc
    xc = heads_to_cpu(x, heads)
    res = orc.forward(xc, orc.params_from_workload(wl),
                      heads=[(0, j) for j in range(len(heads))], rows=rows,
                      threads=len(heads))
    got, ref = [], []
    for j, (b, h) in enumerate(heads):
        r = res[(0, j)]
        got.append(o[b, h].float().cpu().numpy()[r["rows"]])
        ref.append(r["O"])
    return output_errors(np.concatenate(got), np.concatenate(ref))


def extra_workloads(args, dev, stream, peaks):
    """The long-context forward (c4: B=1 H=32 N=65536 d_h=128, b=256,
    r=256) and the training step (c5: forward + backward, B=8 H=12 N=8192
    d_h=64, b=64, r=128), timed in the same run as the headline workload,
    each with its dominant kernel's roofline, the step's roofline fraction
    and errors against the oracle on sampled heads and rows."""
    import numpy as np
    from oracle import backward as obwd
    from oracle import oracle as orc
    from paper_2607_20214_gb300 import elsaa
    out = {}
    # -- c4: forward
    wl = WORKLOADS["c4"]
    x = make_inputs(wl, device=dev)
    p = elsaa.params_for(wl)
    ws = elsaa.new_workspace(p, dev)
    o = torch.empty_like(x["q"])

    def step():
        elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"],
                            x["w_race"], o=o, workspace=ws, stream=stream)

    ms, prof = measure(step, args.steps, args.warmup, dev, stream)
    elsaa.elsaa_check_status(ws)
    fm = perfmodel.flop_model(wl)
    rows = np.random.default_rng(4).choice(wl.N, 512, replace=False)
    rows.sort()
    out["c4"] = {
        "config": workload_config(wl), "ms_per_step": ms,
        "value": wl.tokens / (ms / 1e3), "unit": "tokens/s",
        "tflops": fm["tensor_flops"] / (ms / 1e3) / 1e12,
        "step_roofline_frac": max(
            fm["tensor_flops"] / (peaks["bf16_tflops"] * 1e12),
            fm["bytes"] / (peaks["hbm_gbs"] * 1e9)) / (ms / 1e3),
        "roofline": dominant_roofline(wl, prof, peaks, ms, args.steps),
        "kernels": {k: {"launches": n, "avg_us": 1e3 * t / n}
                    for k, (n, t) in sorted(prof.items())},
        "gpu_launches": sum(n for n, _ in prof.values()),
        "err_vs_oracle": dict(forward_errors(wl, x, o, [(0, 0), (0, 31)],
                                             rows=rows),
                              sample="512 rows of heads (0, 0), (0, 31)"),
    }
    del x, o, ws
    # -- c3 with the per-query top-k selector (k = 128 over two candidate
    # blocks per query block)
    wl = WORKLOADS["c3"].with_(selector=1, topk=128, topk_blocks=2)
    x = make_inputs(wl, device=dev)
    p = elsaa.params_for(wl)
    ws = elsaa.new_workspace(p, dev)
    o = torch.empty_like(x["q"])

    def step():
        elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"],
                            x["w_race"], o=o, workspace=ws, stream=stream)

    ms, prof = measure(step, args.steps, args.warmup, dev, stream)
    elsaa.elsaa_check_status(ws)
    fm = perfmodel.flop_model(wl)
    rows = np.random.default_rng(6).choice(wl.N, 256, replace=False)
    rows.sort()
    out["c3_topk"] = {
        "config": workload_config(wl), "ms_per_step": ms,
        "value": wl.tokens / (ms / 1e3), "unit": "tokens/s",
        "step_roofline_frac": max(
            fm["tensor_flops"] / (peaks["bf16_tflops"] * 1e12),
            fm["bytes"] / (peaks["hbm_gbs"] * 1e9)) / (ms / 1e3),
        "roofline": dominant_roofline(wl, prof, peaks, ms, args.steps),
        "kernels": {k: {"launches": n, "avg_us": 1e3 * t / n}
                    for k, (n, t) in sorted(prof.items())},
        "gpu_launches": sum(n for n, _ in prof.values()),
        "err_vs_oracle": dict(forward_errors(wl, x, o, [(1, 7)], rows=rows),
                              sample="256 rows of head (1, 7)"),
    }
    del x, o, ws
    # -- c3 with learned gates and query-dependent lambda (hidden width 64)
    # computed inside the forward call
    wl = WORKLOADS["c3"]
    x = make_inputs(wl, device=dev)
    p = elsaa.params_for(wl)
    mlp = make_gate_mlp(wl, hidden=64, device=dev)
    ws = torch.empty(max(elsaa.elsaa_forward_gated_workspace_size(p, mlp),
                         256), dtype=torch.uint8, device=dev)
    o = torch.empty_like(x["q"])

    def step():
        elsaa.elsaa_forward_gated(p, mlp, x["q"], x["k"], x["v"],
                                  x["w_sort"], x["w_race"], o=o,
                                  workspace=ws, stream=stream)

    ms, prof = measure(step, args.steps, args.warmup, dev, stream)
    elsaa.elsaa_check_status(ws)
    out["c3_gated"] = {
        "config": dict(workload_config(wl), gate_mlp_hidden=64),
        "step": "elsaa_forward_gated: gate MLP (hidden 64) and lambda_i in "
                "the same call",
        "ms_per_step": ms, "value": wl.tokens / (ms / 1e3),
        "unit": "tokens/s",
        "kernels": {k: {"launches": n, "avg_us": 1e3 * t / n}
                    for k, (n, t) in sorted(prof.items())},
        "gpu_launches": sum(n for n, _ in prof.values()),
    }
    del x, o, ws
    # -- c5: training step, forward + backward
    wl = WORKLOADS["c5"]
    x = make_inputs(wl.with_(backward=True), device=dev)
    p = elsaa.params_for(wl)
    ws = elsaa.new_workspace(p, dev)
    wsb = torch.empty(max(elsaa.elsaa_backward_workspace_size(p), 256),
                      dtype=torch.uint8, device=dev)
    BHN = (wl.B, wl.H, wl.N)
    o = torch.empty_like(x["q"])
    pq = torch.empty(BHN, dtype=torch.int32, device=dev)
    pk = torch.empty(BHN, dtype=torch.int32, device=dev)
    r = wl.r
    rA = torch.empty((wl.B, wl.H, r), dtype=torch.float32, device=dev)
    rB = torch.empty((wl.B, wl.H, r, wl.d_h), dtype=torch.float32,
                     device=dev)
    grads = [torch.empty(x["q"].shape, dtype=torch.float32, device=dev)
             for _ in range(3)]

    def step():
        elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"],
                            x["w_race"], o=o, perm_q=pq, perm_k=pk,
                            workspace=ws, stream=stream)
        elsaa.elsaa_forward_race_summaries(p, ws, rA, rB, stream=stream)
        elsaa.elsaa_backward(p, x["q"], x["k"], x["v"], x["w_sort"],
                             x["w_race"], x["do"], pq, pk, dq=grads[0],
                             dk=grads[1], dv=grads[2], race_A=rA, race_B=rB,
                             workspace=wsb, stream=stream)

    ms, prof = measure(step, args.steps, args.warmup, dev, stream)
    elsaa.elsaa_check_status(ws)
    elsaa.elsaa_check_status(wsb)
    ff = perfmodel.flop_model(wl)
    fb = perfmodel.backward_flop_model(wl)
    flops = ff["tensor_flops"] + fb["tensor_flops"]
    nbytes = ff["bytes"] + fb["bytes"]
    rows = np.random.default_rng(5).choice(wl.N, 512, replace=False)
    rows.sort()
    fwd_err = forward_errors(wl, x, o, [(0, 0), (wl.B - 1, wl.H - 1)],
                             rows=rows)
    # the oracle's fp64 analytic gradient of one whole head
    b, h = wl.B - 1, wl.H - 1
    f32 = lambda t: t[b, h].float().cpu().numpy()  # noqa: E731
    t0 = time.perf_counter()
    ref = obwd.backward_head(
        f32(x["q"]), f32(x["k"]), f32(x["v"]),
        x["w_sort"][h].float().cpu().numpy(),
        x["w_race"][h].double().cpu().numpy(), f32(x["do"]),
        orc.params_from_workload(wl), lam=np.full(wl.N, wl.lam))
    t_cpu = time.perf_counter() - t0
    grad_err = {}
    for name, g in zip(("dQ", "dK", "dV"), grads):
        grad_err[name] = output_errors(g[b, h].cpu().numpy(), ref[name])
    out["c5_train"] = {
        "config": workload_config(wl),
        "step": "elsaa_forward (perms saved) + RACE summaries saved + "
                "elsaa_backward (dQ, dK, dV fp32)",
        "ms_per_step": ms, "value": wl.tokens / (ms / 1e3),
        "unit": "tokens/s", "tflops": flops / (ms / 1e3) / 1e12,
        "step_roofline_frac": max(
            flops / (peaks["bf16_tflops"] * 1e12),
            nbytes / (peaks["hbm_gbs"] * 1e9)) / (ms / 1e3),
        "roofline": dominant_roofline(wl, prof, peaks, ms, args.steps),
        "kernels": {k: {"launches": n, "avg_us": 1e3 * t / n}
                    for k, (n, t) in sorted(prof.items())},
        "gpu_launches": sum(n for n, _ in prof.values()),
        "fwd_err_vs_oracle": dict(fwd_err, sample="512 rows of two heads"),
        "grad_err_vs_oracle": dict(grad_err, sample=(
            "head (%d, %d), every row; fp64 analytic gradient, %.1f s on "
            "one host thread" % (b, h, t_cpu))),
    }
    return out


def run_ours(args, wl):
    from paper_2607_20214_gb300 import build as nvbuild
    from paper_2607_20214_gb300 import elsaa
    from paper_2607_20214_gb300 import multirank

    world, rank, local = dist_setup(args.gpus)
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    nvbuild.build()
    elsaa.load_library()
    peaks = load_peaks()

    wl_rank = multirank.rank_workload(wl, rank)
    if args.backward:
        wl_rank = wl_rank.with_(backward=True)
    x = make_inputs(wl_rank, device=dev)
    p = elsaa.params_for(wl)
    ws = elsaa.new_workspace(p, dev)
    o = torch.empty_like(x["q"])
    stream = torch.cuda.current_stream(dev)

    def step():
        elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"],
                            x["w_race"], o=o, workspace=ws, stream=stream)

    if args.gate_mlp:
        # learned gates and query-dependent lambda feeding the fusion, in
        # the same call (elsaa_forward_gated: inside the sort hash where the
        # shape allows, else the gate kernel first)
        mlp = make_gate_mlp(wl_rank, hidden=args.gate_mlp, device=dev)
        ws = torch.empty(
            max(elsaa.elsaa_forward_gated_workspace_size(p, mlp), 256),
            dtype=torch.uint8, device=dev)

        def step():
            elsaa.elsaa_forward_gated(p, mlp, x["q"], x["k"], x["v"],
                                      x["w_sort"], x["w_race"], o=o,
                                      workspace=ws, stream=stream)

    if args.backward:
        # the backward pass of the same inputs: permutations and the RACE
        # summaries A, B saved from one forward (outside the timed region,
        # as a training step keeps them), then elsaa_backward per step
        BHN = (wl.B, wl.H, wl.N)
        perm_q = torch.empty(BHN, dtype=torch.int32, device=dev)
        perm_k = torch.empty(BHN, dtype=torch.int32, device=dev)
        elsaa.elsaa_forward(p, x["q"], x["k"], x["v"], x["w_sort"],
                            x["w_race"], o=o, perm_q=perm_q, perm_k=perm_k,
                            workspace=ws, stream=stream)
        race_A, race_B = elsaa.elsaa_forward_race_summaries(p, ws,
                                                            stream=stream)
        wsb = torch.empty(max(elsaa.elsaa_backward_workspace_size(p), 256),
                          dtype=torch.uint8, device=dev)
        grads = [torch.empty(x["q"].shape, dtype=torch.float32, device=dev)
                 for _ in range(3)]

        def step():
            elsaa.elsaa_backward(p, x["q"], x["k"], x["v"], x["w_sort"],
                                 x["w_race"], x["do"], perm_q, perm_k,
                                 dq=grads[0], dk=grads[1], dv=grads[2],
                                 race_A=race_A, race_B=race_B,
                                 workspace=wsb, stream=stream)

    barrier = multirank.barrier

    sampler = ClockSampler(local)
    sampler.start()
    for _ in range(args.warmup):
        step()
    elsaa.elsaa_check_status(ws)
    # time-based pre-roll so the clock record covers a loaded GPU
    t_pre = time.time()
    while not args.no_preroll and time.time() - t_pre < 1.0:
        step()
        torch.cuda.synchronize(dev)
    torch.cuda.synchronize(dev)
    barrier()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    elsaa.elsaa_profile_start()
    ev0.record(stream)
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    t_end = time.time()
    barrier()
    prof = elsaa.elsaa_profile_stop()
    ms = ev0.elapsed_time(ev1)
    elsaa.elsaa_check_status(wsb if args.backward else ws)
    sampler.stop()
    clocks = sampler.summary(t_pre, t_end)
    ms = multirank.max_over_ranks(ms, dev)
    ms_step = ms / args.steps
    value = multirank.job_throughput(world, wl.tokens, ms_step)

    # dominant kernel roofline (device time of each launch, CUDA events on
    # the launching stream over the timed region)
    launches = sum(n for n, _ in prof.values())
    dom = max(prof, key=lambda k: prof[k][1])
    n_dom, ms_dom = prof[dom]
    work = perfmodel.kernel_work(wl, dom)
    roof = perfmodel.roofline(work, ms_dom / n_dom / 1e3, peaks)
    roof["kernel"] = dom
    # the dominant kernel's device time against the step's wall time (the
    # RACE key side overlaps the sort chain, so summed kernel times exceed
    # the step)
    roof["share_of_step"] = ms_dom / args.steps / ms_step
    roof["peak_source"] = peaks.get("source", "measured")
    roof["traffic"] = ncu_traffic(dom, wl.name)
    roof["algorithmic"] = work["bytes"] if roof["bound"] == "hbm" else \
        work["flops"]
    kernels = {k: {"launches": n, "avg_us": 1e3 * t / n}
               for k, (n, t) in sorted(prof.items())}

    fm = perfmodel.flop_model(wl)
    t_s = ms_step / 1e3
    step_roof = max(fm["tensor_flops"] / (peaks["bf16_tflops"] * 1e12),
                    fm["bytes"] / (peaks["hbm_gbs"] * 1e9)) / t_s

    # end to end through the public API: pinned host inputs -> device ->
    # forward -> host output, every step
    e2e = None
    if args.backward and not args.no_e2e:
        names = ("q", "k", "v", "w_race", "do")
        hx = {k: x[k].cpu().pin_memory() for k in names}
        hp = [perm_q.cpu().pin_memory(), perm_k.cpu().pin_memory(),
              race_A.cpu().pin_memory(), race_B.cpu().pin_memory()]
        dx = {k: torch.empty_like(x[k]) for k in hx}
        dp = [torch.empty_like(perm_q), torch.empty_like(perm_k),
              torch.empty_like(race_A), torch.empty_like(race_B)]
        hg = [torch.empty(g.shape, dtype=g.dtype).pin_memory() for g in grads]
        h2d = sum(t.numel() * t.element_size() for t in hx.values()) + sum(
            t.numel() * t.element_size() for t in hp)
        d2h = sum(t.numel() * t.element_size() for t in hg)

        def e2e_step():
            for k in hx:
                dx[k].copy_(hx[k], non_blocking=True)
            for dd, hh in zip(dp, hp):
                dd.copy_(hh, non_blocking=True)
            elsaa.elsaa_backward(p, dx["q"], dx["k"], dx["v"], None,
                                 dx["w_race"], dx["do"], dp[0], dp[1],
                                 dq=grads[0], dk=grads[1], dv=grads[2],
                                 race_A=dp[2], race_B=dp[3],
                                 workspace=wsb, stream=stream)
            for hh, g in zip(hg, grads):
                hh.copy_(g, non_blocking=True)

        for _ in range(max(3, args.warmup)):
            e2e_step()
        torch.cuda.synchronize(dev)
        a = torch.cuda.Event(enable_timing=True)
        bq = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(args.steps):
            e2e_step()
        bq.record(stream)
        torch.cuda.synchronize(dev)
        ms_e2e = a.elapsed_time(bq) / args.steps
        e2e = {"value": world * wl.tokens / (ms_e2e / 1e3),
               "unit": "tokens/s", "ms_per_step": ms_e2e,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}
    if not args.no_e2e and not args.backward and not args.gate_mlp:
        # every step copies its own inputs from pinned host memory, runs
        # elsaa_forward and copies its output back; copy-in, compute and
        # copy-out run on three streams with two device buffer sets, so the
        # copies of neighbouring steps overlap a step's compute (a streaming
        # deployment's pipeline)
        names = ("q", "k", "v", "w_sort", "w_race")
        hx = {k: x[k].cpu().pin_memory() for k in names}
        sets = [({k: torch.empty_like(x[k]) for k in names},
                 torch.empty_like(o)) for _ in range(2)]
        hos = [torch.empty(o.shape, dtype=o.dtype).pin_memory()
               for _ in range(2)]
        h2d = sum(t.numel() * t.element_size() for t in hx.values())
        d2h = hos[0].numel() * hos[0].element_size()
        s_in, s_cmp, s_out = (torch.cuda.Stream(dev) for _ in range(3))
        ev_in = [torch.cuda.Event() for _ in range(2)]
        ev_done = [torch.cuda.Event() for _ in range(2)]
        ev_out = [torch.cuda.Event() for _ in range(2)]

        def e2e_step(kk):
            j = kk % 2
            dx, do_ = sets[j]
            if kk >= 2:  # set j's inputs were read by step kk - 2
                s_in.wait_event(ev_done[j])
            with torch.cuda.stream(s_in):
                for k in names:
                    dx[k].copy_(hx[k], non_blocking=True)
                ev_in[j].record(s_in)
            s_cmp.wait_event(ev_in[j])
            if kk >= 2:  # set j's output was copied out by step kk - 2
                s_cmp.wait_event(ev_out[j])
            elsaa.elsaa_forward(p, dx["q"], dx["k"], dx["v"], dx["w_sort"],
                                dx["w_race"], o=do_, workspace=ws,
                                stream=s_cmp)
            ev_done[j].record(s_cmp)
            s_out.wait_event(ev_done[j])
            with torch.cuda.stream(s_out):
                hos[j].copy_(do_, non_blocking=True)
                ev_out[j].record(s_out)

        for kk in range(max(3, args.warmup)):
            e2e_step(kk)
        torch.cuda.synchronize(dev)
        barrier()
        a = torch.cuda.Event(enable_timing=True)
        bq = torch.cuda.Event(enable_timing=True)
        a.record(s_in)
        for kk in range(args.steps):
            e2e_step(kk)
        bq.record(s_out)
        torch.cuda.synchronize(dev)
        barrier()
        ms_e2e = multirank.max_over_ranks(a.elapsed_time(bq) / args.steps,
                                          dev)
        e2e = {"value": multirank.job_throughput(world, wl.tokens, ms_e2e),
               "unit": "tokens/s", "ms_per_step": ms_e2e,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "pipeline": "copy-in, compute and copy-out on three streams "
                           "with two device buffer sets"}

    # CPU oracle on the host cores (rank 0, N = 1): one whole step when it
    # fits in the sample budget, also used as a parity spot check
    cpu = None
    err = None
    errs = None
    if args.backward and rank == 0 and world == 1 and \
            not args.no_cpu_baseline:
        # the oracle's fp64 gradient of whole heads on one host core, also a
        # parity spot check (relative to the largest reference gradient)
        import numpy as np
        from oracle import backward as obwd
        from oracle import oracle as orc
        po = orc.params_from_workload(wl)
        heads = [(0, 0), (wl.B - 1, wl.H - 1)]
        t0 = time.perf_counter()
        err = 0.0
        for (b, h) in heads:
            f32 = lambda t: t[b, h].float().cpu().numpy()
            r = obwd.backward_head(
                f32(x["q"]), f32(x["k"]), f32(x["v"]),
                x["w_sort"][h].float().cpu().numpy(),
                x["w_race"][h].double().cpu().numpy(), f32(x["do"]), po,
                lam=np.full(wl.N, wl.lam))
            for name, g in zip(("dQ", "dK", "dV"), grads):
                ref = r[name]
                err = max(err, float(np.abs(g[b, h].cpu().numpy() - ref).max()
                                     / np.abs(ref).max()))
        t_cpu = time.perf_counter() - t0
        cpu = {"value": wl.N * len(heads) / t_cpu, "unit": "tokens/s",
               "cores": 1, "kind": "oracle",
               "sample": "%d of %d heads (fp64 numpy gradient, one thread), "
                         "%.1f s wall" % (len(heads), wl.heads, t_cpu)}
    if rank == 0 and world == 1 and not args.no_cpu_baseline and \
            not args.backward and not args.gate_mlp:
        cores = os.cpu_count() or 1
        n_heads = 2 if wl.causal else min(wl.heads, 2 * cores)
        heads = [(i // wl.H, i % wl.H) for i in range(n_heads)]
        xc = heads_to_cpu(x, heads)
        t_cpu, res = cpu_oracle_time(wl, xc, [(0, j) for j in range(n_heads)],
                                     threads=min(cores, n_heads))
        cpu = {"value": wl.tokens * (n_heads / wl.heads) / t_cpu,
               "unit": "tokens/s",
               "cores": cores if wl.causal else min(cores, n_heads),
               "kind": "oracle",
               "sample": ("%d of %d heads of one step (fp64 numpy causal "
                          "oracle, one head at a time, BLAS threads up to "
                          "%d cores), %.1f s wall" % (n_heads, wl.heads,
                                                      cores, t_cpu))
               if wl.causal else
               "%d of %d heads of one step (fp64 C oracle, "
               "threads over heads), %.1f s wall" % (
                   n_heads, wl.heads, t_cpu)}
        import numpy as np
        of = o.float()
        errs = output_errors(
            np.concatenate([of[b, h].cpu().numpy()
                            for b, h in heads]),
            np.concatenate([res[(0, j)]["O"] for j in range(len(heads))]))
        err = errs["max_abs"]

    extra = None
    if rank == 0 and world == 1 and not args.no_extra and \
            args.workload == "c3" and not (args.backward or args.gate_mlp or
                                           args.batch or args.heads or
                                           args.neighbors or args.topk):
        extra = extra_workloads(args, dev, stream, peaks)

    if rank != 0:
        return 0
    line = {
        "metric": METRIC_BWD if args.backward else METRIC, "value": value,
        "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": dict(workload_config(wl),
                       **({"gate_mlp_hidden": args.gate_mlp}
                          if args.gate_mlp else {})),
        "tflops": fm["tensor_flops"] / t_s / 1e12,
        "step_roofline_frac": step_roof,
        "roofline": roof, "kernels": kernels,
        "gpu_launches": launches,
        "clocks": clocks,
        "e2e": e2e,
        "cpu_baseline": cpu,
        ("max_rel_grad_err_vs_oracle" if args.backward else
         "max_abs_err_vs_oracle"): err,
    }
    if errs is not None:
        line["rel_l2_err_vs_oracle"] = errs["rel_l2"]
        line["max_abs_over_max_ref_vs_oracle"] = errs["max_abs_over_max_ref"]
    if extra is not None:
        line["extra_workloads"] = extra
    print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="c3", choices=sorted(WORKLOADS))
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the c4 forward and c5 training-step lines "
                         "that the default c3 run adds")
    ap.add_argument("--batch", type=int, default=0,
                    help="override B (smaller cases for profiler captures)")
    ap.add_argument("--neighbors", type=int, default=0, metavar="R",
                    help="R neighbouring sorted key blocks per side "
                         "(sparse branch on CUDA cores when R > 0)")
    ap.add_argument("--topk", type=int, default=0, metavar="K",
                    help="per-query top-k selector with K keys per query "
                         "(default: the sorted-block selector)")
    ap.add_argument("--topk-blocks", type=int, default=2, metavar="C",
                    help="candidate key blocks per query block for --topk")
    ap.add_argument("--heads", type=int, default=0,
                    help="override H (smaller cases for profiler captures)")
    ap.add_argument("--no-preroll", action="store_true",
                    help="skip the 1 s loaded pre-roll (profiler captures)")
    ap.add_argument("--gate-mlp", type=int, default=0, metavar="HIDDEN",
                    help="also run the gate MLP / lambda kernel (hidden "
                         "width HIDDEN, e.g. 64) in every step; its gates "
                         "and lambda feed the fusion")
    ap.add_argument("--backward", action="store_true",
                    help="time elsaa_backward (dQ, dK, dV) instead of the "
                         "forward; use with --workload c5")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    wl = WORKLOADS[args.workload]
    if args.batch:
        wl = wl.with_(B=args.batch)
    if args.heads:
        wl = wl.with_(H=args.heads)
    if args.neighbors:
        wl = wl.with_(neighbor_blocks=args.neighbors)
    if args.topk:
        wl = wl.with_(selector=1, topk=args.topk,
                      topk_blocks=args.topk_blocks)
    if args.impl == "reference":
        return run_reference(args, wl)
    return run_ours(args, wl)


if __name__ == "__main__":
    sys.exit(main())
