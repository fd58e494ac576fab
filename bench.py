"""Benchmark of the PolyQ mixed-bit linear layer on GB300.

Default workload (one step): the seven decode linears of a Llama2-13B-shaped
layer (q, k, v, o 5120x5120; gate, up 13824x5120; down 5120x13824), batch 1,
average budget 3.0 bits, synthetic seeded weights and activations.  Each step
runs the seven GEMVs through the library; the weights rotate over several
device copies of the layer so that no step finds its weights in L2.

Output: one JSON line (rank 0).  ``value`` is whole-job packed-layer bytes
moved per second (TB/s) with inputs resident in HBM; ``e2e`` is the same
metric through the public API with host<->device copies of each step's
activations and results inside the timed region.

``--impl reference`` times the CPU oracle on the host cores instead (a
bounded sample of the same workload per step).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

# The oracle's fp64 product goes through BLAS, which would use every host core
# unless told otherwise: the reference arm and the one-thread CPU baseline pin
# it to one thread before numpy loads (the driver's own setting wins).
if "--cpu-baseline-child" in sys.argv or ("--impl" in sys.argv and "reference" in sys.argv):
    for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        os.environ.setdefault(_v, "1")

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "mixed-bit GEMV HBM TB/s (% of peak) at 3.0b avg; prefill GEMM TFLOPS (% peak)"
LLAMA = [("q", 5120, 5120), ("k", 5120, 5120), ("v", 5120, 5120), ("o", 5120, 5120),
         ("gate", 13824, 5120), ("up", 13824, 5120), ("down", 5120, 13824)]
WORKLOAD = ("llama2-13b decode linears q,k,v,o 5120x5120, gate,up 13824x5120, "
            "down 5120x13824; batch 1; B=3.0")
# launches of one decoder layer: q/k/v and gate/up read the same input
GROUPS = [(0, 1, 2), (3,), (4, 5), (6,)]
# DRAM bytes (read + write) of one step's eight GEMV launches, summed from the
# ncu launch list in profiles/gemv_decode_llama13b_b3_launches.md, with the
# SHA-1 of the kernel sources it was taken on; reported as null once those
# sources change.
TRAFFIC = {"bytes_per_step": 143122432,
           "sources_sha1": "65e281d00aa988c0e29db934964992dba7e2f900",
           "profile": "profiles/gemv_decode_llama13b_b3_launches.md"}
GEMV_SOURCES = ("polyq_gemv.cu", "polyq_gemv_dev.cuh", "polyq_gemv_layout.cuh", "polyq_dev.cuh")
REF_SECONDS = 120.0  # the reference arm's warm-up and timed steps together


def _gemv_sources_sha1():
    import hashlib
    h = hashlib.sha1()
    for f in GEMV_SOURCES:
        with open(os.path.join(ROOT, "paper_2607_14618_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    with open(os.path.join(ROOT, "include", "polyq.h"), "rb") as fh:  # launch parameter layout
        h.update(fh.read())
    return h.hexdigest()


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), d.get("bf16_tflops", 1900.0), \
            d.get("bf16_tflops_sustained", 1700.0), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi samples (200 ms) taken while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.p = None

    def __enter__(self):
        try:
            self.p = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.p = None
        return self

    def __exit__(self, *a):
        self.rows = []
        if self.p is None:
            return
        self.p.terminate()
        try:
            out, _ = self.p.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
            out, _ = self.p.communicate()
        for line in out.splitlines():
            f = [c.strip() for c in line.split(",")]
            if len(f) >= 9:
                self.rows.append(f)

    def summary(self):
        if not getattr(self, "rows", None):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in self.rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in self.rows for i in range(4)
                          if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(self.rows)}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(ms, ws, device=None):
    """The job's time: the slowest replica's (one all-reduce over the ranks'
    timings; ``device`` is where the process group's backend wants the
    tensor, a GPU for NCCL, the CPU for gloo)."""
    if ws <= 1:
        return float(ms)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def window_max_over_ranks(win_ms, ws, device=None):
    """Per window, the slowest rank's duration (all ranks time the same
    number of windows)."""
    if ws == 1:
        return list(win_ms)
    import torch
    import torch.distributed as dist
    t = torch.tensor(win_ms, dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.cpu().tolist()


def job_tbs(ws, step_bytes, steps, ms):
    """Whole-job throughput: every replica streams ``step_bytes`` per step,
    over the slowest replica's time."""
    return ws * step_bytes * steps / (ms * 1e-3) / 1e12


def build_layers(polyq, synth, budget, copies, device):
    """Pack the seven linears once (seeded), upload, and clone on device.
    Linears of one launch group share their input activation."""
    layers, xs = [], [None] * len(LLAMA)
    hosts = []
    for i, (name, N, K) in enumerate(LLAMA):
        W, a = synth.layer_weights(N, K, synth.seed_for(2, i))
        host = polyq.HostLayer.pack(W, a, budget)
        dev = polyq.DeviceLayer(host, device)
        hosts.append((name, host.info()))
        layers.append([dev] + [dev.clone() for _ in range(copies - 1)])
        for grp in GROUPS:
            if grp[0] == i:
                xb, _ = synth.activations(a, 1, synth.seed_for(2, i))
                for k in grp:
                    xs[k] = xb
        del W
    return layers, xs, hosts


def layer_bytes(info, batch):
    """Algorithmic bytes of one GEMV launch: packed codes (incl. segment
    padding) + scale/zero metadata + gathered activations + gather indices +
    outputs."""
    return (info["packed_bytes"] + info["meta_bytes"] + batch * info["K"] * 2
            + info["K"] * 4 + batch * info["N"] * 4)


def run_polyq(args):
    import torch
    import torch.distributed as dist

    ws, rank, local = _dist()
    if ws > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    from paper_2607_14618_gb300 import build as _b
    if rank == 0:
        _b.build_library()
    if ws > 1:
        dist.barrier()
    from paper_2607_14618_gb300 import polyq, synth

    hbm, tf_burst, tf_sus, peak_kind = _peaks()
    batch = args.batch
    layers, xs_np, infos = build_layers(polyq, synth, args.budget, args.copies, device)
    L2 = torch.cuda.get_device_properties(device).L2_cache_size
    n_lin = len(LLAMA)
    per_lin_bytes = [layer_bytes(inf, batch) for _, inf in infos]
    step_bytes = sum(per_lin_bytes)
    copy_bytes = sum(inf["packed_bytes"] + inf["meta_bytes"] for _, inf in infos)
    xs = [torch.from_numpy(np.repeat(x, batch, 0).view(np.int16)).to(device).view(torch.bfloat16)
          for x in xs_np]
    ys = [torch.empty((batch, N), dtype=torch.float32, device=device) for _, N, _ in LLAMA]
    wsz = max(polyq.gemv_group_workspace_bytes([layers[i][0] for i in grp], batch)
              for grp in GROUPS)
    wbuf = torch.zeros(max(wsz, 256), dtype=torch.uint8, device=device)
    kernels_per_call = polyq.gemv_launches_per_call(layers[0][0], batch)

    def run_step(c):
        for grp in GROUPS:
            polyq.linear_gemv_group([layers[i][c] for i in grp], [xs[i] for i in grp],
                                    ys=[ys[i] for i in grp], workspace=wbuf, stream=stream)

    stream = torch.cuda.Stream(device)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        run_step(0)  # warm the launch path once before capture
    stream.synchronize()
    # Steps run as a decoder stack does: one CUDA graph holds `copies`
    # consecutive steps (each on its own copy of the layer, so the weights
    # stream from HBM every step); a K-step run replays it K // copies times
    # and then a graph of the remaining K % copies steps.
    def step_graph(n):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for c in range(n):
                run_step(c)
        return g

    cycle = step_graph(args.copies)
    rest = {}

    def run_steps(k):
        for _ in range(k // args.copies):
            cycle.replay()
        r = k % args.copies
        if r:
            if r not in rest:
                rest[r] = step_graph(r)
            rest[r].replay()

    # the same seven GEMVs (each on its own input) in one grouped launch per
    # step: the streaming kernel's rate with one launch boundary per step
    one_graph = torch.cuda.CUDAGraph()
    wsz1 = polyq.gemv_group_workspace_bytes([layers[i][0] for i in range(n_lin)], batch)
    wbuf1 = torch.zeros(max(wsz1, 256), dtype=torch.uint8, device=device)
    with torch.cuda.graph(one_graph, stream=stream):
        for c in range(args.copies):
            polyq.linear_gemv_group([layers[i][c] for i in range(n_lin)], xs, ys=ys,
                                    workspace=wbuf1, stream=stream)
    lin_graphs = []  # per linear: one graph of that linear on every copy
    for i in range(n_lin):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for c in range(args.copies):
                polyq.linear_gemv(layers[i][c], xs[i], y=ys[i], workspace=wbuf, stream=stream)
        lin_graphs.append(g)
    torch.cuda.synchronize()

    # graph replays launch on the current stream: make it `stream`
    with torch.cuda.stream(stream):
        run_steps(args.warmup)
        run_steps(args.steps % args.copies)  # captures the remainder graph outside the timing
    torch.cuda.synchronize()
    # The timed unit is a window of exactly `steps` steps between two events
    # on the launching stream, synchronised on both sides.  A window of the
    # default 20 steps lasts about a millisecond, far below the clock
    # sampler's period, so the window is repeated back to back for about
    # 1.5 s; the reported time is the median window (max over ranks).
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(2)]
    with torch.cuda.stream(stream):
        ev[0][0].record(stream)
        run_steps(args.steps)
        ev[0][1].record(stream)
    torch.cuda.synchronize()
    probe_ms = ev[0][0].elapsed_time(ev[0][1])
    n_win = int(min(args.max_windows, max(1, np.ceil(args.timed_seconds * 1e3 / (probe_ms + 0.05)))))
    if ws > 1:
        n_win = int(max_over_ranks(float(n_win), ws, device))
        dist.barrier()
    torch.cuda.synchronize()
    win_ms = []
    with ClockSampler(local) as clk, torch.cuda.stream(stream):
        for w in range(n_win):
            t0, t1 = ev[w % 2]
            t0.record(stream)
            run_steps(args.steps)
            t1.record(stream)
            t1.synchronize()
            win_ms.append(t0.elapsed_time(t1))
    torch.cuda.synchronize()
    if ws > 1:
        dist.barrier()
    win_ms = window_max_over_ranks(win_ms, ws, device)
    ms = statistics.median(win_ms)
    ms_step = ms / args.steps
    value_tbs = job_tbs(ws, step_bytes, args.steps, ms)
    timing = {"windows": n_win, "steps_per_window": args.steps,
              "window_ms_median": round(ms, 5), "window_ms_min": round(min(win_ms), 5),
              "window_ms_max": round(max(win_ms), 5), "first_window_ms": round(win_ms[0], 5),
              "what": "each window: exactly `steps` steps between CUDA events on the launching "
                      "stream, synchronised on both sides; value from the median window"}

    # Roofline of the dominant kernel.  The timed region holds only GEMV
    # launches (pre-pass + streaming kernel per linear), back to back, so its
    # duration per launch is the step time split over the launches.  A
    # per-linear breakdown comes from graphs of one linear on every copy.
    with torch.cuda.stream(stream):
        for _ in range(3):
            one_graph.replay()
        o0 = torch.cuda.Event(enable_timing=True)
        o1 = torch.cuda.Event(enable_timing=True)
        o0.record(stream)
        for _ in range(50):
            one_graph.replay()
        o1.record(stream)
    stream.synchronize()
    one_us = o0.elapsed_time(o1) * 1e3 / (50 * args.copies)
    one_tbs = step_bytes / (one_us * 1e-6) / 1e12
    one_launch = {"us_per_step": round(one_us, 2), "TB/s": round(one_tbs, 4),
                  "frac_of_hbm": round(one_tbs * 1e3 / hbm, 4),
                  "what": "the seven GEMVs of a step, each on its own input, as one "
                          "polyq_linear_gemv_group call (2 kernels) per step"}
    per_lin_us = {}
    reps = 8
    for i in range(n_lin):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            lin_graphs[i].replay()
            e0.record(stream)
            for r in range(reps):
                lin_graphs[i].replay()
            e1.record(stream)
        torch.cuda.synchronize()
        us = 1e3 * e0.elapsed_time(e1) / (reps * args.copies)
        per_lin_us[LLAMA[i][0]] = {"us": round(us, 2),
                                   "GB/s": round(per_lin_bytes[i] / (us * 1e-6) / 1e9, 1)}
    ach = step_bytes / (ms_step * 1e-3) / 1e9
    traffic = (TRAFFIC["bytes_per_step"] if batch == 1 and args.budget == 3.0
               and _gemv_sources_sha1() == TRAFFIC["sources_sha1"] else None)
    roof = {"bound": "hbm", "achieved": round(ach, 1), "peak": hbm, "unit": "GB/s",
            "frac": round(ach / hbm, 4), "traffic": traffic, "peak_kind": peak_kind,
            "kernel": "gemv_main (+ gemv_prep) of polyq_linear_gemv_group",
            "launch_unit": "one step: 4 grouped GEMV calls (8 launches), "
                           f"{step_bytes} algorithmic bytes",
            "traffic_source": TRAFFIC["profile"] if traffic else None,
            "codes_only_GBps": round(sum(inf["packed_bytes"] for _, inf in infos)
                                     / (ms_step * 1e-3) / 1e9, 1),
            "per_linear": per_lin_us}

    # end to end through the public API: pinned host x -> device, GEMVs,
    # y -> host, the host waiting for every step's results
    e2e = None
    if not args.no_e2e:
        # The step's inputs (one bf16 x per call) and outputs (one fp32 y per
        # linear) each sit in one contiguous buffer, so that a step moves
        # them with one host-to-device and one device-to-host copy.
        in_off, o = {}, 0
        for grp in GROUPS:
            in_off[grp[0]] = o
            o += batch * LLAMA[grp[0]][2]
        hx_all = torch.empty(o, dtype=torch.int16).pin_memory()
        for grp in GROUPS:
            K0 = LLAMA[grp[0]][2]
            hx_all[in_off[grp[0]]:in_off[grp[0]] + batch * K0] = torch.from_numpy(
                np.repeat(xs_np[grp[0]], batch, 0).view(np.int16).reshape(-1))
        dx_all = torch.empty(o, dtype=torch.int16, device=device)
        dxs = {g0: dx_all[in_off[g0]:in_off[g0] + batch * LLAMA[g0][2]].view(batch, LLAMA[g0][2])
               .view(torch.bfloat16) for g0 in in_off}
        out_off, o = [], 0
        for _, N, _ in LLAMA:
            out_off.append(o)
            o += batch * N
        ys_all = torch.empty(o, dtype=torch.float32, device=device)
        hy_all = torch.empty(o, dtype=torch.float32).pin_memory()
        ye = [ys_all[out_off[i]:out_off[i] + batch * N].view(batch, N)
              for i, (_, N, _) in enumerate(LLAMA)]
        h2d = hx_all.numel() * 2
        d2h = hy_all.numel() * 4
        e_steps = max(3, min(args.steps, 50))

        def e2e_step(c):
            dx_all.copy_(hx_all, non_blocking=True)
            for grp in GROUPS:
                polyq.linear_gemv_group([layers[i][c] for i in grp], [dxs[grp[0]]] * len(grp),
                                        ys=[ye[i] for i in grp], workspace=wbuf, stream=stream)
            hy_all.copy_(ys_all, non_blocking=True)

        # (1) the calls made eagerly every step
        with torch.cuda.stream(stream):
            for s in range(args.warmup + e_steps):
                if s == args.warmup:
                    stream.synchronize()
                    ta = time.perf_counter()
                e2e_step(s % args.copies)
                stream.synchronize()
            tb = time.perf_counter()
        eager = {"value": round(step_bytes * e_steps / (tb - ta) / 1e12, 4), "unit": "TB/s",
                 "ms_per_step": round(1e3 * (tb - ta) / e_steps, 4),
                 "mode": "API calls and copies issued eagerly every step"}
        # (2) each layer copy's step (copies and API calls) captured once as a
        # CUDA graph, replayed every step, the host synchronising every step
        e_graphs = []
        for c in range(args.copies):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                e2e_step(c)
            e_graphs.append(g)
        with torch.cuda.stream(stream):
            for s in range(args.warmup + e_steps):
                if s == args.warmup:
                    stream.synchronize()
                    ta = time.perf_counter()
                e_graphs[s % args.copies].replay()
                stream.synchronize()
            tb = time.perf_counter()
        e2e = {"value": round(step_bytes * e_steps / (tb - ta) / 1e12, 4), "unit": "TB/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": e_steps,
               "ms_per_step": round(1e3 * (tb - ta) / e_steps, 4),
               "mode": "each step's H2D copy of its inputs, 4 GEMV API calls and D2H copy of its "
                       "7 outputs captured as a CUDA graph, replayed and synchronised every step",
               "eager": eager}
        del e_graphs

    decode = None
    if not args.no_decode:
        decode = bench_decode_step(polyq, synth, torch, device, stream, args, hbm)

    qwen = None
    if not args.no_qwen:
        qwen = bench_qwen(polyq, synth, torch, device, stream, args, hbm)

    gemm = None
    if not args.no_gemm:
        gemm = bench_gemm(polyq, synth, torch, device, stream, args, tf_burst, tf_sus)

    sweep = None
    if not args.no_sweep and batch == 1:
        sweep = bench_budgets(polyq, synth, torch, device, stream, hbm)

    dense = None
    if not args.no_dense and batch == 1:
        dense = bench_dense(torch, device, stream, hbm)
        dense["polyq_step_speedup"] = round(dense["us_per_step"] / (ms_step * 1e3), 3)

    if rank == 0:
        cpu = None if (args.no_cpu_baseline or ws > 1) else cpu_baseline(args.cpu_seconds)
        plan = plan_report(polyq)
        quanta = quanta_report(polyq, synth)
        out = {
            "metric": METRIC, "value": round(value_tbs, 4), "unit": "TB/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 5),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "budget_bits": args.budget, "batch": batch,
                       "parallelism": f"replicas{ws}" if ws > 1 else "single-gpu",
                       "layer_copies": args.copies,
                       "l2": f"weights rotate over {args.copies} device copies "
                             f"({copy_bytes * args.copies / 2**20:.0f} MiB > L2 "
                             f"{L2 / 2**20:.0f} MiB)",
                       "bytes_per_step": step_bytes,
                       "b_real": {n: round(inf["b_real"], 5) for n, inf in infos},
                       "launch_groups": "q+k+v, o, gate+up, down (4 calls of 2 kernels)",
                       "graph": f"one CUDA graph of {args.copies} steps (one per layer "
                                "copy), replayed",
                       "timing": f"median of {n_win} windows of {args.steps} steps"},
            "pct_of_peak": round(100 * value_tbs * 1e3 / (hbm * ws), 2),
            "roofline": roof,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": args.steps * len(GROUPS) * kernels_per_call,
            "clocks": clk.summary(),
            "timing": timing,
            # the long reports first, the measured paths after them and a
            # compact summary last, where a tail of the output keeps them
            "permutation_plan": plan,
            "quanta_matching": quanta,
            "budget_sweep": sweep,
            "dense_bf16_context": dense,
            "one_launch_step": one_launch,
            "qwen3_32b_gemv": qwen,
            "decode_step": decode,
            "prefill_gemm": gemm,
        }
        out["summary"] = summary(out)
        print(json.dumps(out), flush=True)
    if ws > 1:
        dist.destroy_process_group()


def summary(out):
    """The headline figures of every measured path, compact."""
    sm = {"step_TBps": out["value"], "frac": out["roofline"]["frac"],
          "e2e_TBps": (out.get("e2e") or {}).get("value"),
          "one_launch_TBps": (out.get("one_launch_step") or {}).get("TB/s"),
          "sm_mhz": out["clocks"].get("sm_mhz"), "reasons": out["clocks"].get("reasons")}
    g = out.get("prefill_gemm")
    if g:
        sm["gemm_TFLOPs"] = {k: v["tflops"] for k, v in g.items() if isinstance(v, dict)
                             and "tflops" in v}
    d = out.get("decode_step")
    if d:
        sm["decode_40L_ms_per_token"] = {k: v.get("ms_per_token") for k, v in d.items()
                                         if isinstance(v, dict) and "ms_per_token" in v}
        ch = (d.get("grouped") or {}).get("chained")
        if ch:
            sm["decode_40L_chained_ms"] = ch.get("ms_per_token")
    q = out.get("qwen3_32b_gemv")
    if q:
        sm["qwen3_32b_TBps"] = {k: v.get("TB/s") for k, v in q.items() if isinstance(v, dict)
                                and "TB/s" in v}
    bs = out.get("budget_sweep")
    if bs:
        sm["budget_sweep_TBps"] = {k: v.get("TB/s") for k, v in bs.items() if isinstance(v, dict)
                                   and "TB/s" in v}
    return sm


def bench_decode_step(polyq, synth, torch, device, stream, args, hbm):
    """A whole batch-1 decode step of a Llama2-13B-shaped stack: for each of
    the layers, RMSNorm -> q,k,v -> o (+ residual) -> RMSNorm -> gate,up ->
    SiLU*up -> down (+ residual), attention at position 0 (output = v).  The
    glue runs inside the GEMV pre-passes and the §4.3 merges make o and down
    read their inputs without a gather.  Two modes: `separate` (seven linears,
    v -> o and gate/up -> down merged) and `grouped` (q/k/v and gate/up each
    allocated jointly over their stacked rows, sharing one permutation).
    The layers are device copies of one packed layer set, so every step
    streams all weights from HBM."""
    hidden, ffn, L = 5120, 13824, args.decode_layers
    W = {}
    for i, (name, N, K) in enumerate(LLAMA):
        W[name] = synth.layer_weights(N, K, synth.seed_for(5, i))
    a_in = {"q": W["q"][1], "k": W["q"][1], "v": W["q"][1], "o": W["o"][1],
            "gate": W["gate"][1], "up": W["gate"][1], "down": W["down"][1]}
    gathered = {}
    out = {}
    for mode in ("separate", "grouped"):
        if mode == "separate":
            hosts = {n: polyq.HostLayer.pack(W[n][0], a_in[n], args.budget) for n in W}
            p_o = hosts["o"].export()["perm"]
            p_d = hosts["down"].export()["perm"]
            hosts["v"].permute_rows(p_o)
            hosts["gate"].permute_rows(p_d)
            hosts["up"].permute_rows(p_d)
            names = list(W)
        else:
            hosts = {"qkv": polyq.HostLayer.pack(np.vstack([W["q"][0], W["k"][0], W["v"][0]]),
                                                 a_in["q"], args.budget),
                     "o": polyq.HostLayer.pack(W["o"][0], a_in["o"], args.budget),
                     "gu": polyq.HostLayer.pack(np.vstack([W["gate"][0], W["up"][0]]),
                                                a_in["gate"], args.budget),
                     "down": polyq.HostLayer.pack(W["down"][0], a_in["down"], args.budget)}
            p_o = hosts["o"].export()["perm"]
            p_d = hosts["down"].export()["perm"]
            hosts["qkv"].permute_rows(np.concatenate([np.arange(2 * hidden), 2 * hidden + p_o]))
            hosts["gu"].permute_rows(np.concatenate([p_d, ffn + p_d]))
            names = list(hosts)
        base = {n: polyq.DeviceLayer(hosts[n], device, identity_gather=n in ("o", "down"))
                for n in names}
        stack = [base] + [{n: base[n].clone() for n in names} for _ in range(L - 1)]
        step_bytes = L * sum(base[n].info["packed_bytes"] + base[n].info["meta_bytes"]
                             for n in names)
        s = torch.zeros((1, hidden), dtype=torch.float32, device=device)
        s0 = torch.from_numpy(np.random.default_rng(5).standard_normal((1, hidden))
                              .astype(np.float32)).to(device)
        if mode == "separate":
            q, k, v = (torch.empty((1, hidden), dtype=torch.float32, device=device)
                       for _ in range(3))
            g, u = (torch.empty((1, ffn), dtype=torch.float32, device=device) for _ in range(2))
            wsb = torch.zeros(max(polyq.gemv_group_workspace_bytes(
                [base["gate"], base["up"]], 1), 1 << 20), dtype=torch.uint8, device=device)
        else:
            yqkv = torch.empty((1, 3 * hidden), dtype=torch.float32, device=device)
            ygu = torch.empty((1, 2 * ffn), dtype=torch.float32, device=device)
            wsb = torch.zeros(max(polyq.gemv_group_workspace_bytes([base["gu"]], 1), 1 << 20),
                              dtype=torch.uint8, device=device)

        def run_step():
            for lay in stack:
                if mode == "separate":
                    polyq.linear_gemv_input([lay["q"], lay["k"], lay["v"]], polyq.X_RMSNORM, s,
                                            ys=[q, k, v], workspace=wsb, stream=stream)
                    polyq.linear_gemv_input([lay["o"]], polyq.X_F32, v, ys=[s], residuals=[s],
                                            workspace=wsb, stream=stream)
                    polyq.linear_gemv_input([lay["gate"], lay["up"]], polyq.X_RMSNORM, s,
                                            ys=[g, u], workspace=wsb, stream=stream)
                    polyq.linear_gemv_input([lay["down"]], polyq.X_SILU_MUL, g, b=u, ys=[s],
                                            residuals=[s], workspace=wsb, stream=stream)
                else:
                    polyq.linear_gemv_input([lay["qkv"]], polyq.X_RMSNORM, s, ys=[yqkv],
                                            workspace=wsb, stream=stream)
                    polyq.linear_gemv_input([lay["o"]], polyq.X_F32, yqkv[:, 2 * hidden:],
                                            ys=[s], residuals=[s], workspace=wsb, stream=stream)
                    polyq.linear_gemv_input([lay["gu"]], polyq.X_RMSNORM, s, ys=[ygu],
                                            workspace=wsb, stream=stream)
                    polyq.linear_gemv_input([lay["down"]], polyq.X_SILU_MUL, ygu[:, :ffn],
                                            b=ygu[:, ffn:], ys=[s], residuals=[s],
                                            workspace=wsb, stream=stream)

        with torch.cuda.stream(stream):
            s.copy_(s0)
            run_step()
        stream.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            s.copy_(s0)  # every token starts from the same stream state
            run_step()
        reps = max(3, args.decode_steps)
        with torch.cuda.stream(stream):
            for _ in range(3):
                graph.replay()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(reps):
                graph.replay()
            e1.record(stream)
        stream.synchronize()
        ms = e0.elapsed_time(e1) / reps
        finite = bool(torch.isfinite(s).all())
        tbs = step_bytes / (ms * 1e-3) / 1e12
        gathered[mode] = (5 * hidden if mode == "separate" else 2 * hidden)
        out[mode] = {"ms_per_token": round(ms, 4), "packed_bytes_per_token": step_bytes,
                     "TB/s": round(tbs, 4), "frac_of_hbm": round(tbs * 1e3 / hbm, 4),
                     "kernel_launches_per_token": 8 * L, "stream_finite": finite}
        if mode == "grouped":
            # the same token as one persistent launch (polyq_linear_gemv_chain)
            phases = []
            for lay in stack:
                phases += [
                    dict(layers=[lay["qkv"]], kind=polyq.X_RMSNORM, a=s, eps=1e-6, ys=[yqkv]),
                    dict(layers=[lay["o"]], kind=polyq.X_F32, a=yqkv[:, 2 * hidden:], ys=[s],
                         residuals=[s]),
                    dict(layers=[lay["gu"]], kind=polyq.X_RMSNORM, a=s, eps=1e-6, ys=[ygu]),
                    dict(layers=[lay["down"]], kind=polyq.X_SILU_MUL, a=ygu[:, :ffn],
                         b=ygu[:, ffn:], ys=[s], residuals=[s])]
            chain = polyq.GemvChain(phases, batch=1, stream=stream)
            s_graph = s.clone()  # the graph's token (every replay starts from s0)
            with torch.cuda.stream(stream):
                s.copy_(s0)
                chain.run(stream=stream)
            stream.synchronize()
            agree = float((s - s_graph).norm() / s_graph.norm())
            with torch.cuda.stream(stream):
                c0 = torch.cuda.Event(enable_timing=True)
                c1 = torch.cuda.Event(enable_timing=True)
                c0.record(stream)
                for _ in range(reps):
                    s.copy_(s0)
                    chain.run(stream=stream)
                c1.record(stream)
            stream.synchronize()
            cms = c0.elapsed_time(c1) / reps
            out[mode]["chained"] = {
                "ms_per_token": round(cms, 4),
                "TB/s": round(step_bytes / (cms * 1e-3) / 1e12, 4),
                "kernel_launches_per_token": 1, "phases": len(phases),
                "rel_diff_vs_graph": round(agree, 6),
                "status": int(chain.workspace[:4].view(torch.int32).item())}
            del chain
        del stack, base, hosts
        torch.cuda.empty_cache()
    # §5.4 model of activation-reorder traffic per token (A16 read + write of
    # each explicit shuffle): without merges every linear shuffles its input
    no_merge = 4 * L * sum(k for _, _, k in LLAMA)
    for mode in out:
        kept = 4 * L * gathered[mode]
        out[mode]["reorder_traffic_mib"] = round(kept / 2 ** 20, 3)
        out[mode]["reorder_traffic_removed"] = round(1 - kept / no_merge, 4)
    out["reorder_traffic_no_merge_mib"] = round(no_merge / 2 ** 20, 3)
    out["workload"] = (f"llama2-13b decode step, {L} layers (device copies of one packed "
                       f"layer set), batch 1, B={args.budget}, position 0")
    return out


def plan_report(polyq):
    """§4.4 planning of the whole decode graph (host, no GPU) on the
    Llama2-13B and Qwen3-32B shapes: modelled activation-reorder traffic per
    token (§5.4 model) without merges and with the library planner, for
    separately allocated linears and for q/k/v and gate/up allocated jointly.
    Every layer gets its own seeded permutations (distinct allocations)."""
    shapes = {"llama2_13b": dict(layers=40, hidden=5120, ffn=13824, kv=None, qdim=None,
                                 paper_polyq_mib=1.14, paper_no_merge_mib=6.80),
              "qwen3_32b": dict(layers=64, hidden=5120, ffn=25600, kv=1024, qdim=8192,
                                paper_polyq_mib=2.95, paper_no_merge_mib=14.50)}
    out = {}
    for name, c in shapes.items():
        res = {}
        for mode in ("separate", "grouped"):
            rng = np.random.default_rng(7)
            perms, ids = [], {}

            def perm_of(l, nm):
                key = (l, {"q": "qkv", "k": "qkv", "v": "qkv", "gate": "gu", "up": "gu"}
                       .get(nm, nm) if mode == "grouped" else nm)
                if key not in ids:
                    width = {"o": c["qdim"] or c["hidden"], "down": c["ffn"]}.get(nm, c["hidden"])
                    ids[key] = len(perms)
                    perms.append(rng.permutation(width).astype(np.int32))
                return ids[key]

            nodes, dims, _ = polyq.decoder_plan_graph(c["layers"], c["hidden"], c["ffn"], perm_of,
                                                      c["kv"], c["qdim"])
            t0 = time.perf_counter()
            _, cost = polyq.plan_graph(nodes, dims, perms)
            dt = time.perf_counter() - t0
            no_merge = 4 * sum(dims[i[0]] for k, i, o, p in nodes if k == polyq.NODE_LINEAR)
            res[mode] = {"planned_mib": round(cost / 2 ** 20, 3),
                         "removed": round(1 - cost / no_merge, 4), "planner_ms": round(dt * 1e3, 2)}
            # the same stack entered from an embedding whose columns may be
            # permuted and left through a linear output head (its own gather
            # counted): the stream region may then take one layer's order
            perms.append(rng.permutation(c["hidden"]).astype(np.int32))
            nodes, dims, _ = polyq.decoder_plan_graph(c["layers"], c["hidden"], c["ffn"], perm_of,
                                                      c["kv"], c["qdim"], True,
                                                      (len(perms) - 1, 32000))
            _, cost_h = polyq.plan_graph(nodes, dims, perms)
            res[mode]["free_embedding_linear_head_mib"] = round(cost_h / 2 ** 20, 3)
        res["no_merge_mib"] = round(no_merge / 2 ** 20, 3)
        res["paper_no_merge_mib"] = c["paper_no_merge_mib"]
        res["paper_polyq_mib"] = c["paper_polyq_mib"]
        out[name] = res
    return out


def quanta_report(polyq, synth):
    """§3.3 quanta matching on the synthetic layer generator (host, no GPU):
    realised mean width and segment padding before and after snapping to
    the GPU quanta (one 16-byte chunk per quantum), over the §5.2 budget
    sweep, for the input widths of the Llama2-13B and Qwen3-32B linears
    (256 rows each: the allocation depends on the rows only through the
    column norms)."""
    out = {}
    for K in (5120, 8192, 13824, 25600):
        W, a = synth.layer_weights(256, K, 40000 + K)
        rows = []
        for B in (3.0, 3.5, 4.0, 4.5, 5.0, 5.5, 6.0):
            raw = polyq.HostLayer.pack(W, a, B).info()
            snap = polyq.HostLayer.pack(W, a, B, snap_quanta=True).info()
            rows.append({"B": B, "b_real_raw": round(raw["b_real"], 5),
                         "b_real_snapped": round(snap["b_real"], 5),
                         "pad_pct_raw": round(100 * raw["pad_bytes"] / raw["row_stride"], 3),
                         "pad_pct_snapped": round(100 * snap["pad_bytes"] / snap["row_stride"], 3)})
        out[f"K{K}"] = {"max_abs_mismatch": round(max(abs(r["b_real_snapped"] - r["B"])
                                                      for r in rows), 5),
                        "sweep": rows}
    return out


QWEN = [("q", 8192, 5120), ("k", 1024, 5120), ("v", 1024, 5120), ("o", 5120, 8192),
        ("gate", 25600, 5120), ("up", 25600, 5120), ("down", 5120, 25600)]


def time_grouped_step(polyq, synth, torch, device, stream, shapes, config, budget, batches,
                      copies, hbm):
    """One decoder layer's seven linears of ``shapes`` (seeded from synthetic
    config ``config``) packed at ``budget`` and run as the four grouped calls
    (q+k+v, o, gate+up, down), timed as a CUDA graph of steps over ``copies``
    device copies of the layer."""
    layers, xs_np, infos = [], [None] * len(shapes), []
    for i, (name, N, K) in enumerate(shapes):
        W, a = synth.layer_weights(N, K, synth.seed_for(config, i))
        host = polyq.HostLayer.pack(W, a, budget)
        dev = polyq.DeviceLayer(host, device)
        infos.append(host.info())
        layers.append([dev] + [dev.clone() for _ in range(copies - 1)])
        xs_np[i] = a
        del W
    out = {}
    for batch in batches:
        xs = []
        for grp in GROUPS:
            xb, _ = synth.activations(xs_np[grp[0]], batch, 11 + grp[0])
            t = torch.from_numpy(xb.view(np.int16)).to(device).view(torch.bfloat16)
            xs += [t] * len(grp)
        ys = [torch.empty((batch, N), dtype=torch.float32, device=device) for _, N, _ in shapes]
        wsz = max(polyq.gemv_group_workspace_bytes([layers[i][0] for i in grp], batch)
                  for grp in GROUPS)
        wbuf = torch.zeros(max(wsz, 256), dtype=torch.uint8, device=device)
        step_bytes = sum(layer_bytes(inf, batch) for inf in infos)
        codes = sum(inf["packed_bytes"] for inf in infos)

        def run_step(c):
            for grp in GROUPS:
                polyq.linear_gemv_group([layers[i][c] for i in grp], [xs[i] for i in grp],
                                        ys=[ys[i] for i in grp], workspace=wbuf, stream=stream)

        with torch.cuda.stream(stream):
            run_step(0)
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for c in range(copies):
                run_step(c)
        reps = 50
        with torch.cuda.stream(stream):
            for _ in range(3):
                g.replay()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(reps):
                g.replay()
            e1.record(stream)
        stream.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / (reps * copies)
        tbs = step_bytes / (us * 1e-6) / 1e12
        out[f"batch{batch}"] = {"us_per_step": round(us, 2), "bytes_per_step": step_bytes,
                                "TB/s": round(tbs, 4), "frac_of_hbm": round(tbs * 1e3 / hbm, 4),
                                "codes_only_TB/s": round(codes / (us * 1e-6) / 1e12, 4)}
    out["b_real"] = {n: round(inf["b_real"], 5) for (n, _, _), inf in zip(shapes, infos)}
    del layers
    torch.cuda.empty_cache()
    return out


def bench_qwen(polyq, synth, torch, device, stream, args, hbm):
    """The Qwen3-32B-shaped decode linears (q 8192x5120, k/v 1024x5120,
    o 5120x8192, gate/up 25600x5120, down 5120x25600) at the budget of the
    run, batch 1 and 4: one step is the four grouped calls (q+k+v, o,
    gate+up, down), timed as a CUDA graph of steps over two device copies of
    the layer (372 MB at B = 3, larger than L2)."""
    out = {"workload": f"qwen3-32b decode linears, B={args.budget}, groups q+k+v, o, gate+up, "
                       "down, 2 device copies"}
    out.update(time_grouped_step(polyq, synth, torch, device, stream, QWEN, 3, args.budget,
                                 (1, 4), 2, hbm))
    return out


def bench_budgets(polyq, synth, torch, device, stream, hbm):
    """The other budgets of the Llama2-13B (B = 4.5) and Qwen3-32B (B = 3.5,
    4, 5, 6) decode linears, batch 1: the same four grouped calls per step,
    timed over two device copies (every set is larger than L2)."""
    out = {"what": "four grouped GEMV calls per step, batch 1, 2 device copies"}
    for model, shapes, config, budgets in (("llama2_13b", LLAMA, 2, (4.5,)),
                                           ("qwen3_32b", QWEN, 3, (3.5, 4.0, 5.0, 6.0))):
        for B in budgets:
            r = time_grouped_step(polyq, synth, torch, device, stream, shapes, config, B, (1,), 2,
                                  hbm)
            out[f"{model}_B{B}"] = dict(r["batch1"], b_real_min=min(r["b_real"].values()),
                                        b_real_max=max(r["b_real"].values()))
    return out


def bench_dense(torch, device, stream, hbm, copies=2):
    """Context, not the product: the same seven Llama2-13B decode linears as
    dense bf16 matrix-vector products through torch (cuBLAS), batch 1, timed
    as a CUDA graph over two copies of the weights (1.27 GB)."""
    g = torch.Generator(device=device)
    g.manual_seed(7)
    Ws = [[(torch.randn((N, K), device=device, generator=g) * 0.02).to(torch.bfloat16)
           for _, N, K in LLAMA] for _ in range(copies)]
    xs = [torch.randn((1, K), device=device, generator=g).to(torch.bfloat16) for _, _, K in LLAMA]
    ys = [None] * len(LLAMA)
    step_bytes = sum(2 * N * K + 2 * K + 2 * N for _, N, K in LLAMA)

    def run_step(c):
        for i in range(len(LLAMA)):
            ys[i] = torch.nn.functional.linear(xs[i], Ws[c][i])

    with torch.cuda.stream(stream):
        run_step(0)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for c in range(copies):
            run_step(c)
    reps = 50
    with torch.cuda.stream(stream):
        for _ in range(3):
            graph.replay()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            graph.replay()
        e1.record(stream)
    stream.synchronize()
    us = e0.elapsed_time(e1) * 1e3 / (reps * copies)
    tbs = step_bytes / (us * 1e-6) / 1e12
    del Ws
    torch.cuda.empty_cache()
    return {"what": "context only: dense bf16 y = x W^T of the seven Llama2-13B linears, "
                    "torch/cuBLAS, batch 1, 7 launches per step",
            "us_per_step": round(us, 2), "bytes_per_step": step_bytes, "TB/s": round(tbs, 4),
            "frac_of_hbm": round(tbs * 1e3 / hbm, 4)}


def bench_gemm(polyq, synth, torch, device, stream, args, tf_burst, tf_sus):
    """Prefill GEMM on the gate/up/down linears at M=2048 (TFLOP/s)."""
    res = {}
    try:
        for name, N, K in (("gate", 13824, 5120), ("down", 5120, 13824)):
            W, a = synth.layer_weights(N, K, synth.seed_for(4, 0 if name == "gate" else 2))
            host = polyq.HostLayer.pack(W, a, args.budget)
            dev = polyq.DeviceLayer(host, device)
            for M in (512, 2048):
                Xb, _ = synth.activations(a, M, synth.seed_for(4, 10))
                X = torch.from_numpy(Xb.view(np.int16)).to(device).view(torch.bfloat16)
                Y = torch.empty((M, N), dtype=torch.float32, device=device)
                wsb = torch.empty(max(polyq.gemm_workspace_bytes(dev, M), 256), dtype=torch.uint8,
                                  device=device)
                with torch.cuda.stream(stream):
                    for _ in range(3):
                        polyq.linear_gemm(dev, X, Y=Y, workspace=wsb, stream=stream)
                    e0 = torch.cuda.Event(enable_timing=True)
                    e1 = torch.cuda.Event(enable_timing=True)
                    reps = 20
                    e0.record(stream)
                    for _ in range(reps):
                        polyq.linear_gemm(dev, X, Y=Y, workspace=wsb, stream=stream)
                    e1.record(stream)
                stream.synchronize()
                ms = e0.elapsed_time(e1) / reps
                tf = 2.0 * M * N * K / (ms * 1e-3) / 1e12
                res[f"{name}_M{M}"] = {"tflops": round(tf, 1), "us": round(1e3 * ms, 1),
                                       "frac_of_burst": round(tf / tf_burst, 4)}
            del W
    except polyq.PolyqError as e:
        return {"unavailable": str(e)}
    return res


def sample_bytes(L, x, N):
    """Algorithmic bytes of an oracle run on a row sample of a linear with N
    rows: the sample's packed codes and metadata, plus the layer's
    activations, gather indices and outputs in proportion to the sample's
    share of the rows (over the full layer they are spread over all N)."""
    rows = L["N"]
    return (L["packed"].nbytes + L["meta"].nbytes
            + (x.size * 2 + L["K"] * 4 + x.shape[0] * N * 4) * rows / N)


def _blas_threads():
    v = os.environ.get("OPENBLAS_NUM_THREADS") or os.environ.get("OMP_NUM_THREADS")
    return int(v) if v else os.cpu_count()


def cpu_baseline(seconds):
    """The oracle timed on the host cores in child processes (no CUDA state):
    with BLAS pinned to one thread (the reported baseline) and with BLAS free
    to use every core."""
    runs = {}
    for threads in (1, os.cpu_count() or 1):
        env = dict(os.environ, OPENBLAS_NUM_THREADS=str(threads), OMP_NUM_THREADS=str(threads))
        r = subprocess.run([sys.executable, os.path.abspath(__file__), "--cpu-baseline-child",
                            "--cpu-seconds", str(seconds)], env=env, capture_output=True,
                           text=True, timeout=600)
        if r.returncode != 0:
            return {"unavailable": f"oracle child exited {r.returncode}: {r.stderr[-300:]}"}
        runs[threads] = json.loads(r.stdout.strip().splitlines()[-1])
    one = runs[1]
    many = runs[max(runs)]
    one["all_cores"] = {"value": many["value"], "unit": many["unit"], "cores": many["cores"],
                        "note": "BLAS free to use every host core; unpacking and dequantising "
                                "stay single-threaded numpy"}
    return one


def cpu_baseline_child(seconds):
    """The oracle's linear (unpack + dequantise + fp64 dot from the packed
    bytes) on a bounded sample of the workload: row slices of the seven
    linears, repeated until about ``seconds`` of CPU time."""
    from oracle import polyq_oracle as O
    from paper_2607_14618_gb300 import synth
    rows = 256
    layers = []
    for i, (name, N, K) in enumerate(LLAMA):
        W, a = synth.layer_weights(N, K, synth.seed_for(2, i))
        bits = O.allocate_bits(O.saliency(W, a), 3.0)
        L = O.pack_layer(W[:rows], a, 3.0, bits=bits)
        _, x = synth.activations(a, 1, synth.seed_for(2, i))
        layers.append((L, x))
        del W
    nbytes = 0
    t0 = time.perf_counter()
    while time.perf_counter() - t0 < seconds:
        for (L, x), (_, N, _) in zip(layers, LLAMA):
            O.linear(L, x)
            nbytes += sample_bytes(L, x, N)
    dt = time.perf_counter() - t0
    return {"value": round(nbytes / dt / 1e12, 8), "unit": "TB/s",
            "cores": _blas_threads(), "host_cpus": os.cpu_count(),
            "kind": "oracle",
            "sample": f"{rows} output rows of each of the 7 linears, oracle linear "
                      f"(unpack+dequant+fp64 dot) repeated for {dt:.1f} s"}


def run_reference(args):
    """The reference arm: the oracle's linear on the host cores, on a row
    sample of each of the seven linears per step.  The sample is sized so that
    the warm-up and timed steps together take about ``REF_SECONDS`` whatever
    --steps is (from 1 to 128 rows per linear; the metric is bytes per second,
    so the sample size does not change what is measured)."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    from oracle import polyq_oracle as O
    from paper_2607_14618_gb300 import synth
    max_rows = 128
    srcs = []  # (first max_rows rows of W, channel magnitudes, widths) per linear
    for i, (name, N, K) in enumerate(LLAMA):
        W, a = synth.layer_weights(N, K, synth.seed_for(2, i))
        bits = O.allocate_bits(O.saliency(W, a), args.budget)
        srcs.append((W[:max_rows].copy(), a, bits))
        del W

    def build(rows):
        out = []
        for i, (Wr, a, bits) in enumerate(srcs):
            L = O.pack_layer(Wr[:rows], a, args.budget, bits=bits)
            _, x = synth.activations(a, 1, synth.seed_for(2, i))
            out.append((L, x))
        return out

    def step(layers):
        n = 0
        for (L, x), (_, N, _) in zip(layers, LLAMA):
            O.linear(L, x)
            n += sample_bytes(L, x, N)
        return n

    def step_seconds(rows):
        layers = build(rows)
        step(layers)
        t0 = time.perf_counter()
        for _ in range(3):
            step(layers)
        return (time.perf_counter() - t0) / 3

    t1, t8 = step_seconds(1), step_seconds(8)
    per_row = max((t8 - t1) / 7, 1e-6)
    fixed = max(t1 - per_row, 0.0)
    rows = int((REF_SECONDS / max(args.steps + args.warmup, 1) - fixed) / per_row)
    rows = max(1, min(max_rows, rows))
    layers = build(rows)
    for _ in range(args.warmup):
        step(layers)
    t0 = time.perf_counter()
    nb = sum(step(layers) for _ in range(args.steps))
    dt = time.perf_counter() - t0
    v = nb / dt / 1e12
    out = {"impl": "reference", "metric": METRIC, "value": round(v, 8), "unit": "TB/s",
           "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(1e3 * dt / args.steps, 3), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": WORKLOAD, "budget_bits": args.budget, "batch": 1},
           "cpu_baseline": {"kind": "oracle", "cores": _blas_threads(), "host_cpus": os.cpu_count(),
                            "value": round(v, 8), "unit": "TB/s",
                            "sample": f"{rows} output rows of each of the 7 linears per step "
                                      f"(sized for about {REF_SECONDS:.0f} s of steps)"},
           "e2e": {"value": round(v, 8), "unit": "TB/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="polyq", choices=["polyq", "reference"])
    ap.add_argument("--budget", type=float, default=3.0)
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--copies", type=int, default=6)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-gemm", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-qwen", action="store_true")
    ap.add_argument("--decode-layers", type=int, default=40)
    ap.add_argument("--decode-steps", type=int, default=20)
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-dense", action="store_true")
    ap.add_argument("--timed-seconds", type=float, default=1.5,
                    help="repeat the timed window of --steps steps for about this long")
    ap.add_argument("--max-windows", type=int, default=2000)
    ap.add_argument("--cpu-baseline-child", action="store_true", help=argparse.SUPPRESS)
    args = ap.parse_args()
    if args.cpu_baseline_child:
        print(json.dumps(cpu_baseline_child(args.cpu_seconds)), flush=True)
        return
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_polyq(args)


if __name__ == "__main__":
    main()
