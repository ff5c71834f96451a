"""Benchmark: block-restricted bidirectional selective scan, forward + backward.

One step = the all-block forward (bdscan_forward) and backward
(bdscan_backward) of one layer on one batch of synthetic input, through the
C ABI, on the 87M-scale layer configuration: batch 8, clean and noisy streams
of 2048 tokens, block 16, d_inner 1536, d_state 16, bf16 inputs/outputs with
fp32 state. Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
  python bench.py --workload sweep|prefill65k|prefill262k   (one GPU; extra lines)

The extra workloads print one JSON line per measurement instead of the
step line: the block-size sweep at d_inner 2048 (forward+backward for block
4, 8, 16, 32, 64), and the inference cache path: boundary_states over a
65,536-token prefix (block 32) or a 262,144-token prefix (block 16), then
active-block calls from the cached state, each call timed on its own and all
calls replayed as one CUDA graph, and the cost of the same layer step without
the cache (full-sequence bidirectional scan).

Under torchrun each rank runs an independent replica on its own GPU (the
scan needs no exchange between replicas); the elapsed time is the maximum
over ranks and the value counts the tokens of all ranks. --impl reference
times the fp64 CPU oracle (the reference arm of this method) on a bounded
sample of the same workload, on rank 0 only.
"""

from __future__ import annotations

import argparse
import ctypes
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

METRIC = "block-bidir scan fwd+bwd tokens/sec on 1 GB300; achieved HBM GB/s vs ~8 TB/s"
CFG = dict(batch=8, seq_len=2048, block=16, d_inner=1536, d_state=16)
WORKLOAD = ("87M-scale layer: batch 8, clean+noisy streams of 2048 tokens each, block 16, d_inner 1536, "
            "d_state 16, bf16 inputs/outputs, fp32 state; all-block forward + backward")
KERNELS = ["chunk_local", "chunk_carry", "block_scan", "bwd_noisy", "bwd_carry", "bwd_clean", "reduce_tok",
           "reduce_par"]


def algorithmic_bytes(Bt, L, D, N, Bs, in_b=2, out_b=2):
    """Bytes one forward+backward step must move at least: every input read
    once per pass, every output written once, boundary states written by the
    forward and read by the backward (no recompute or workspace traffic)."""
    nb = L // Bs
    td = Bt * L * D
    tn = Bt * L * N
    fwd = 5 * td * in_b + 6 * tn * in_b + 2 * td * out_b + Bt * nb * D * N * 4
    bwd = (5 * td * in_b + 2 * td * in_b + 6 * tn * in_b + Bt * nb * D * N * 4
           + 5 * td * out_b + 6 * tn * out_b)
    return fwd, bwd


def kernel_bytes(Bt, L, D, N, Bs, in_b=2, out_b=2):
    """Per-kernel algorithmic bytes (the layer's own inputs and outputs each
    kernel has to touch; workspace exchange between kernels excluded)."""
    td, tn, nb = Bt * L * D, Bt * L * N, L // Bs
    S = Bt * nb * D * N * 4
    return {
        "chunk_local": 2 * td * in_b + tn * in_b,
        "chunk_carry": 0,
        "block_scan": 5 * td * in_b + 6 * tn * in_b + 2 * td * out_b + S,
        "bwd_noisy": 6 * td * in_b + 5 * tn * in_b + S + 3 * td * out_b,
        "bwd_carry": 0,
        "bwd_clean": 3 * td * in_b + 2 * tn * in_b + S + 2 * td * out_b,
        "reduce_tok": 6 * tn * out_b,
        "reduce_par": 0,
    }


# DRAM bytes (read + write) per launch of the dominant kernel, from one
# `ncu --set full` capture of the same kernel at batch 4, scaled by batch / 4:
# the kernel's traffic is proportional to the batch. Set to None whenever the
# kernel changes until it is captured again.
MEASURED_TRAFFIC_BATCH4 = {"bwd_noisy": 330_749_440}

# FP32 operations per (token, channel, state) element of each pass the scan
# kernels make, listed as the kernels write them (an FMA counts 2, ex2, mul,
# add and a reduction add 1 each):
#   scan       forward step with output: dt*A, ex2, u*B, a*h+uB, C*h+acc
#   scan_state forward step without output: dt*A, ex2, u*B, a*h+uB
#   recompute  backward recompute: dt*A, ex2, a*h, u*B+p, dy*h, channel add (dC)
#   adjoint    backward adjoint: dt*A, ex2, C*dy+g, a*gb, gb*p, A*q+sa, dt*q+dA,
#              gb*B+sg, gb*u, channel add (dB)
#   half       the half-state scheme's rebuild of every other state, per
#              element and token: (u*B + a*S) every second token
#   local      chunk-local adjoint carry: dt*A, ex2, C*dy+carry, a*(...)
PASS_FLOPS = {
    "scan": 1 + 1 + 1 + 2 + 2,
    "scan_state": 1 + 1 + 1 + 2,
    "recompute": 1 + 1 + 1 + 2 + 1 + 1,
    "adjoint": 1 + 1 + 2 + 1 + 1 + 2 + 2 + 2 + 1 + 1,
    "half": (2 + 1) / 2,
    "local": 1 + 1 + 2 + 1,
}
# The passes of each kernel per element (blocks of one 16-token segment).
KERNEL_PASSES = {
    "chunk_local": ["scan_state"],
    "block_scan": ["scan", "scan", "scan"],                     # clean rescan, noisy forward, noisy reverse
    "bwd_noisy": ["local"] + ["recompute", "adjoint"] * 2,      # clean local adjoint, both noisy directions
    "bwd_clean": ["recompute", "adjoint", "half"],
}


def kernel_flops_per_elem(name):
    return sum(PASS_FLOPS[q] for q in KERNEL_PASSES.get(name, []))


def sample_clocks(stop, rows, bus_id):
    cmd = ["nvidia-smi", "--query-gpu=pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
           "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
           "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
           "--format=csv,noheader,nounits", "-lms", "200"]
    try:
        p = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
    except OSError:
        return
    try:
        for line in p.stdout:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            if bus_id and bus_id.lower() not in f[0].lower() and f[0].lower() not in bus_id.lower():
                continue
            rows.append((time.time(), f))
            if stop.is_set():
                break
    finally:
        p.terminate()
        try:
            p.wait(timeout=2)
        except Exception:
            p.kill()


def summarize_clocks(rows, t0, t1):
    inside = [f for (ts, f) in rows if t0 <= ts <= t1]
    used = inside if len(inside) >= 3 else [f for (_, f) in rows]
    if not used:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"], "samples": 0}

    def num(x):
        try:
            return float(x)
        except ValueError:
            return None

    sm = [num(f[1]) for f in used if num(f[1]) is not None]
    reasons = set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for f in used:
        for name, v in zip(names, f[5:9]):
            if v.strip().lower() == "active":
                reasons.add(name)
    return {"sm_mhz": statistics.median(sm) if sm else None,
            "sm_max_mhz": max(num(f[2]) or 0 for f in used),
            "power_w_max": max((num(f[3]) or 0) for f in used),
            "reasons": sorted(reasons), "samples": len(used),
            "window": "timed region" if len(inside) >= 3 else "warm-up and timed region"}


def max_over_ranks(x, device, world):
    """The largest value of x over all ranks (the slowest replica's time)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_rank, world, ms_per_step):
    """Whole-job throughput: the tokens every replica processed in one step,
    over the slowest replica's step time (weak scaling: fixed work per GPU)."""
    return tokens_per_rank * world / (ms_per_step / 1e3)


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "sm_max_mhz": 2070.0}, "fallback"


# ---------------------------------------------------------------------------
# CPU oracle (reference arm and cpu_baseline)
# ---------------------------------------------------------------------------
def oracle_run(d_sample, seed=0, threads=None):
    """fp64 oracle forward+backward on the configuration restricted to
    `d_sample` channels (channels are independent, so the work is exactly
    d_sample/d_inner of the full step). Returns (seconds, threads)."""
    import oracle
    from paper_2607_02805_gb300.inputs import Workload
    oracle.build()
    th = threads or max(1, min(os.cpu_count() or 1, 64))
    oracle.set_threads(th)
    wl = Workload(CFG["batch"], CFG["seq_len"], CFG["block"], d_sample, CFG["d_state"], dtype="bf16", seed=seed)
    names = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r", "A_f", "D_f", "A_r",
             "D_r")
    d = {k: wl.f64(k) for k in wl.t32}
    t0 = time.perf_counter()
    y_c, y_n, st = oracle.forward(CFG["block"], *[d[k] for k in names])
    oracle.backward(CFG["block"], *[d[k] for k in names], st, d["dy_c"], d["dy_n"], None)
    return time.perf_counter() - t0, th


def run_reference(args, rank, world):
    if rank != 0:
        return
    # size each step so the whole run stays within about 90 s of wall time
    per_step = 90.0 / max(1, args.steps + args.warmup)
    # measured: about 20 ns per (token, channel, state, stream) on one core, fwd+bwd
    full_core_s = CFG["batch"] * CFG["seq_len"] * CFG["d_inner"] * CFG["d_state"] * 3 * 20e-9
    th = max(1, min(os.cpu_count() or 1, 64))
    eff = min(th, CFG["batch"])  # the oracle's backward runs one batch row per thread
    d_s = int(max(8, min(CFG["d_inner"], CFG["d_inner"] * per_step * eff / full_core_s)))
    for _ in range(args.warmup):
        oracle_run(d_s, threads=th)
    times = [oracle_run(d_s, threads=th)[0] for _ in range(args.steps)]
    tok = CFG["batch"] * CFG["seq_len"] * d_s / CFG["d_inner"]
    total = sum(times)
    value = tok * args.steps / total
    sample = (f"fp64 oracle fwd+bwd on {d_s} of {CFG['d_inner']} channels (batch 8, 2048 tokens, block 16, "
              f"d_state 16); tokens scaled by {d_s}/{CFG['d_inner']}")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": WORKLOAD, **CFG, "parallelism": "cpu threads"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": th, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    from paper_2607_02805_gb300 import binding
    from paper_2607_02805_gb300.inputs import Workload
    from paper_2607_02805_gb300.layer import Layer

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    Bt, L, Bs, D, N = CFG["batch"], CFG["seq_len"], CFG["block"], CFG["d_inner"], CFG["d_state"]
    wl = Workload(Bt, L, Bs, D, N, dtype="bf16", seed=rank, with_grads=True)
    lay = Layer(wl, device=dev)
    lay.alloc_backward()
    stream = torch.cuda.current_stream(dev)

    def step():
        lay.forward(stream)
        lay.backward(stream, use_dstates=False)

    # per-kernel events through the library's timing hook
    nk = len(KERNELS)
    ev_start = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev_k = [[torch.cuda.Event(enable_timing=True) for _ in range(nk)] for _ in range(args.steps)]
    for evs in ev_k:  # torch creates the CUDA event on its first record
        for e in evs:
            e.record(stream)
    torch.cuda.synchronize(dev)
    arr_f = [(ctypes.c_void_p * 3)(*[e.cuda_event for e in evs[:3]]) for evs in ev_k]
    arr_b = [(ctypes.c_void_p * (nk - 3))(*[e.cuda_event for e in evs[3:]]) for evs in ev_k]

    def step_profiled(i):
        ev_start[i].record(stream)
        binding.bdscan_profile_events(arr_f[i], 3)
        lay.forward(stream)
        nf = binding.bdscan_last_launch_count()
        binding.bdscan_profile_events(arr_b[i], nk - 3)
        lay.backward(stream, use_dstates=False)
        nb_ = binding.bdscan_last_launch_count()
        binding.bdscan_profile_events(None, 0)
        return nf + nb_

    bus = ""
    try:
        bus = torch.cuda.get_device_properties(dev).pci_bus_id
    except Exception:
        pass
    rows, stop = [], threading.Event()
    sampler = threading.Thread(target=sample_clocks, args=(stop, rows, bus), daemon=True)
    if rank == 0:
        sampler.start()

    # warm-up: at least W steps and about a second under load
    t_w = time.time()
    i = 0
    while i < args.warmup or time.time() - t_w < args.warmup_seconds:
        step()
        i += 1
        if i % 50 == 0:
            torch.cuda.synchronize(dev)
    torch.cuda.synchronize(dev)
    launches_per_step = 0

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_start_wall = time.time()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(args.steps):
        launches_per_step = step_profiled(i)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    t_end_wall = time.time()
    ms = e0.elapsed_time(e1)
    if launches_per_step != nk:
        raise RuntimeError(f"expected {nk} kernel launches per step, the library reported {launches_per_step}")

    # per-kernel average durations (event after kernel i minus event after kernel i-1)
    per = [[] for _ in range(nk)]
    for i in range(args.steps):
        prev = ev_start[i]
        for j in range(nk):
            per[j].append(prev.elapsed_time(ev_k[i][j]))
            prev = ev_k[i][j]
    avg_us = [1e3 * statistics.mean(p) for p in per]

    ms = max_over_ranks(ms, dev, world)

    # end-to-end through the public API with host buffers
    e2e = run_e2e(lay, wl, stream, dev, args)
    e2e["ms"] = max_over_ranks(e2e["ms"], dev, world)
    e2e_full = run_e2e(lay, wl, stream, dev, args, full_readback=True)
    e2e_full["ms"] = max_over_ranks(e2e_full["ms"], dev, world)
    stop.set()

    if rank != 0:
        return
    sampler.join(timeout=3)
    clocks = summarize_clocks(rows, t_start_wall, t_end_wall)
    ms_step = ms / args.steps
    value = job_tokens_per_s(Bt * L, world, ms_step)
    peaks, peak_kind = measured_peaks()
    fb, bb = algorithmic_bytes(Bt, L, D, N, Bs)
    kb = kernel_bytes(Bt, L, D, N, Bs)
    total_us = sum(avg_us)
    kernels = [{"name": k, "avg_us": round(u, 2), "share": round(u / total_us, 4),
                "alg_bytes": kb[k], "alg_gbs": round(kb[k] / (u * 1e3), 1) if u > 0 else None}
               for k, u in zip(KERNELS, avg_us)]
    dom = max(range(nk), key=lambda j: avg_us[j])
    dname = KERNELS[dom]
    elems = Bt * L * D * N
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    fp32_peak_tflops = 152 * 128 * 2 * sm_max * 1e6 / 1e12
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    dom_flops = kernel_flops_per_elem(dname) * elems
    dom_gbs = kb[dname] / (avg_us[dom] * 1e-6) / 1e9
    # the dominant kernel against the FP32 ALU roofline that binds it, with its
    # algorithmic-byte HBM fraction beside it
    roofline = {"bound": "alu", "kernel": dname,
                "achieved": round(dom_flops / (avg_us[dom] * 1e-6) / 1e12, 2),
                "peak": round(fp32_peak_tflops, 1), "unit": "TFLOP/s",
                "frac": round(dom_flops / (avg_us[dom] * 1e-6) / 1e12 / fp32_peak_tflops, 4),
                "traffic": (None if MEASURED_TRAFFIC_BATCH4.get(dname) is None
                            else int(MEASURED_TRAFFIC_BATCH4[dname] * Bt / 4)),
                "peak_kind": "derived: 152 SMs x 128 FP32 lanes x 2 flop/FMA x max SM clock",
                "flops_per_launch": dom_flops,
                "flops_per_elem": {"passes": KERNEL_PASSES.get(dname, []), "total": kernel_flops_per_elem(dname)},
                "hbm": {"achieved": round(dom_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                        "frac": round(dom_gbs / hbm_peak, 4), "alg_bytes_per_launch": kb[dname],
                        "peak_kind": peak_kind}}
    hbm = {"bound": "hbm", "achieved": round((fb + bb) / (ms_step * 1e-3) / 1e9, 1),
           "peak": peaks.get("hbm_gbs"), "unit": "GB/s",
           "frac": round((fb + bb) / (ms_step * 1e-3) / 1e9 / hbm_peak, 4),
           "frac_of_8tbs": round((fb + bb) / (ms_step * 1e-3) / 8e12, 4),
           "alg_bytes_per_step": fb + bb, "peak_kind": peak_kind,
           "dominant_kernel_gbs": round(dom_gbs, 1)}

    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        secs, th = oracle_run(CFG["d_inner"])
        cpu = {"value": Bt * L / secs, "unit": "tokens/s", "cores": th, "kind": "oracle",
               "sample": "fp64 oracle fwd+bwd of one full step of the same configuration (seed 0), "
                         f"{th} OpenMP threads (the backward uses one per batch row)", "seconds": round(secs, 2)}

    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32 state, bf16 I/O", "data": "synthetic",
            "config": {"workload": WORKLOAD, **CFG, "parallelism": "replicas" if world > 1 else "single",
                       "l2": "inputs larger than L2 (about 0.36 GB of token tensors per step; no flush)"},
            "roofline": roofline, "hbm": hbm, "cpu_baseline": cpu,
            "e2e": {"value": job_tokens_per_s(Bt * L, world, e2e["ms"]), "unit": "tokens/s",
                    "h2d_bytes_per_step": e2e["h2d"], "d2h_bytes_per_step": e2e["d2h"],
                    "readback": "the step's result: the parameter gradients (dA, dD of both directions)"},
            "e2e_full_readback": {"value": job_tokens_per_s(Bt * L, world, e2e_full["ms"]), "unit": "tokens/s",
                                  "h2d_bytes_per_step": e2e_full["h2d"], "d2h_bytes_per_step": e2e_full["d2h"],
                                  "readback": "every output and every gradient (y_c, y_n and all 15 gradients)"},
            "gpu_launches": launches_per_step * args.steps, "clocks": clocks, "kernels": kernels}
    print(json.dumps(line), flush=True)


def time_layer_steps(lay, stream, steps, warmup):
    """Average ms of one forward+backward step and per-kernel averages (us)."""
    import torch
    from paper_2607_02805_gb300 import binding
    nk = len(KERNELS)
    for _ in range(warmup):
        lay.forward(stream)
        lay.backward(stream, use_dstates=False)
    ev_s = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ev_k = [[torch.cuda.Event(enable_timing=True) for _ in range(nk)] for _ in range(steps)]
    for evs in ev_k:
        for e in evs:
            e.record(stream)
    torch.cuda.synchronize()
    arr_f = [(ctypes.c_void_p * 3)(*[e.cuda_event for e in evs[:3]]) for evs in ev_k]
    arr_b = [(ctypes.c_void_p * (nk - 3))(*[e.cuda_event for e in evs[3:]]) for evs in ev_k]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        ev_s[i].record(stream)
        binding.bdscan_profile_events(arr_f[i], 3)
        lay.forward(stream)
        binding.bdscan_profile_events(arr_b[i], nk - 3)
        lay.backward(stream, use_dstates=False)
        binding.bdscan_profile_events(None, 0)
    e1.record(stream)
    torch.cuda.synchronize()
    per = [[] for _ in range(nk)]
    for i in range(steps):
        prev = ev_s[i]
        for j in range(nk):
            per[j].append(prev.elapsed_time(ev_k[i][j]))
            prev = ev_k[i][j]
    return e0.elapsed_time(e1) / steps, {k: round(1e3 * statistics.mean(v), 2) for k, v in zip(KERNELS, per)}


def run_sweep(args):
    """Forward+backward at batch 8, 2048 tokens, d_inner 2048, d_state 16 for
    each block size (the 350M-scale layer), one line per block size."""
    import torch
    from paper_2607_02805_gb300.inputs import Workload
    from paper_2607_02805_gb300.layer import Layer
    peaks, peak_kind = measured_peaks()
    Bt, L, D, N = 8, 2048, 2048, 16
    for Bs in (4, 8, 16, 32, 64):
        wl = Workload(Bt, L, Bs, D, N, dtype="bf16", seed=1, with_grads=True)
        lay = Layer(wl)
        lay.alloc_backward()
        stream = torch.cuda.current_stream()
        ms, kern = time_layer_steps(lay, stream, args.steps, max(3, args.warmup))
        fb, bb = algorithmic_bytes(Bt, L, D, N, Bs)
        gbs = (fb + bb) / (ms * 1e-3) / 1e9
        print(json.dumps({
            "metric": METRIC, "value": Bt * L / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": args.steps,
            "ms_per_step": ms, "higher_is_better": True, "dtype": "f32 state, bf16 I/O", "data": "synthetic",
            "config": {"workload": f"350M-scale layer block sweep: batch 8, 2048 tokens per stream, block {Bs}, "
                                   "d_inner 2048, d_state 16; all-block forward + backward",
                       "batch": Bt, "seq_len": L, "block": Bs, "d_inner": D, "d_state": N},
            "hbm": {"achieved": round(gbs, 1), "peak": peaks.get("hbm_gbs"), "unit": "GB/s",
                    "frac": round(gbs / float(peaks.get("hbm_gbs", 6800.0)), 4), "alg_bytes_per_step": fb + bb,
                    "peak_kind": peak_kind},
            "kernels_us": kern}), flush=True)
        del lay
        torch.cuda.empty_cache()


SSD_KERNELS = ("ssd_block_state", "ssd_state_pass", "ssd_scan_clean", "ssd_scan_noisy")


def ssd_costs(Bt, L, Bs, H, N, hg):
    """Algorithmic HBM bytes and tensor-core flops of each SSD forward kernel.
    Bytes: every tensor a kernel must touch, once (x, dt, B, C of its streams,
    the states it writes or reads as seeds, its outputs). Flops: the MMAs the
    kernels issue, counting the high and low bf16 parts of split operands."""
    P, nb, m = 64, L // Bs, Bs // 128
    tok = Bt * L
    x, dt, bc = tok * H * P * 2, tok * H * 2, tok * N * 2
    st = Bt * nb * H * P * N * 4
    sd = Bt * nb * H * 4
    groups = -(-H // hg)
    b = {"ssd_block_state": x + dt + bc + st + sd,
         "ssd_state_pass": 2 * st + sd,
         "ssd_scan_clean": x + dt + 2 * bc + st + x,
         "ssd_scan_noisy": x + 2 * dt + 4 * bc + st + x}
    tiles = Bt * nb * m
    gram_c = sum(i + 1 for i in range(m))       # Gram products per block, clean
    gram_n = m * (m + 1)                        # forward + reverse per block
    mix_c = gram_c                              # mixing tiles per head and block
    mix_n = m * m
    f = {"ssd_block_state": Bt * nb * H * 2 * (2.0 * 128 * P * Bs),
         "ssd_state_pass": 0.0,
         "ssd_scan_clean": Bt * nb * (groups * gram_c * 2.0 * 128 * 128 * N + H * (mix_c * 2.0 * 128 * 128 * P)
                                      + H * m * 2 * 2.0 * 128 * P * N),
         "ssd_scan_noisy": Bt * nb * (groups * gram_n * 2.0 * 128 * 128 * N + H * (mix_n * 2.0 * 128 * 128 * P)
                                      + H * m * 2 * 2.0 * 128 * P * N)}
    del tiles
    return b, f


def run_ssd(args):
    """Forward of the SSD (Mamba-2) form at the paper's two model sizes, one
    line each: clean scan with every block-end state, noisy blocks (seeded
    forward + block-local reverse), through bdscan_ssd_forward."""
    import torch
    from paper_2607_02805_gb300 import binding
    from paper_2607_02805_gb300.inputs import SsdWorkload
    from paper_2607_02805_gb300.layer import to_device
    peaks, peak_kind = measured_peaks()
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    tc_peak = float(peaks.get("bf16_tflops", 1900.0))
    for name, (Bt, L, Bs, H, N) in (("350M-class Mamba-2 layer: 26 heads of 64, state 128", (8, 8192, 256, 26, 128)),
                                   ("87M-class Mamba-2 layer: 14 heads of 64, state 64", (8, 8192, 256, 14, 64))):
        if args.batch:
            Bt = args.batch
        wl = SsdWorkload(Bt, L, Bs, H, N, seed=0)
        t = {k: to_device(wl.dev_bits(k), binding.BDSCAN_F32 if k in ("A_f", "A_r", "D_f", "D_r")
                          else binding.BDSCAN_BF16, "cuda") for k in wl.t32}
        d = binding.make_ssd_dims(Bt, L, Bs, H, N)
        y_c = torch.empty((Bt, L, H, 64), dtype=torch.bfloat16, device="cuda")
        y_n = torch.empty_like(y_c)
        st = torch.empty((Bt, L // Bs, H, 64, N), dtype=torch.float32, device="cuda")
        ws = torch.empty(binding.bdscan_ssd_forward_workspace_size(d), dtype=torch.uint8, device="cuda")
        stream = torch.cuda.current_stream()
        for _ in range(max(3, args.warmup)):
            binding.ssd_forward(d, t, y_c, y_n, st, ws)
        nk = len(SSD_KERNELS)
        steps = max(1, args.steps)
        ev_s = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
        ev_k = [[torch.cuda.Event(enable_timing=True) for _ in range(nk)] for _ in range(steps)]
        for evs in ev_k:
            for e in evs:
                e.record(stream)
        torch.cuda.synchronize()
        arr = [(ctypes.c_void_p * nk)(*[e.cuda_event for e in evs]) for evs in ev_k]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(steps):
            ev_s[i].record(stream)
            binding.bdscan_profile_events(arr[i], nk)
            binding.ssd_forward(d, t, y_c, y_n, st, ws)
            binding.bdscan_profile_events(None, 0)
        e1.record(stream)
        torch.cuda.synchronize()
        flag = binding.bdscan_ssd_wait_flag(1)
        ms = e0.elapsed_time(e1) / steps
        per = {k: [] for k in SSD_KERNELS}
        for i in range(steps):
            prev = ev_s[i]
            for j, k in enumerate(SSD_KERNELS):
                per[k].append(prev.elapsed_time(ev_k[i][j]))
                prev = ev_k[i][j]
        hg = -(-H // -(-H // 16))  # heads per block-scan CTA at these sizes (grids above the SM count)
        bts, fls = ssd_costs(Bt, L, Bs, H, N, hg)
        kern = []
        for k in SSD_KERNELS:
            us = 1e3 * statistics.mean(per[k])
            kern.append({"name": k, "avg_us": round(us, 2), "alg_bytes": bts[k],
                         "alg_gbs": round(bts[k] / (us * 1e-6) / 1e9, 1),
                         "tflops": round(fls[k] / (us * 1e-6) / 1e12, 1)})
        tot_b = sum(bts.values())
        dom = max(kern, key=lambda r: r["avg_us"])
        print(json.dumps({
            "metric": "SSD-form block-bidirectional forward tokens/s (clean + noisy stream pair counts once)",
            "value": Bt * L / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": steps, "ms_per_step": ms,
            "higher_is_better": True, "dtype": "bf16 operands, fp32 accumulate and state", "data": "synthetic",
            "config": {"workload": f"{name}; batch {Bt}, {L} tokens per stream, block {Bs}; forward with every "
                                   "block-end state", "batch": Bt, "seq_len": L, "block": Bs, "heads": H,
                       "head_dim": 64, "d_state": N},
            "hbm": {"achieved": round(tot_b / (ms * 1e-3) / 1e9, 1), "peak": hbm_peak, "unit": "GB/s",
                    "frac": round(tot_b / (ms * 1e-3) / 1e9 / hbm_peak, 4), "alg_bytes_per_step": tot_b,
                    "peak_kind": peak_kind},
            "dominant": {"name": dom["name"], "hbm_frac": round(dom["alg_gbs"] / hbm_peak, 4),
                         "tensor_frac": round(dom["tflops"] / tc_peak, 4)},
            "wait_flag": flag, "kernels": kern}), flush=True)
        del t, y_c, y_n, st, ws
        torch.cuda.empty_cache()


SSD_BWD_KERNELS = ("bwd_tile_clean", "bwd_tile_fwd", "bwd_tile_rev", "bwd_vec_clean", "bwd_vec_fwd", "bwd_vec_rev",
                   "bwd_state_pass", "bwd_block_state", "bwd_dx", "bwd_dbc", "bwd_par")


def ssd_bwd_head_groups(Bt, L, Bs, H):
    """Heads per tile CTA and the number of head groups the backward picks
    (about 1024 CTAs per launch, at most 16 heads per CTA)."""
    units = Bt * (L // Bs) * (Bs // 128)
    want = -(-1024 // units) if units > 0 else 1
    want = min(max(want, -(-H // 16)), H)
    want = max(want, 1)
    hg = -(-H // want)
    return hg, -(-H // hg)


def ssd_bwd_tile_flops(Bt, L, Bs, H, N, seeded):
    """Tensor-core flops one backward tile launch (one stream and direction)
    issues. Per block and (tile i, s-tile j) pair the direction reaches: per
    head group G = C B^T (K = N) and, with the head-summed dG split into bf16
    high and low parts, dC += dG B and dB = dG^T C (K = 128, twice each); per
    head Q = dy x^T (K = 64) and D = M'^T dy (K = 128) with M' split into its
    two bf16 parts (dx and the column sums come from D). Per head and tile of a
    seeded block after the first: (E dy) S (K = 64) and C S^T (K = N) with the
    seed's two parts, and C^T (E dy) (K = 128, C padded to 128 rows)."""
    m, nb = Bs // 128, L // Bs
    _, ngrp = ssd_bwd_head_groups(Bt, L, Bs, H)
    pairs = m * (m + 1) // 2
    per_pair = ngrp * (2.0 * 128 * 128 * N + 2 * 2 * (2.0 * 128 * N * 128)) + H * 3 * (2.0 * 128 * 128 * 64)
    f = Bt * nb * pairs * per_pair
    if seeded:
        f += Bt * (nb - 1) * m * H * (2 * (2.0 * 128 * N * 64) + 2 * (2.0 * 128 * 64 * N) + 2.0 * 128 * 64 * 128)
    return f


def run_ssd_train(args):
    """Forward + backward of the SSD (Mamba-2) form at the paper's two model
    sizes (training length 8192, block 256), one line each."""
    import torch
    from paper_2607_02805_gb300 import binding
    from paper_2607_02805_gb300.inputs import SsdWorkload
    from paper_2607_02805_gb300.layer import to_device
    peaks, peak_kind = measured_peaks()
    tc_peak = float(peaks.get("bf16_tflops", 1900.0))
    hbm_peak = float(peaks.get("hbm_gbs", 6800.0))
    for name, (Bt, L, Bs, H, N) in (("350M-class Mamba-2 layer: 26 heads of 64, state 128", (8, 8192, 256, 26, 128)),
                                   ("87M-class Mamba-2 layer: 14 heads of 64, state 64", (8, 8192, 256, 14, 64))):
        if args.batch:
            Bt = args.batch
        wl = SsdWorkload(Bt, L, Bs, H, N, seed=0, with_grads=True)
        t = {k: to_device(wl.dev_bits(k), binding.BDSCAN_F32 if k in ("A_f", "A_r", "D_f", "D_r")
                          else binding.BDSCAN_BF16, "cuda") for k in wl.t32}
        d = binding.make_ssd_dims(Bt, L, Bs, H, N)
        y_c = torch.empty((Bt, L, H, 64), dtype=torch.bfloat16, device="cuda")
        y_n = torch.empty_like(y_c)
        st = torch.empty((Bt, L // Bs, H, 64, N), dtype=torch.float32, device="cuda")
        wsf = torch.empty(binding.bdscan_ssd_forward_workspace_size(d), dtype=torch.uint8, device="cuda")
        wsb = torch.empty(binding.bdscan_ssd_backward_workspace_size(d), dtype=torch.uint8, device="cuda")
        names = ("x_c", "dt_c", "B_c", "C_c", "x_n", "dt_f", "B_f", "C_f", "dt_r", "B_r", "C_r", "A_f", "D_f", "A_r",
                 "D_r")
        g = {k: torch.empty(t[k].shape, dtype=torch.float32 if k in ("A_f", "A_r", "D_f", "D_r") else torch.bfloat16,
                            device="cuda") for k in names}
        stream = torch.cuda.current_stream()

        def step():
            binding.ssd_forward(d, t, y_c, y_n, st, wsf)
            binding.ssd_backward(d, t, st, t["dy_c"], t["dy_n"], None, g, wsb)

        for _ in range(max(3, args.warmup)):
            step()
        steps = max(3, min(args.steps, 20))
        nf, nb_ = len(SSD_KERNELS), len(SSD_BWD_KERNELS)
        ev_s = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
        ev_k = [[torch.cuda.Event(enable_timing=True) for _ in range(nf + nb_)] for _ in range(steps)]
        for evs in ev_k:
            for e in evs:
                e.record(stream)
        torch.cuda.synchronize()
        arr_f = [(ctypes.c_void_p * nf)(*[e.cuda_event for e in evs[:nf]]) for evs in ev_k]
        arr_b = [(ctypes.c_void_p * nb_)(*[e.cuda_event for e in evs[nf:]]) for evs in ev_k]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        launches = 0
        for i in range(steps):
            ev_s[i].record(stream)
            binding.bdscan_profile_events(arr_f[i], nf)
            binding.ssd_forward(d, t, y_c, y_n, st, wsf)
            launches = binding.bdscan_last_launch_count()
            binding.bdscan_profile_events(arr_b[i], nb_)
            binding.ssd_backward(d, t, st, t["dy_c"], t["dy_n"], None, g, wsb)
            launches += binding.bdscan_last_launch_count()
            binding.bdscan_profile_events(None, 0)
        e1.record(stream)
        torch.cuda.synchronize()
        flag = binding.bdscan_ssd_wait_flag(1)
        ms = e0.elapsed_time(e1) / steps
        allk = SSD_KERNELS + SSD_BWD_KERNELS
        per = {k: [] for k in allk}
        for i in range(steps):
            prev = ev_s[i]
            for j, k in enumerate(allk):
                per[k].append(prev.elapsed_time(ev_k[i][j]))
                prev = ev_k[i][j]
        kern = []
        for k in allk:
            us = 1e3 * statistics.mean(per[k])
            row = {"name": k, "avg_us": round(us, 2)}
            if k.startswith("bwd_tile"):
                fl = ssd_bwd_tile_flops(Bt, L, Bs, H, N, seeded=k != "bwd_tile_rev")
                row["tflops"] = round(fl / (us * 1e-6) / 1e12, 1)
                row["tensor_frac"] = round(fl / (us * 1e-6) / 1e12 / tc_peak, 4)
            kern.append(row)
        fwd_ms = sum(r["avg_us"] for r in kern[:nf]) / 1e3
        bwd_ms = sum(r["avg_us"] for r in kern[nf:]) / 1e3
        dom = max(kern, key=lambda r: r["avg_us"])
        print(json.dumps({
            "metric": "SSD-form block-bidirectional forward+backward tokens/s (clean + noisy stream pair counts once)",
            "value": Bt * L / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": steps, "ms_per_step": ms,
            "higher_is_better": True, "dtype": "bf16 operands, fp32 accumulate and state", "data": "synthetic",
            "config": {"workload": f"{name}; batch {Bt}, {L} tokens per stream, block {Bs}; forward with every "
                                   "block-end state, then the backward of every input", "batch": Bt, "seq_len": L,
                       "block": Bs, "heads": H, "head_dim": 64, "d_state": N},
            "forward_ms": round(fwd_ms, 4), "backward_ms": round(bwd_ms, 4),
            "dominant": {"name": dom["name"], "avg_us": dom["avg_us"], "tensor_frac": dom.get("tensor_frac")},
            "tensor_peak_tflops": tc_peak, "hbm_peak_gbs": hbm_peak, "peak_kind": peak_kind,
            "gpu_launches": launches * steps, "wait_flag": flag, "kernels": kern}), flush=True)
        del t, y_c, y_n, st, wsf, wsb, g
        torch.cuda.empty_cache()


def run_ssd_cache(args, L=65536, Bs=256, calls=16):
    """Inference cache path of the SSD form (350M-class Mamba-2 layer, 26 heads
    of 64, state 128, batch 1): cache build over an L-token prefix (final state
    only; every block-end state and the clean outputs), then `calls`
    active-block calls from the cached state, each timed on its own and all
    replayed as one CUDA graph."""
    import torch
    from paper_2607_02805_gb300 import binding
    from paper_2607_02805_gb300.inputs import SsdWorkload
    from paper_2607_02805_gb300.layer import to_device
    peaks, peak_kind = measured_peaks()
    H, N = 26, 128
    wl = SsdWorkload(1, L, Bs, H, N, seed=7)
    t = {k: to_device(wl.dev_bits(k), binding.BDSCAN_F32 if k in ("A_f", "A_r", "D_f", "D_r")
                      else binding.BDSCAN_BF16, "cuda") for k in wl.t32}
    d = binding.make_ssd_dims(1, L, Bs, H, N)
    stream = torch.cuda.current_stream()
    nb = L // Bs
    fin = torch.empty((1, 1, H, 64, N), dtype=torch.float32, device="cuda")
    allst = torch.empty((1, nb, H, 64, N), dtype=torch.float32, device="cuda")
    y_c = torch.empty((1, L, H, 64), dtype=torch.bfloat16, device="cuda")
    ws = {e: torch.empty(binding.bdscan_ssd_boundary_states_workspace_size(d, e), dtype=torch.uint8, device="cuda")
          for e in (0, 1)}
    read_b = L * (H * 64 * 2 + H * 2 + N * 2)  # x, dt, B
    st_b = nb * H * 64 * N * 4
    for name, emit_all, y, st, alg in (("final state only", 0, None, fin, read_b + 2 * st_b),
                                       ("every block-end state and the clean outputs", 1, y_c, allst,
                                        read_b + L * N * 2 + 3 * st_b + L * H * 64 * 4)):
        def one():
            binding.ssd_boundary_states(d, t, None, y, st, emit_all, ws[emit_all], stream)
        for _ in range(max(3, args.warmup)):
            one()
        reps = max(3, min(args.steps, 20))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            one()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        gbs = alg / (ms * 1e-3) / 1e9
        print(json.dumps({
            "metric": "SSD-form cache build (bdscan_ssd_boundary_states) prefix tokens/s", "value": L / (ms * 1e-3),
            "unit": "tokens/s", "n_gpus": 1, "steps": reps, "ms_per_call": ms, "higher_is_better": True,
            "dtype": "bf16 operands, fp32 accumulate and state", "data": "synthetic",
            "config": {"workload": f"SSD cache build over a {L}-token prefix, block {Bs}, 26 heads of 64, state 128, "
                                   f"batch 1; {name}", "seq_len": L, "block": Bs, "emit_all": emit_all},
            "hbm": {"achieved": round(gbs, 1), "peak": peaks.get("hbm_gbs"), "unit": "GB/s",
                    "frac": round(gbs / float(peaks.get("hbm_gbs", 6800.0)), 4), "alg_bytes_per_call": alg,
                    "peak_kind": peak_kind}}), flush=True)
    # active blocks: fresh noisy draws per call, seeded from the cached final state
    da = binding.make_ssd_dims(1, Bs, Bs, H, N)
    blocks = []
    for c in range(calls):
        nw = SsdWorkload(1, Bs, Bs, H, N, seed=7, part=c + 1)
        blocks.append({k: to_device(nw.dev_bits(k), binding.BDSCAN_F32 if k in ("A_f", "A_r", "D_f", "D_r")
                                    else binding.BDSCAN_BF16, "cuda") for k in nw.t32})
    ya = torch.empty((1, Bs, H, 64), dtype=torch.bfloat16, device="cuda")
    seed = fin[:, 0].contiguous()
    for _ in range(max(3, args.warmup)):
        binding.ssd_active_block(da, seed, blocks[0], ya, stream)
    per = []
    for c in range(calls):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        binding.ssd_active_block(da, seed, blocks[c], ya, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        per.append(e0.elapsed_time(e1) * 1e3)
    gs = torch.cuda.Stream()
    gs.wait_stream(stream)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(gs):
        binding.ssd_active_block(da, seed, blocks[0], ya, gs)
        torch.cuda.synchronize()
        with torch.cuda.graph(graph, stream=gs):
            for c in range(calls):
                binding.ssd_active_block(da, seed, blocks[c], ya, gs)
    torch.cuda.synchronize()
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 20
    e0.record(stream)
    for _ in range(reps):
        graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    graph_us = e0.elapsed_time(e1) * 1e3 / (reps * calls)
    # the same denoising step without a cache: a full-sequence bidirectional
    # layer over the whole context (both directions rescan all L tokens)
    yf = torch.empty((1, L, H, 64), dtype=torch.bfloat16, device="cuda")
    wsf = torch.empty(binding.bdscan_ssd_full_bidir_workspace_size(d), dtype=torch.uint8, device="cuda")
    for _ in range(max(3, args.warmup)):
        binding.ssd_full_bidir_forward(d, t, yf, wsf, stream)
    reps_f = max(3, min(args.steps, 10))
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    f0.record(stream)
    for _ in range(reps_f):
        binding.ssd_full_bidir_forward(d, t, yf, wsf, stream)
    f1.record(stream)
    torch.cuda.synchronize()
    full_ms = f0.elapsed_time(f1) / reps_f
    flag = binding.bdscan_ssd_wait_flag(1)
    print(json.dumps({
        "metric": "SSD-form layer step per denoising step: full-sequence bidirectional (no cache) over cached "
                  "active block", "value": full_ms * 1e3 / graph_us, "unit": "x", "n_gpus": 1,
        "higher_is_better": True, "dtype": "bf16 operands, fp32 accumulate and state", "data": "synthetic",
        "config": {"workload": f"one 350M-class Mamba-2 layer at a {L}-token context, block {Bs}, batch 1: "
                               "bdscan_ssd_full_bidir_forward over the whole sequence vs bdscan_ssd_active_block "
                               "from the cached state (in a CUDA graph)", "context": L, "block": Bs},
        "full_bidir_ms": round(full_ms, 4), "active_block_us": round(graph_us, 3), "wait_flag": flag}), flush=True)
    print(json.dumps({
        "metric": "SSD-form active-block call latency (bdscan_ssd_active_block)", "value": statistics.median(per),
        "unit": "us per call", "n_gpus": 1, "higher_is_better": False,
        "dtype": "bf16 operands, fp32 accumulate and state", "data": "synthetic",
        "config": {"workload": f"active block of {Bs} tokens from the cached state of a {L}-token prefix, 26 heads of "
                               "64, state 128, batch 1", "calls": calls},
        "per_call_us": [round(v, 2) for v in per],
        "graph_replay_us_per_call": graph_us, "wait_flag": flag}), flush=True)


def run_mixer(args):
    """The mixer around the scan (conv1d of width 4 with SiLU, softplus step
    size, SiLU gate) at the benchmark layer's geometry: all-block forward then
    the backward of every input, against the bare scan's forward + backward on
    the same sizes."""
    import torch
    from paper_2607_02805_gb300 import binding
    from paper_2607_02805_gb300.inputs import MixerWorkload, Workload
    from paper_2607_02805_gb300.layer import Layer, to_device
    Bt, L, Bs, D, N = (args.batch or 8), 2048, 16, 1536, 16
    code = binding.BDSCAN_BF16
    wl = MixerWorkload(Bt, L, Bs, D, N, dtype="bf16", seed=0)
    t = {k: to_device(wl.dev_bits(k), code, "cuda") for k in wl.t32}
    dims = binding.make_dims(Bt, L, Bs, D, N, code)
    out_c = torch.empty((Bt, L, D), dtype=torch.bfloat16, device="cuda")
    out_n = torch.empty_like(out_c)
    st = torch.empty((Bt, L // Bs, D, N), dtype=torch.float32, device="cuda")
    wsf = torch.empty(binding.bdscan_mixer_forward_workspace_size(dims), dtype=torch.uint8, device="cuda")
    wsb = torch.empty(binding.bdscan_mixer_backward_workspace_size(dims), dtype=torch.uint8, device="cuda")
    per_ch = ("A_f", "D_f", "A_r", "D_r", "conv_w", "conv_b", "dt_bias_f", "dt_bias_r")
    g = {k: torch.empty(v.shape, dtype=torch.float32 if k in per_ch else torch.bfloat16, device="cuda")
         for k, v in t.items() if k not in ("dy_c", "dy_n")}
    stream = torch.cuda.current_stream()

    def step_mixer():
        binding.mixer_forward(dims, t, out_c, out_n, st, wsf, stream)
        binding.mixer_backward(dims, t, t["dy_c"], t["dy_n"], None, g, wsb, stream)

    lay = Layer(Workload(Bt, L, Bs, D, N, dtype="bf16", seed=0, with_grads=True), device="cuda")
    lay.alloc_backward()

    def step_scan():
        lay.forward(stream)
        lay.backward(stream, use_dstates=False)

    res = {}
    for name, fn in (("mixer", step_mixer), ("scan", step_scan)):
        for _ in range(max(3, args.warmup)):
            fn()
        reps = max(3, min(args.steps, 50))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        res[name] = e0.elapsed_time(e1) / reps
    # per-launch times of one forward and one backward (the events hook records
    # an event after each launch)
    per_launch = {}
    for name, fn in (("forward", lambda: binding.mixer_forward(dims, t, out_c, out_n, st, wsf, stream)),
                     ("backward", lambda: binding.mixer_backward(dims, t, t["dy_c"], t["dy_n"], None, g, wsb,
                                                                 stream))):
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(33)]
        for e in evs:
            e.record(stream)
        torch.cuda.synchronize()
        arr = (ctypes.c_void_p * 32)(*[e.cuda_event for e in evs[1:]])
        evs[0].record(stream)
        binding.bdscan_profile_events(arr, 32)
        fn()
        n = binding.bdscan_last_launch_count()
        binding.bdscan_profile_events(None, 0)
        torch.cuda.synchronize()
        per_launch[name] = [round(1e3 * evs[j].elapsed_time(evs[j + 1]), 1) for j in range(min(n, 32))]
    print(json.dumps({
        "metric": "mixer (conv1d + softplus + gate around the block-bidirectional scan) forward+backward tokens/s",
        "value": Bt * L / (res["mixer"] * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": reps,
        "ms_per_step": res["mixer"], "higher_is_better": True, "dtype": "bf16 I/O, fp32 scan inputs and state",
        "data": "synthetic",
        "config": {"workload": f"87M-scale layer geometry with the mixer around the scan: batch {Bt}, {L} tokens "
                               f"per stream, block {Bs}, d_inner {D}, d_state {N}; all-block forward then the "
                               "backward of every input", "batch": Bt, "seq_len": L, "block": Bs, "d_inner": D,
                   "d_state": N},
        "scan_only_ms_per_step": round(res["scan"], 4),
        "mixer_overhead_ms": round(res["mixer"] - res["scan"], 4),
        "launch_us": per_launch}), flush=True)


def run_prefill(args, L, Bs, calls):
    """Inference cache path at d_inner 2048, d_state 16, batch 1: the cache
    build over an L-token clean prefix (final state only, and every block-end
    state plus the clean outputs), then `calls` active-block calls from the
    cached state, each timed on its own and all replayed as one CUDA graph,
    against the same layer step without a cache (a full-sequence
    bidirectional scan over the L tokens, as a DiffuMamba sampler must run
    at every denoising step)."""
    import torch
    from paper_2607_02805_gb300 import binding
    from paper_2607_02805_gb300.inputs import Workload
    from paper_2607_02805_gb300.layer import to_device
    peaks, peak_kind = measured_peaks()
    D, N = 2048, 16
    code = binding.BDSCAN_BF16
    wl = Workload(1, L, Bs, D, N, dtype="bf16", seed=5, with_grads=False, parts=("clean",))
    t = {k: to_device(wl.dev_bits(k), code, "cuda") for k in wl.t32}
    dims = binding.make_dims(1, L, Bs, D, N, code)
    stream = torch.cuda.current_stream()
    nb = L // Bs
    fin = torch.empty((1, 1, D, N), dtype=torch.float32, device="cuda")
    allst = torch.empty((1, nb, D, N), dtype=torch.float32, device="cuda")
    y_c = torch.empty((1, L, D), dtype=torch.bfloat16, device="cuda")
    ws = {}
    for emit_all in (0, 1):
        nbytes = binding.bdscan_boundary_states_workspace_size(dims, emit_all)
        ws[emit_all] = torch.empty(max(1, (nbytes + 3) // 4), dtype=torch.float32, device="cuda")
    read_b = L * (2 * D * 2 + 2 * N * 2)  # x, dt [L, D] and B, C [L, N], bf16
    modes = [("final state only", 0, None, fin, 0),
             ("every block-end state and the clean outputs", 1, y_c, allst, nb * D * N * 4 + L * D * 2)]
    for name, emit_all, y, st, extra_b in modes:
        def one():
            binding.boundary_states(dims, t, None, y, st, emit_all, ws[emit_all], stream)
        for _ in range(max(3, args.warmup)):
            one()
        reps = max(3, min(args.steps, 20))
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(reps):
            one()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        gbs = (read_b + extra_b) / (ms * 1e-3) / 1e9
        print(json.dumps({
            "metric": "cache build (bdscan_boundary_states) prefix tokens/s", "value": L / (ms * 1e-3),
            "unit": "tokens/s", "n_gpus": 1, "steps": reps, "ms_per_call": ms, "higher_is_better": True,
            "dtype": "f32 state, bf16 I/O", "data": "synthetic",
            "config": {"workload": f"cache build over a {L}-token prefix, block {Bs}, d_inner 2048, d_state 16, "
                                   f"batch 1, bf16; emits {name}",
                       "batch": 1, "seq_len": L, "block": Bs, "d_inner": D, "d_state": N, "emit_all": emit_all},
            "hbm": {"achieved": round(gbs, 1), "peak": peaks.get("hbm_gbs"), "unit": "GB/s",
                    "frac": round(gbs / float(peaks.get("hbm_gbs", 6800.0)), 4),
                    "alg_bytes_per_call": read_b + extra_b, "peak_kind": peak_kind}}), flush=True)
    # active blocks from the cached final state (read-only seed)
    binding.boundary_states(dims, t, None, None, fin, 0, ws[0], stream)
    blocks = []
    for j in range(calls):
        blk = Workload(1, Bs, Bs, D, N, dtype="bf16", seed=5, with_grads=False, parts=("noisy",), part=j + 1)
        tb = {k: to_device(blk.dev_bits(k), code, "cuda") for k in blk.t32}
        blocks.append((tb, torch.empty((1, Bs, D), dtype=torch.bfloat16, device="cuda")))
    bdims = binding.make_dims(1, Bs, Bs, D, N, code)
    seed = fin[:, 0].contiguous()

    def call(j, s):
        binding.active_block(bdims, seed, blocks[j][0], blocks[j][1], s)

    for j in range(calls):
        call(j, stream)
    torch.cuda.synchronize()
    per_call = []
    for j in range(calls):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        call(j, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        per_call.append(1e3 * e0.elapsed_time(e1))
    graph_us = None
    try:
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        with torch.cuda.graph(g, stream=side):
            for j in range(calls):
                call(j, side)
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        reps = 20
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        graph_us = 1e3 * e0.elapsed_time(e1) / (reps * calls)
    except Exception as exc:  # report the failure in the line, keep the rest
        graph_us = f"capture failed: {exc}"
    # the same calls with AdaLN on the block (a fresh modulation per step),
    # replayed as one CUDA graph
    adaln_us = None
    try:
        from paper_2607_02805_gb300.inputs import draw
        mods = [{k: torch.from_numpy(draw(k, (1, D), 5, j + 1)).cuda() for k in ("shift", "scale", "gate")}
                for j in range(calls)]
        ws_ad = torch.empty(max(1, (binding.bdscan_active_block_adaln_workspace_size(bdims) + 3) // 4),
                            dtype=torch.float32, device="cuda")

        def call_ad(j, s):
            m = mods[j]
            binding.active_block_adaln(bdims, seed, blocks[j][0], m["shift"], m["scale"], m["gate"], 1e-5,
                                       blocks[j][1], ws_ad, s)

        for j in range(calls):
            call_ad(j, stream)
        torch.cuda.synchronize()
        g2 = torch.cuda.CUDAGraph()
        side2 = torch.cuda.Stream()
        side2.wait_stream(stream)
        with torch.cuda.graph(g2, stream=side2):
            for j in range(calls):
                call_ad(j, side2)
        torch.cuda.synchronize()
        g2.replay()
        torch.cuda.synchronize()
        reps = 20
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            g2.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        adaln_us = 1e3 * e0.elapsed_time(e1) / (reps * calls)
    except Exception as exc:
        adaln_us = f"capture failed: {exc}"
    # the same layer step without the cache: a full-sequence bidirectional
    # layer (DiffuMamba) rescans the whole sequence in both directions at every
    # denoising step, because its reverse states depend on the active block
    tf = {"x_n": t["x_c"], "dt_f": t["dt_c"], "B_f": t["B_c"], "C_f": t["C_c"], "dt_r": t["dt_c"],
          "B_r": t["B_c"], "C_r": t["C_c"], "A_f": t["A_f"], "D_f": t["D_f"], "A_r": t["A_f"], "D_r": t["D_f"]}
    y_full = torch.empty((1, L, D), dtype=torch.bfloat16, device="cuda")
    fbytes = binding.bdscan_full_bidir_workspace_size(dims)
    ws_full = torch.empty(max(1, (fbytes + 3) // 4), dtype=torch.float32, device="cuda")
    for _ in range(2):
        binding.full_bidir_forward(dims, tf, y_full, ws_full, stream)
    reps = 5
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        binding.full_bidir_forward(dims, tf, y_full, ws_full, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    full_ms = e0.elapsed_time(e1) / reps
    del ws_full, y_full
    blk_bytes = Bs * (D * 2 + 2 * D * 2 + 4 * N * 2 + D * 2) + D * N * 4
    graph_us_num = graph_us if isinstance(graph_us, float) else statistics.median(per_call)
    print(json.dumps({
        "metric": "layer step per denoising step: full-sequence bidirectional (no cache) over cached active block",
        "value": full_ms * 1e3 / graph_us_num, "unit": "x", "n_gpus": 1, "higher_is_better": True,
        "dtype": "f32 state, bf16 I/O", "data": "synthetic",
        "config": {"workload": f"one layer at a {L}-token context, block {Bs}, d_inner 2048, d_state 16, batch 1: "
                               "bdscan_full_bidir_forward over the whole sequence vs bdscan_active_block from "
                               "the cached state (in a CUDA graph)", "context": L, "block": Bs},
        "full_bidir_ms": round(full_ms, 4), "active_block_us": round(graph_us_num, 3)}), flush=True)
    print(json.dumps({
        "metric": "active-block call latency (bdscan_active_block)", "value": statistics.median(per_call),
        "unit": "us per call", "n_gpus": 1, "higher_is_better": False, "dtype": "f32 state, bf16 I/O",
        "data": "synthetic",
        "config": {"workload": f"active block of {Bs} tokens from the cached state of a {L}-token prefix, "
                               "d_inner 2048, d_state 16, batch 1, bf16", "calls": calls},
        "per_call_us": [round(u, 2) for u in per_call], "graph_replay_us_per_call": graph_us,
        "adaln_graph_replay_us_per_call": adaln_us, "bytes_per_call": blk_bytes}), flush=True)


def run_e2e(lay, wl, stream, dev, args, full_readback=False):
    """Forward + backward through the C ABI end to end: every step copies all
    of its inputs (both streams' x, dt, B, C and the upstream gradients) from
    pinned host memory to the device and reads the step's result back: the
    layer's parameter gradients (dA, dD of both directions), which is what a
    training step hands to its optimizer. The outputs and per-token gradients
    stay on the device, where the neighbouring layers consume them; with
    full_readback they are read back as well (y_c, y_n and every gradient),
    the host-to-host reading of the same step. Copies run
    on their own streams and two device buffer sets alternate, so that step
    i+1's inputs go up and step i-1's result comes down while step i computes.
    The timed region covers all copies of every step."""
    import torch
    from paper_2607_02805_gb300.layer import Layer
    lays = [lay, Layer(wl, device=dev)]
    lays[1].alloc_backward()
    ins = [k for k in wl.t32]
    host_in = {k: lay.t[k].detach().to("cpu").pin_memory() for k in ins}
    if full_readback:
        outs = [[la.y_c, la.y_n] + [la.g[k] for k in la.g] for la in lays]
    else:
        outs = [[la.g[k] for k in ("A_f", "D_f", "A_r", "D_r")] for la in lays]
    host_out = [[torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for o in outs[0]] for _ in range(2)]
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(t.numel() * t.element_size() for t in host_out[0])
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    steps = max(4, min(args.steps, 20))

    def run(n):
        ev_in = [torch.cuda.Event() for _ in range(n)]
        ev_comp = [torch.cuda.Event() for _ in range(n)]
        ev_out = [torch.cuda.Event() for _ in range(n)]
        for i in range(n):
            j = i % 2
            la = lays[j]
            if i >= 2:
                s_in.wait_event(ev_comp[i - 2])  # this buffer set's inputs are no longer read
            with torch.cuda.stream(s_in):
                for k in ins:
                    la.t[k].copy_(host_in[k], non_blocking=True)
            ev_in[i].record(s_in)
            stream.wait_event(ev_in[i])
            if i >= 2:
                stream.wait_event(ev_out[i - 2])  # its outputs have been read back
            la.forward(stream)
            la.backward(stream, use_dstates=False)
            ev_comp[i].record(stream)
            s_out.wait_event(ev_comp[i])
            with torch.cuda.stream(s_out):
                for o, h in zip(outs[j], host_out[j]):
                    h.copy_(o, non_blocking=True)
            ev_out[i].record(s_out)
        stream.wait_event(ev_out[n - 1])

    run(3)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_in.wait_event(e0)
    s_out.wait_event(e0)
    run(steps)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    del lays[1]
    return {"ms": e0.elapsed_time(e1) / steps, "h2d": h2d, "d2h": d2h}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--warmup-seconds", type=float, default=1.0,
                    help="keep warming up for at least this long (clock sampling under load)")
    ap.add_argument("--batch", type=int, default=None, help="override the batch (smaller profiling case)")
    ap.add_argument("--workload", default="layer", choices=["layer", "sweep", "prefill65k", "prefill262k", "ssd", "ssd_cache", "ssd_train",
                             "mixer"],
                    help="layer: the step line; others: extra lines on one GPU")
    args = ap.parse_args()
    if args.batch:
        CFG["batch"] = args.batch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.workload != "layer":
        if rank == 0:
            if args.workload == "sweep":
                run_sweep(args)
            elif args.workload == "ssd":
                run_ssd(args)
            elif args.workload == "ssd_cache":
                run_ssd_cache(args)
            elif args.workload == "ssd_train":
                run_ssd_train(args)
            elif args.workload == "mixer":
                run_mixer(args)
            elif args.workload == "prefill65k":
                run_prefill(args, 65536, 32, 1)
            else:
                run_prefill(args, 262144, 16, 16)
        return
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    try:
        run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
