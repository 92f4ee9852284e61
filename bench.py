#!/usr/bin/env python
"""Benchmark of the Seer hot path on GB300 (prints ONE JSON line on rank 0).

A step is one pass of the whole hot path over one batch of synthetic input:
step-0 boundary detection (SwiGLU GEMM + fused sparsity count + SNR scan),
routing + device-resident compaction, and one truncated denoising layer
(RMSNorm, QKV, varlen bidirectional attention, O projection, SwiGLU MLP).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload suite|0..4] [--impl ours|reference]

The default run (``--workload suite``) leads with the video-shaped layer
(workload 4: batch 4, 11.8k-row visual prefixes, window 2048), the largest
single-layer configuration, and carries the ragged batch-16 layer (workload 2)
and the 32-layer x 64-step stack (workload 3) as sub-records of the same line,
each with its own timing, roofline, oracle baseline, end-to-end figure and
clock record.

``value``  valid tokens per second of the device-resident step (inputs in HBM);
``e2e``    the same metric with the host->device copy of the step's input and
           the device->host copy of its output inside the timed region;
``--impl reference`` times the CPU oracle (a plain fp64 statement of the
method; the paper ships no code to run instead) on a bounded sample of the
same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

PRECISION = "bf16 layer inputs/outputs, f16 tensor-core operands and intermediates, fp32 accumulation"
METRIC = "truncated denoise-layer tokens/s & TFLOP/s vs BF16 peak; speedup over padded"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
KERNELS_PER_STEP = 11   # detect GEMM, scan, pack, norm, QKV, attn schedule, attn, O proj, norm, gate/up, down
SUITE = (4, 2, 3)       # headline first: the video layer, then the ragged batch-16 layer and the 32-layer stack
TENSOR_PHASES = ("detect_gemm", "qkv", "attention", "o_proj", "gate_up", "down")
KERNEL_OF_PHASE = {
    "detect_gemm": "tc_gemm_kernel<Count> (step-0 detector, counts only)",
    "qkv": "tc_gemm_kernel<Store> (QKV projection)",
    "attention": "tc_attn_kernel (varlen bidirectional attention)",
    "o_proj": "tc_gemm_kernel<Residual> (O projection + residual)",
    "gate_up": "tc_gemm_kernel<Swiglu> (gate/up + SwiGLU)",
    "down": "tc_gemm_kernel<Residual> (down projection + residual)",
}
# kept rows above which the oracle's layer time is extrapolated from a key/value
# pass and a sample of query rows instead of measured on every row
ORACLE_FULL_ROWS = 4096


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", default="suite", choices=["suite", "0", "1", "2", "3", "4"])
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--launch-overlap", default="on", choices=["on", "off"],
                    help="programmatic dependent launch of the library kernels (default on)")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def code_digest(paths) -> str:
    """SHA-1 of the code in `paths` (files relative to the repository root) with
    `//` comments, trailing blanks and empty lines removed, so that editing a
    comment does not invalidate a capture."""
    import hashlib
    import re
    h = hashlib.sha1()
    for s in paths:
        with open(os.path.join(ROOT, s)) as f:
            for line in f:
                code = re.sub(r"//.*$", "", line).rstrip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()


def measured_traffic(workload: int, phase: str):
    """DRAM bytes per launch of the kernel of `phase` from the committed ncu
    capture of this workload, or None when the kernel code changed since that
    capture."""
    path = os.path.join(ROOT, "profiles", f"traffic_workload{workload}.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        doc = json.load(f)
    k = doc["kernels"].get(phase)
    if k is None or code_digest(k["sources"]) != k.get("sources_code_sha1"):
        return None
    return k["traffic_bytes"]


def graph_capacity(total: int) -> int:
    """Smallest m * 2^e >= total with m in 8..15 (the launch capacity the pack
    kernel reports for graph replay)."""
    if total <= 8:
        return 8
    e = 0
    while (15 << e) < total:
        e += 1
    return ((total + (1 << e) - 1) >> e) << e


def layer_flops(seg, kv, d, F):
    """Algorithmic FLOPs of one layer (Eq. 2 made exact): projections 8*T*d^2,
    MLP 6*T*d*F, attention 4*d*sum(L_q * L_kv)."""
    seg = np.asarray(seg, dtype=np.float64)
    kv = np.asarray(kv, dtype=np.float64)
    return float(8.0 * seg.sum() * d * d + 6.0 * seg.sum() * d * F + 4.0 * d * np.sum(seg * kv))


# ----------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or self.path is None:
            return None
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 8:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[4:8]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------------- oracle arm
_ORACLE_INPUTS = {}


def oracle_sample(wl):
    """Time the CPU oracle on one sequence of the workload (the shortest one):
    detection over its whole window, the boundary scan, and one truncated layer
    over its kept rows.

    Where the kept rows exceed ORACLE_FULL_ROWS (the video workload: ~12k rows,
    about a minute of fp64 work), the layer time is extrapolated from two
    measurements: the key/value pass over every kept row alone (RMSNorm and the
    K and V projections, ``oracle.kv_prefill``: work the layer does once) and the
    layer on a sample of n query rows (the same key/value pass plus, per query
    row, its projections, attention over every key including the softmax's
    exponentials, and the MLP).  The per-row part is the difference of the two,
    scaled to every kept row: t = t_kv + (t_rows(n) - t_kv) * keep / n.

    Returns ``(kept_rows, seconds, description)``, seconds being the detection
    time plus the (possibly extrapolated) layer time."""
    import oracle
    if wl.index not in _ORACLE_INPUTS:
        lens = synth.lengths(wl)
        x, cu_full, resp = synth.hidden_full(wl, lens)
        _ORACLE_INPUTS[wl.index] = (lens, x, cu_full, resp, synth.layer_weights(wl, 0))
    lens, x, cu_full, resp, w = _ORACLE_INPUTS[wl.index]
    b = int(np.argmin(lens.full))
    t0 = time.perf_counter()
    rows = x[resp[b]:resp[b] + wl.window]
    counts = oracle.sparsity_counts(rows, w["wg"], w["wu"], wl.act_eps)
    _, L = oracle.snr_boundary(counts, wl.d_ff)
    keep = int(lens.ctx[b] + L)
    seg = x[cu_full[b]:cu_full[b] + keep]
    t_detect = time.perf_counter() - t0
    if keep <= ORACLE_FULL_ROWS:
        t1 = time.perf_counter()
        oracle.layer_forward_segment(seg, w, wl.n_heads)
        t_layer = time.perf_counter() - t1
        how = "one truncated layer"
    else:
        n = 512
        q_rows = np.sort(np.random.default_rng(0).choice(keep, size=n, replace=False))
        t1 = time.perf_counter()
        oracle.kv_prefill(seg, w, wl.n_heads)
        t_kv = time.perf_counter() - t1
        t1 = time.perf_counter()
        oracle.layer_forward_rows(seg, w, wl.n_heads, q_rows)
        t_n = time.perf_counter() - t1
        t_layer = t_kv + max(t_n - t_kv, 0.0) * keep / n
        how = (f"one truncated layer, extrapolated from the key/value pass over all {keep} rows ({t_kv:.2f} s) and the "
               f"layer on {n} sampled query rows ({t_n:.2f} s): t_kv + (t_rows - t_kv) * {keep} / {n}")
    dt = t_detect + t_layer
    return keep, dt, (f"sequence {b} ({keep} kept rows of {int(lens.full[b])}): detection over its {wl.window}-token "
                      f"window + {how}, fp64 numpy")


def layer_config(wl, world, args, L, groups, pad_rows, capacity, T_full, T_valid, T_exec) -> dict:
    """``config`` of a layer workload (the same dict in both arms)."""
    d, F = wl.d, wl.d_ff
    es = 2 if wl.dtype == "bf16" else 4
    return {"workload": f"{wl.name} (workload {wl.index}): batch {wl.batch}, window {wl.window}, "
                        f"d {d}, heads {wl.n_heads}x{wl.head_dim}, F {F}",
            "batch": wl.batch, "window": wl.window, "tokens_full": T_full, "tokens_valid": T_valid,
            "tokens_executed": T_exec, "L_star": [int(v) for v in L],
            "l2": "inputs larger than L2 (x_full %.0f MB, weights %.0f MB)" % (T_full * d * es / 1e6,
                                                                              (4 * d * d + 3 * d * F) * 2 / 1e6),
            "route": {"groups": groups, "pad_rows": int(pad_rows), "capacity": int(capacity)},
            "parallelism": f"replicas x{world}", "launch_overlap": args.launch_overlap}


def stack_config(wl, args, L, groups, capacity, T_full, T_valid, T_exec) -> dict:
    d, F = wl.d, wl.d_ff
    return {"workload": f"{wl.name} (workload 3): {wl.n_layers} layers x {wl.steps} denoising steps, batch "
                        f"{wl.batch}, window {wl.window}, d {d}, F {F}; tokens counted once per layer and step",
            "tokens_full": T_full, "tokens_valid": T_valid, "tokens_executed": T_exec, "L_star": [int(v) for v in L],
            "route": {"groups": groups, "capacity": int(capacity)},
            "l2": "inputs larger than L2 (weights %.1f GB)" % (wl.n_layers * (4 * d * d + 3 * d * F) * 2 / 1e9),
            "launch_overlap": args.launch_overlap}


def suite_note() -> str:
    return ("headline: workload 4 (the largest single-layer configuration); sub_records: workload 2 (ragged "
            "batch-16 layer) and workload 3 (32-layer x 64-step stack)")


def reference_config(wl, world, args) -> dict:
    """The ``config`` of this workload as our arm reports it, computed on the
    host from the synthetic lengths and the oracle's routing (the planted
    boundaries give L* = b + 1, which the GPU detection reproduces exactly)."""
    import oracle
    lens = synth.lengths(wl)
    L = (lens.boundary + 1).astype(np.int64)
    tau = 0.2
    seg, kv, cu = oracle.segment_layout(lens.ctx, L, wl.window, tau)
    T_full, T_valid, T_exec = int(lens.full.sum()), int(kv.sum()), int(cu[-1])
    route = oracle.route(L, wl.window, tau)
    groups = [{"bucket": g["bucket"], "members": len(g["members"]), "path": g["path"],
               "rho": int(np.floor(g["rho"] * 1e6)) / 1e6} for g in route]
    pad = int(sum(g["bucket"] * len(g["members"]) - int(L[g["members"]].sum())
                  for g in route if g["path"] == oracle.PATH_STATIC))
    if wl.index == 3:
        return stack_config(wl, args, L, groups, graph_capacity(T_exec), T_full, T_valid, T_exec)
    return layer_config(wl, world, args, L, groups, pad, graph_capacity(T_exec), T_full, T_valid, T_exec)


def run_reference(args, wl, rank, world, suite):
    if rank != 0:
        return
    cores = len(os.sched_getaffinity(0))
    for _ in range(args.warmup):
        oracle_sample(wl)
    toks, secs = 0, 0.0
    sample = ""
    for _ in range(args.steps):
        k, dt, sample = oracle_sample(wl)
        toks += k
        secs += dt
    v = toks / secs
    cfg = reference_config(wl, world, args)
    if suite:
        cfg["suite"] = suite_note()
    line = {"metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": cfg,
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def cpu_baseline(wl, unit="tokens/s"):
    k, dt, sample = oracle_sample(wl)
    return {"value": k / dt, "unit": unit, "cores": len(os.sched_getaffinity(0)), "kind": "oracle",
            "sample": sample, "seconds": dt}


# ----------------------------------------------------------------- environment of our arm
class Env:
    def __init__(self):
        import torch
        import torch.distributed as dist
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        torch.cuda.set_device(self.local)
        self.dev = torch.device("cuda", self.local)
        if self.world > 1:
            dist.init_process_group("nccl", device_id=self.dev)
        from paper_2607_14557_gb300 import replicas as R
        self.R = R

    def barrier(self):
        self.R.barrier(self.dev)

    def max_over_ranks(self, v):
        return self.R.max_over_ranks(v, self.dev)

    def sum_over_ranks(self, v):
        return self.R.sum_over_ranks(v, self.dev)

    def close(self):
        if self.world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


# ----------------------------------------------------------------- stack (workload 3)
def run_stack(args, wl, env, with_cpu):
    """32-layer stack, 64 denoising steps: step 0 over the full windows (with the
    fused count hook at the detection layer), detection + route/pack, then 63
    truncated steps replayed from a CUDA graph; against 64 untruncated steps
    replayed from their own graph.  Returns the JSON record."""
    import torch

    from paper_2607_14557_gb300 import driver as D
    from paper_2607_14557_gb300 import seer as S

    dev, world, R = env.dev, env.world, env.R
    detect_layer = 3
    lens = synth.lengths(wl)
    x_np, cu_full_np, resp_np = synth.hidden_full(wl, lens)
    x_full = torch.from_numpy(x_np).to(torch.bfloat16).to(dev)
    i32 = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32)).to(dev)
    cu_full, resp, ctx = i32(cu_full_np), i32(resp_np), i32(lens.ctx)
    t0 = time.perf_counter()
    layers = [None] * wl.n_layers
    for l, bits in synth.stack_weights_bf16_bits(wl, range(wl.n_layers)):
        layers[l] = D.LayerWeights.from_bf16_bits(bits, dev, keep_model=("w_gate", "w_up") if l == detect_layer else ())
    t_weights = time.perf_counter() - t0
    dims = S.make_dims(wl.d, wl.n_heads, wl.head_dim, wl.d_ff)
    params = S.make_params(wl.act_eps)
    T_full = int(cu_full_np[-1])
    stack = D.SeerStack(dims, "bf16", wl.batch, wl.window, T_full, params, layers, detect_layer, dev)
    stream = torch.cuda.current_stream()
    n_steps = wl.steps

    # warm-up: step 0, the graphs, a few steps of each
    stack.step0(x_full, cu_full, resp, ctx, stream)
    route = stack.path.route()
    g_trunc = stack.truncated_graph(route["capacity"])
    g_pad = stack.capture("padded", lambda stream: stack.padded_step(x_full, cu_full, stream=stream))
    for _ in range(max(args.warmup, 3)):
        g_trunc.replay()
        g_pad.replay()
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
    L = stack.path.L_star.cpu().numpy()
    seg = np.diff(stack.path.cu.cpu().numpy())
    kv = stack.path.kv.cpu().numpy()
    T_valid, T_exec = int(kv.sum()), int(seg.sum())
    d, F, nl = wl.d, wl.d_ff, wl.n_layers

    ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
    env.barrier()
    with ClockSampler(env.local) as clk:
        ev[0].record(stream)
        stack.step0(x_full, cu_full, resp, ctx, stream)
        ev[1].record(stream)
        r = stack.path.route()
        g = stack.truncated_graph(r["capacity"])
        for _ in range(n_steps - 1):
            g.replay()
        ev[2].record(stream)
        for _ in range(n_steps):
            g_pad.replay()
        ev[3].record(stream)
        stack.step0_truncating(x_full, cu_full, resp, ctx, stream)
        ev[4].record(stream)
        torch.cuda.synchronize()
    # prefix K/V caching composed with truncation: step 0 full, step 1 truncated
    # with the cache prefill, steps 2..63 over the response rows only
    resp_total = int(r["total"]) - int(lens.ctx.sum())
    resp_cap = graph_capacity(resp_total)
    stack.step0(x_full, cu_full, resp, ctx, stream)
    stack.path.route()
    stack.prefill_step(stream)
    g_cached = stack.cached_graph(resp_cap)
    for _ in range(max(args.warmup, 3)):
        g_cached.replay()
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
    evc = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    with ClockSampler(env.local) as clk_c:
        evc[0].record(stream)
        stack.step0(x_full, cu_full, resp, ctx, stream)
        evc[1].record(stream)
        stack.path.route()
        stack.prefill_step(stream)
        evc[2].record(stream)
        for _ in range(n_steps - 2):
            g_cached.replay()
        evc[3].record(stream)
        torch.cuda.synchronize()
    assert S.seer_check_device() == 0

    # ---- end to end: one generation through the public API from pinned host
    # memory: upload the step-0 input, step 0 + route/pack, the 63 truncated steps,
    # then download the last step's packed output rows and L*
    e2e = None
    if not args.no_e2e:
        x_host = torch.from_numpy(x_np).to(torch.bfloat16).pin_memory()
        x_dev = torch.empty_like(x_full)
        out_host = torch.empty((T_full, wl.d), dtype=torch.bfloat16).pin_memory()
        L_host = torch.empty(wl.batch, dtype=torch.int32).pin_memory()
        torch.cuda.synchronize()
        a_e, b_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t_e = time.perf_counter()
        a_e.record(stream)
        x_dev.copy_(x_host, non_blocking=True)
        stack.step0(x_dev, cu_full, resp, ctx, stream)
        r_e = stack.path.route()
        g_e = stack.truncated_graph(r_e["capacity"])
        for _ in range(n_steps - 1):
            g_e.replay()
        out_dev = stack.buf[(wl.n_layers - 1) % 2]
        out_host[:r_e["total"]].copy_(out_dev[:r_e["total"]], non_blocking=True)
        L_host.copy_(stack.path.L_star, non_blocking=True)
        b_e.record(stream)
        torch.cuda.synchronize()
        ms_e2e = max(a_e.elapsed_time(b_e), (time.perf_counter() - t_e) * 1e3)
        tok_e = (T_full + (n_steps - 1) * T_valid) * wl.n_layers
        e2e = {"value": env.sum_over_ranks(tok_e) / (env.max_over_ranks(ms_e2e) * 1e-3), "unit": "tokens/s",
               "ms_per_generation": ms_e2e,
               "h2d_bytes_per_step": x_host.numel() * x_host.element_size() / n_steps,
               "d2h_bytes_per_step": (r_e["total"] * wl.d * 2 + wl.batch * 4) / n_steps,
               "note": "one generation (64 steps): the input uploaded once, the last step's rows downloaded once"}
        assert S.seer_check_device() == 0
    ms0 = ev[0].elapsed_time(ev[1])
    ms_rest = ev[1].elapsed_time(ev[2])
    ms_pad = ev[2].elapsed_time(ev[3])
    ms_seer = ms0 + ms_rest
    ms0_f1 = ev[3].elapsed_time(ev[4])
    dl = detect_layer + 1
    ms_c0, ms_c1, ms_cr = evc[0].elapsed_time(evc[1]), evc[1].elapsed_time(evc[2]), evc[2].elapsed_time(evc[3])
    ms_cached_total = ms_c0 + ms_c1 + ms_cr
    fl_full = layer_flops(lens.full, lens.full, d, F) * nl
    fl_trunc = layer_flops(seg, kv, d, F) * nl
    fl_valid = layer_flops(kv, kv, d, F) * nl
    tok_layers = (T_full + (n_steps - 1) * T_valid) * nl
    # replicas: every rank runs its own batch; the job's rate is all ranks'
    # token-layers over the slowest rank's time
    value = env.sum_over_ranks(tok_layers) / (env.max_over_ranks(ms_seer) * 1e-3)
    pk, src = peaks()
    tflops_rest = fl_trunc * (n_steps - 1) / (ms_rest * 1e-3) / 1e12
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": n_steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_seer / n_steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f16", "precision": PRECISION, "data": "synthetic",
        "config": dict(stack_config(wl, args, L, r["groups"], r["capacity"], T_full, T_valid, T_exec),
                       weights_setup_s=t_weights),
        "stack": {"ms_step0_full": ms0, "ms_steps_1_to_%d" % (n_steps - 1): ms_rest, "ms_padded_%d_steps" % n_steps: ms_pad,
                  "speedup_vs_padded": ms_pad / ms_seer,
                  "ideal_ratio": fl_full * n_steps / (fl_full + fl_valid * (n_steps - 1)),
                  "tflops_truncated_steps": tflops_rest, "frac_of_burst_peak": tflops_rest / pk["bf16_tflops"],
                  "frac_of_sustained_peak": tflops_rest / pk["bf16_tflops_sustained"],
                  "tflops_padded": fl_full * n_steps / (ms_pad * 1e-3) / 1e12,
                  "truncated_tokens_per_s": T_valid * nl * (n_steps - 1) / (ms_rest * 1e-3)},
        "step0_truncated_after_detection": {
            "ms_step0": ms0_f1, "layers_full": dl, "layers_packed": nl - dl,
            "ms_total_%d_steps" % n_steps: ms0_f1 + ms_rest, "speedup_vs_padded": ms_pad / (ms0_f1 + ms_rest),
            "ideal_ratio": fl_full * n_steps / (fl_full * dl / nl + fl_valid * (nl - dl) / nl + fl_valid * (n_steps - 1)),
            "tokens_per_s": (T_full * dl + T_valid * (nl - dl) + (n_steps - 1) * T_valid * nl) / ((ms0_f1 + ms_rest) * 1e-3)},
        "prefix_kv_cache": {
            "ms_step0_full": ms_c0, "ms_step1_truncated_with_prefill": ms_c1,
            "ms_steps_2_to_%d_response_rows" % (n_steps - 1): ms_cr, "ms_per_cached_step": ms_cr / (n_steps - 2),
            "response_rows_per_step": resp_total, "launch_capacity": resp_cap,
            "ms_total_%d_steps" % n_steps: ms_cached_total, "speedup_vs_padded": ms_pad / ms_cached_total,
            "speedup_vs_truncated_uncached": ms_seer / ms_cached_total,
            "tokens_per_s": (T_full + (n_steps - 1) * T_valid) * nl / (ms_cached_total * 1e-3),
            "clocks": clk_c.summary()},
        "roofline": {"kernel": "the truncated layer's kernels under graph replay (steps 1..%d)" % (n_steps - 1),
                     "bound": "tensor", "achieved": tflops_rest, "peak": pk["bf16_tflops_sustained"],
                     "unit": "TFLOP/s", "frac": tflops_rest / pk["bf16_tflops_sustained"], "traffic": None,
                     "peak_source": f"{src} bf16 dense, sustained (a {ms_rest / 1e3:.0f} s region under the power cap)"},
        "e2e": e2e,
        "gpu_launches": nl * 8 * (2 * n_steps) + 3 + (nl * 8 + 4)
                        + (nl * 8 + 3) + nl * 13 + (n_steps - 2) * (2 + nl * 9), "clocks": clk.summary(),
        "peak_source": src,
    }
    if with_cpu:
        line["cpu_baseline"] = cpu_baseline(wl, "tokens/s (token-layers: one layer pass)")
    del stack, layers, x_full, g, g_trunc, g_pad, g_cached
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return line


# ----------------------------------------------------------------- a single-layer workload
def run_layer(args, wl, env, with_cpu):
    """Detect + route/pack + one truncated layer per step (workloads 0, 1, 2, 4).
    Returns the JSON record."""
    import torch

    from paper_2607_14557_gb300 import driver as D
    from paper_2607_14557_gb300 import seer as S

    dev, world = env.dev, env.world

    # ---- synthetic inputs, resident in HBM before timing
    lens = synth.lengths(wl)
    x_np, cu_full_np, resp_np = synth.hidden_full(wl, lens)
    w_np = synth.layer_weights(wl, 0)
    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    x_host = torch.from_numpy(x_np).to(tdt).pin_memory()
    del x_np
    x_full = x_host.to(dev)
    i32 = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32)).to(dev)
    cu_full, resp, ctx = i32(cu_full_np), i32(resp_np), i32(lens.ctx)
    W = D.LayerWeights.from_host(w_np, wl.dtype, dev)
    W.drop_model_copy()
    dims = S.make_dims(wl.d, wl.n_heads, wl.head_dim, wl.d_ff)
    params = S.make_params(wl.act_eps)
    T_full = int(cu_full_np[-1])
    path = D.SeerPath(dims, wl.dtype, wl.batch, wl.window, T_full, params, dev)
    stream = torch.cuda.current_stream()

    def step():
        path.step(x_full, cu_full, resp, ctx, W, stream)
        return path.route()

    # ---- warm-up and the route of this batch
    for _ in range(max(args.warmup, 3)):
        route = step()
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
    L = path.L_star.cpu().numpy()
    seg = np.diff(path.cu.cpu().numpy())
    kv = path.kv.cpu().numpy()
    T_exec = int(seg.sum())
    T_valid = int(kv.sum())
    d, F = wl.d, wl.d_ff
    flops_exec = layer_flops(seg, kv, d, F)
    flops_valid = layer_flops(kv, kv, d, F)
    flops_pad = layer_flops(lens.full, lens.full, d, F)
    flops_of = {"qkv": 6.0 * T_exec * d * d, "o_proj": 2.0 * T_exec * d * d, "gate_up": 4.0 * T_exec * d * F,
                "down": 2.0 * T_exec * d * F, "attention": 4.0 * d * float(np.sum(seg * kv)),
                "detect_gemm": 4.0 * wl.batch * wl.window * d * F}

    # ---- per-kernel breakdown (untimed for the headline): the same steps with
    # events around every phase; it also names the dominant kernel
    S.seer_profile_reset()
    S.seer_profile_select(None)
    S.seer_profile_enable(True)
    for _ in range(args.steps):
        step()
    torch.cuda.synchronize()
    S.seer_profile_enable(False)
    phases = S.seer_profile_read()
    tensor_ms = {p: phases[p][0] for p in TENSOR_PHASES if phases.get(p, (0, 0))[1]}
    dominant = max(tensor_ms, key=tensor_ms.get) if wl.dtype == "bf16" else "gate_up"

    # ---- timed region: K whole steps (device-resident inputs > L2); CUDA events
    # only around the dominant kernel, so launch overlap elsewhere is kept
    env.barrier()
    S.seer_profile_reset()
    S.seer_profile_select([dominant])
    S.seer_profile_enable(True)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(env.local) as clk:
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        env.barrier()
    S.seer_profile_enable(False)
    ms_step = e0.elapsed_time(e1) / args.steps
    dominant_timed = S.seer_profile_read()[dominant]
    phases[dominant] = dominant_timed
    ms_step_max = env.max_over_ranks(ms_step)
    tokens_all = env.sum_over_ranks(T_valid)
    value = tokens_all / (ms_step_max * 1e-3)

    # ---- layer-only timings: truncated vs untruncated (padded) window
    y_full = torch.empty((T_full, d), dtype=tdt, device=dev)

    def timed(fn, n):
        # each comparison starts from the same thermal state: a second idle, then
        # two untimed calls (the truncated, padded and naive layers run back to
        # back otherwise, and the later ones would meet a power-capped clock)
        env.barrier()
        time.sleep(1.0)
        for _ in range(2):
            fn()
        env.barrier()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(n):
            fn()
        b.record(stream)
        env.barrier()
        return a.elapsed_time(b) / n

    ms_layer = timed(lambda: path.layer(W, stream=stream), args.steps)
    ms_pad = timed(lambda: path.padded_forward(x_full, cu_full, W, y_full, stream), args.steps)
    # naive-pad comparator: truncated sequences padded to the batch's longest L* (keys masked)
    x_nv, cu_nv, kv_nv, T_nv = path.naive_pad_inputs(x_full, cu_full, ctx, stream)
    y_nv = torch.empty((T_nv, d), dtype=tdt, device=dev)
    ms_naive = timed(lambda: path.layer(W, x=x_nv, y=y_nv, cu=cu_nv, kv=kv_nv, T_cap=T_nv, stream=stream),
                     args.steps)
    seg_nv = np.diff(cu_nv.cpu().numpy())
    flops_naive = layer_flops(seg_nv, kv_nv.cpu().numpy(), d, F)
    del x_nv, y_nv
    # the router's padding priced: the same batch with the static path switched
    # off (every segment keeps exactly ctx + L* rows), layer against layer
    x_vo, cu_vo, kv_vo, T_vo = path.varlen_only_inputs(x_full, cu_full, ctx, stream)
    ms_varlen = timed(lambda: path.layer(W, x=x_vo, cu=cu_vo, kv=kv_vo, T_cap=T_vo, stream=stream), args.steps)
    T_vo_exec = int(cu_vo[-1].item())
    del x_vo

    # ---- end to end through the API with host buffers
    e2e = None
    if not args.no_e2e:
        y_host = torch.empty((T_full, d), dtype=tdt).pin_memory()
        L_host = torch.empty(wl.batch, dtype=torch.int32).pin_memory()

        # SeerPath.run_from_host: every step uploads its input from pinned memory and
        # downloads its packed output and L*; copies overlap neighbouring steps' compute
        copy_stream = torch.cuda.Stream(dev)
        path.run_from_host(x_host, cu_full, resp, ctx, W, y_host, L_host, 2, stream, copy_stream)
        env.barrier()
        t0 = time.perf_counter()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        r = path.run_from_host(x_host, cu_full, resp, ctx, W, y_host, L_host, args.steps, stream, copy_stream)
        b.record(stream)
        env.barrier()
        # the call returns after its last copy: the host clock bounds the whole region
        ms_e2e = env.max_over_ranks(max(a.elapsed_time(b), (time.perf_counter() - t0) * 1e3) / args.steps)
        h2d = x_host.numel() * x_host.element_size()
        d2h = r["total"] * d * x_host.element_size() + wl.batch * 4
        e2e = {"value": tokens_all / (ms_e2e * 1e-3), "unit": "tokens/s", "ms_per_step": ms_e2e,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "pipelining": "double-buffered: step i+1's upload and step i-1's download overlap step i"}

    assert S.seer_check_device() == 0

    # ---- roofline of the dominant kernel
    pk, src = peaks()
    kernels = {}
    for name, (ms, n) in phases.items():
        if n:
            kernels[name] = {"ms_per_launch": ms / n, "launches": n}
    for name, fl in flops_of.items():
        if name in kernels:
            kernels[name]["tflops"] = fl / (kernels[name]["ms_per_launch"] * 1e-3) / 1e12
            kernels[name]["frac_of_burst_peak"] = kernels[name]["tflops"] / pk["bf16_tflops"]
    es = 2 if wl.dtype == "bf16" else 4
    bytes_of = {"pack": 2.0 * T_exec * d * es, "norm1": T_exec * d * (es + 2), "norm2": T_exec * d * 4}
    for name, by in bytes_of.items():
        if name in kernels:
            kernels[name]["gbs"] = by / (kernels[name]["ms_per_launch"] * 1e-3) / 1e9
    dk = kernels.get(dominant, {})
    achieved = dk.get("tflops")
    # algorithmic bytes per launch of each tensor kernel (operands read once,
    # outputs written once; intermediates are f16)
    alg_bytes = {"gate_up": 2.0 * T_exec * d + 2 * 2 * F * d + 2.0 * T_exec * F,
                 "down": 2.0 * T_exec * F + 2.0 * F * d + 2 * 2.0 * T_exec * d,
                 "qkv": 2.0 * T_exec * d + 2.0 * 3 * d * d + 2.0 * T_exec * 3 * d,
                 "o_proj": 2.0 * T_exec * d + 2.0 * d * d + 2 * 2.0 * T_exec * d,
                 "attention": 2.0 * T_exec * 3 * d + 2.0 * T_exec * d,
                 "detect_gemm": 2.0 * wl.batch * wl.window * d + 2 * 2 * F * d}
    # the timed region is well under a second at full clocks: the burst figure is
    # the denominator (the sustained one, a seconds-long loop under the power
    # cap, is reported beside it)
    peak = pk["bf16_tflops"]
    roofline = {"kernel": KERNEL_OF_PHASE.get(dominant, dominant), "phase": dominant, "bound": "tensor",
                "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak if achieved else None,
                "frac_of_sustained": achieved / pk["bf16_tflops_sustained"] if achieved else None,
                "traffic": measured_traffic(wl.index, dominant),
                "algorithmic_bytes": float(alg_bytes[dominant]),
                "peak_source": f"{src} bf16 dense, burst (f16 operands run at the bf16 rate)",
                "flops_per_launch": flops_of[dominant],
                "why_this_kernel": "the tensor-core kernel with the largest share of the step's time "
                                   "(per-phase CUDA events)"}
    if wl.dtype == "f32":
        # the fp32 layer runs on CUDA cores: its gate/up GEMM against the fp32 FMA rate,
        # derived from the unit counts and the clock (152 SMs x 128 fp32 lanes x 2 FLOP x 2.07 GHz)
        alu_peak = 152 * 128 * 2 * 2.07e9 / 1e12
        roofline.update({"kernel": "simt_gemm_kernel (gate/up + SwiGLU, fp32 CUDA cores)", "bound": "alu",
                         "peak": alu_peak, "frac": achieved / alu_peak if achieved else None,
                         "frac_of_sustained": None, "traffic": None,
                         "peak_source": "derived: 152 SMs x 128 fp32 FMA lanes x 2 FLOP x 2.07 GHz (80.5 TFLOP/s)",
                         "why_this_kernel": "the gate/up GEMM of the fp32 layer (latency-bound at ~121 rows)"})

    clocks = clk.summary()
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step_max, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f16" if wl.dtype == "bf16" else "f32",
        "precision": PRECISION if wl.dtype == "bf16" else "fp32 storage and arithmetic (CUDA cores)",
        "data": "synthetic",
        "config": layer_config(wl, world, args, L, route["groups"], route["pad_rows"], route["capacity"], T_full,
                               T_valid, T_exec),
        "layer": {"ms_truncated": ms_layer, "ms_padded": ms_pad, "tflops": flops_exec / (ms_layer * 1e-3) / 1e12,
                  "frac_of_burst_peak": flops_exec / (ms_layer * 1e-3) / 1e12 / pk["bf16_tflops"],
                  "frac_of_sustained_peak": flops_exec / (ms_layer * 1e-3) / 1e12 / pk["bf16_tflops_sustained"],
                  "speedup_vs_padded": ms_pad / ms_layer, "ideal_ratio": flops_pad / flops_valid,
                  "flops_executed": flops_exec, "flops_valid": flops_valid, "flops_padded": flops_pad},
        "naive_pad": {"ms": ms_naive, "tokens_executed": int(T_nv), "flops_executed": flops_naive,
                      "speedup_truncated_vs_naive": ms_naive / ms_layer, "ideal_ratio": flops_naive / flops_valid},
        "route_cost": {"tau_pad": 0.2, "pad_rows": int(route["pad_rows"]), "tokens_executed": T_exec,
                       "ms_layer": ms_layer, "ms_layer_varlen_only": ms_varlen,
                       "tokens_executed_varlen_only": T_vo_exec, "ms_cost_of_pad_rows": ms_layer - ms_varlen,
                       "note": "static-path groups pad their responses to the bucket (rows computed as queries, "
                               "masked as keys); varlen-only keeps ctx + L* rows in every segment"},
        "speedup_step_vs_padded_layer": ms_pad / ms_step,
        "kernels": kernels,
        "kernel_timing": f"{dominant}: CUDA events around that kernel alone inside the timed region; the other "
                         "kernels: a separate pass of the same steps with events around every phase",
        "roofline": roofline, "gpu_launches": KERNELS_PER_STEP * args.steps,
        "e2e": e2e, "clocks": clocks,
    }
    if with_cpu:
        line["cpu_baseline"] = cpu_baseline(wl)
    del path, W, x_full, x_host, y_full
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return line


SUB_KEYS = ("value", "unit", "ms_per_step", "steps", "warmup", "config", "layer", "stack", "naive_pad", "route_cost",
            "step0_truncated_after_detection", "prefix_kv_cache", "kernels", "roofline", "gpu_launches", "e2e",
            "clocks", "cpu_baseline")


def sub_record(line: dict) -> dict:
    return {k: line[k] for k in SUB_KEYS if k in line}


# ----------------------------------------------------------------- our arm
def main():
    args = parse()
    suite = args.workload == "suite"
    head = synth.workload(SUITE[0] if suite else int(args.workload))
    if args.impl == "reference":
        run_reference(args, head, int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), suite)
        return
    from paper_2607_14557_gb300 import seer as S_

    S_.seer_set_launch_overlap(args.launch_overlap == "on")
    env = Env()
    with_cpu = env.world == 1 and env.rank == 0 and not args.no_cpu_baseline
    run = run_stack if head.index == 3 else run_layer
    line = run(args, head, env, with_cpu)
    if suite:
        line["config"]["suite"] = suite_note()
        subs = {}
        for idx in SUITE[1:]:
            wl = synth.workload(idx)
            rec = (run_stack if idx == 3 else run_layer)(args, wl, env, with_cpu)
            subs[f"workload_{idx}"] = sub_record(rec)
        line["sub_records"] = subs
        line["gpu_launches_all_records"] = line["gpu_launches"] + sum(s["gpu_launches"] for s in subs.values())
    if env.rank == 0:
        print(json.dumps(line), flush=True)
    env.close()


if __name__ == "__main__":
    main()
