"""Microbenchmark of single hot-path kernels through the C ABI (synthetic inputs).

    python -m paper_2607_14557_gb300.kernel_bench attention --lens 3100x8 [--heads 32] [--dtype f16]
    python -m paper_2607_14557_gb300.kernel_bench linear --M 35194 --N 12288 --K 4096 [--dtype f16]
    python -m paper_2607_14557_gb300.kernel_bench pack [--batch 16 --window 1024 --d 4096]
    python -m paper_2607_14557_gb300.kernel_bench scan [--batch 16 --window 1024]
    python -m paper_2607_14557_gb300.kernel_bench norm [--M 35194 --d 4096]
    python -m paper_2607_14557_gb300.kernel_bench swiglu --M 35194 --F 12288 --K 4096 [--dtype f16]

Each call runs the kernel `--warmup` times, then times `--reps` calls with CUDA
events on the launching stream and prints one JSON line (ms per call and
TFLOP/s of the algorithmic work: 4*d*sum(L^2) for attention, 2*M*N*K for a
linear, 4*M*F*K for the gate/up GEMM with its SwiGLU epilogue; GB/s of algorithmic bytes for pack (each kept row read and written
once) and scan (each count read once)); GB/s for norm (bf16 rows read once, f16 rows
written once).  pack and scan use the lengths of the
ragged 8B-layer workload (visual 729k, k in 1..5; prompt 32..128; boundary
16..400).  Inputs are random and resident in device memory; no output is checked
(the parity tests do that).  Used for per-kernel timings and small ncu captures.
"""
from __future__ import annotations

import argparse
import json

import numpy as np
import torch

from . import seer as S


def _lens(spec: str):
    out = []
    for part in spec.split(","):
        if "x" in part:
            length, count = part.split("x")
            out += [int(length)] * int(count)
        else:
            out.append(int(part))
    return out


def _time(fn, warmup: int, reps: int) -> float:
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        fn()
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / max(reps, 1)


def attention(args) -> dict:
    lens = _lens(args.lens)
    H, dh = args.heads, 128
    D = H * dh
    dev = torch.device("cuda", 0)
    tdt = {"f16": torch.float16, "bf16": torch.bfloat16}[args.dtype]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    g = torch.Generator(device=dev).manual_seed(args.seed)
    qkv = torch.randn((T, 3 * D), device=dev, dtype=torch.float32, generator=g).to(tdt)
    o = torch.empty((T, D), device=dev, dtype=tdt)
    cu_d = torch.as_tensor(cu).to(dev)
    ws_bytes = S.seer_layer_workspace_size(S.make_dims(D, H, dh, 256), args.dtype, T, len(lens))
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
    ms = _time(lambda: S.seer_attention(qkv, o, args.dtype, cu_d, None, len(lens), T, H, dh, ws, ws_bytes),
               args.warmup, args.reps)
    flops = 4.0 * D * float(np.sum(np.asarray(lens, dtype=np.float64) ** 2))
    return {"kernel": "attention", "lens": args.lens, "heads": H, "dtype": args.dtype, "ms": ms,
            "tflops": flops / (ms * 1e-3) / 1e12}


def linear(args) -> dict:
    dev = torch.device("cuda", 0)
    tdt = {"f16": torch.float16, "bf16": torch.bfloat16}[args.dtype]
    g = torch.Generator(device=dev).manual_seed(args.seed)
    a = (0.5 * torch.randn((args.M, args.K), device=dev, generator=g)).to(tdt)
    w = (0.02 * torch.randn((args.N, args.K), device=dev, generator=g)).to(tdt)
    c = torch.empty((args.M, args.N), device=dev, dtype=tdt)
    ms = _time(lambda: S.seer_linear(a, w, args.dtype, None, args.dtype, c, args.dtype, args.M, None, args.N, args.K),
               args.warmup, args.reps)
    return {"kernel": "linear", "M": args.M, "N": args.N, "K": args.K, "dtype": args.dtype, "ms": ms,
            "tflops": 2.0 * args.M * args.N * args.K / (ms * 1e-3) / 1e12}


def swiglu(args) -> dict:
    dev = torch.device("cuda", 0)
    tdt = {"f16": torch.float16, "bf16": torch.bfloat16}[args.dtype]
    g = torch.Generator(device=dev).manual_seed(args.seed)
    a = (0.5 * torch.randn((args.M, args.K), device=dev, generator=g)).to(tdt)
    wg = (0.02 * torch.randn((args.F, args.K), device=dev, generator=g)).to(tdt)
    wu = (0.02 * torch.randn((args.F, args.K), device=dev, generator=g)).to(tdt)
    act = torch.empty((args.M, args.F), device=dev, dtype=tdt)
    ms = _time(lambda: S.seer_swiglu(a, wg, wu, args.dtype, act, args.dtype, args.M, None, args.F, args.K),
               args.warmup, args.reps)
    return {"kernel": "swiglu", "M": args.M, "F": args.F, "K": args.K, "dtype": args.dtype, "ms": ms,
            "tflops": 4.0 * args.M * args.F * args.K / (ms * 1e-3) / 1e12}


def _ragged_lengths(batch, seed):
    rng = np.random.default_rng(seed)
    ctx = 729 * rng.integers(1, 6, batch) + rng.integers(32, 129, batch)
    return ctx, rng.integers(16, 401, batch) + 1


def pack(args) -> dict:
    dev = torch.device("cuda", 0)
    B, N, d = args.batch, args.window, args.d
    ctx, L = _ragged_lengths(B, args.seed)
    cu_full = np.concatenate([[0], np.cumsum(ctx + N)]).astype(np.int32)
    T = int(cu_full[-1])
    g = torch.Generator(device=dev).manual_seed(args.seed)
    x = torch.randn((T, d), device=dev, generator=g).to(torch.bfloat16)
    out = torch.empty_like(x)
    i32 = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32)).to(dev)
    cu_d, ctx_d, L_d = i32(cu_full), i32(ctx), i32(L)
    cu, kv = torch.empty(B + 1, dtype=torch.int32, device=dev), torch.empty(B, dtype=torch.int32, device=dev)
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=dev)
    p = S.make_params(0.0)
    ms = _time(lambda: S.seer_pack_ragged(x, "bf16", cu_d, ctx_d, L_d, B, d, N, T, p, out, cu, kv, meta),
               args.warmup, args.reps)
    rows = int(cu[-1].item())
    return {"kernel": "pack", "batch": B, "window": N, "d": d, "rows_kept": rows, "rows_full": T, "ms": ms,
            "gbs": 2.0 * rows * d * 2 / (ms * 1e-3) / 1e9}


def scan(args) -> dict:
    dev = torch.device("cuda", 0)
    B, N, F = args.batch, args.window, 12288
    _, L = _ragged_lengths(B, args.seed)
    rng = np.random.default_rng(args.seed)
    counts = rng.integers(100, 400, (B, N))
    for b in range(B):
        counts[b, int(L[b]) - 1:] += 6000                # planted plateau past the boundary
    c = torch.as_tensor(counts.astype(np.int32).ravel()).to(dev)
    Ls, Is = torch.empty(B, dtype=torch.int32, device=dev), torch.empty(B, dtype=torch.int32, device=dev)
    p = S.make_params(0.0)
    ms = _time(lambda: S.seer_snr_scan(c, B, N, F, p, Ls, Is), args.warmup, args.reps)
    return {"kernel": "scan", "batch": B, "window": N, "ms": ms, "gbs": B * N * 4 / (ms * 1e-3) / 1e9}


def norm(args) -> dict:
    dev = torch.device("cuda", 0)
    g = torch.Generator(device=dev).manual_seed(args.seed)
    x = torch.randn((args.M, args.d), device=dev, generator=g).to(torch.bfloat16)
    gain = torch.ones(args.d, device=dev, dtype=torch.float16)
    y = torch.empty((args.M, args.d), device=dev, dtype=torch.float16)
    ms = _time(lambda: S.seer_rmsnorm(x, "bf16", gain, y, "f16", args.M, None, args.d, 1e-5), args.warmup, args.reps)
    return {"kernel": "norm", "M": args.M, "d": args.d, "ms": ms, "gbs": args.M * args.d * 4 / (ms * 1e-3) / 1e9}


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    sub = ap.add_subparsers(dest="kernel", required=True)
    pa = sub.add_parser("attention")
    pa.add_argument("--lens", default="3100x8", help="segment lengths, e.g. 3100x8 or 11900x4,500")
    pa.add_argument("--heads", type=int, default=32)
    pl = sub.add_parser("linear")
    pl.add_argument("--M", type=int, default=35194)
    pl.add_argument("--N", type=int, default=12288)
    pl.add_argument("--K", type=int, default=4096)
    pw = sub.add_parser("swiglu")
    pw.add_argument("--M", type=int, default=35194)
    pw.add_argument("--F", type=int, default=12288)
    pw.add_argument("--K", type=int, default=4096)
    for p in (pa, pl, pw):
        p.add_argument("--dtype", default="f16", choices=["f16", "bf16"])
        p.add_argument("--warmup", type=int, default=3)
        p.add_argument("--reps", type=int, default=10)
        p.add_argument("--seed", type=int, default=0)
    pp = sub.add_parser("pack")
    pp.add_argument("--batch", type=int, default=16)
    pp.add_argument("--window", type=int, default=1024)
    pp.add_argument("--d", type=int, default=4096)
    ps = sub.add_parser("scan")
    ps.add_argument("--batch", type=int, default=16)
    ps.add_argument("--window", type=int, default=1024)
    pn = sub.add_parser("norm")
    pn.add_argument("--M", type=int, default=35194)
    pn.add_argument("--d", type=int, default=4096)
    for q in (pp, ps, pn):
        q.add_argument("--warmup", type=int, default=3)
        q.add_argument("--reps", type=int, default=10)
        q.add_argument("--seed", type=int, default=0)
    args = ap.parse_args(argv)
    res = {"attention": attention, "linear": linear, "pack": pack, "scan": scan, "norm": norm, "swiglu": swiglu}[args.kernel](args)
    assert S.seer_check_device() == 0, "a kernel recorded a device-side error"
    print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
