"""Routing ablation on one GPU: layer time under the micro-bucket router (Sec. 3.4,
Eqs. 3-4) as the padding-waste threshold tau_pad and the batch size vary, next
to the naive batch-max padding and the untruncated window.

    python -m paper_2607_14557_gb300.routing_sweep [--batches 16,32,64,128] [--taus 0.1,0.2,...,0.9]
                                                   [--bucket-mins 8,16,32,64]

Lengths follow the ragged 8B-layer workload (visual 729k tokens with k in
1..5, prompt 32..128, window 1024, planted boundary b in 16..400; L* = b + 1);
hidden states and weights are random device tensors (the timing does not
depend on their values, and detection is not part of this sweep).  For every
(batch, tau_pad) the route is built by the library's pack kernel and the
layer is timed with CUDA events over `--reps` calls; one JSON line per point.
tau_pad < 0 gives the all-varlen layout (no bucket padding).  --bucket-mins sets the
smallest micro-bucket of the doubling bucket set (the paper's set starts at 8).
"""
from __future__ import annotations

import argparse
import dataclasses
import json

import numpy as np
import torch

from . import driver as D
from . import seer as S


def _lengths(batch: int, seed: int):
    rng = np.random.default_rng(seed)
    visual = 729 * rng.integers(1, 6, batch)
    prompt = rng.integers(32, 129, batch)
    boundary = rng.integers(16, 401, batch)
    return visual + prompt, boundary + 1


def _weights(d, F, dev, seed):
    g = torch.Generator(device=dev).manual_seed(seed)
    r = lambda *shape: (0.02 * torch.randn(shape, device=dev, generator=g)).to(torch.float16)
    run = {"w_qkv": r(3 * d, d), "w_o": r(d, d), "w_gate": r(F, d), "w_up": r(F, d), "w_down": r(d, F),
           "g_attn": torch.ones(d, device=dev, dtype=torch.float16),
           "g_mlp": torch.ones(d, device=dev, dtype=torch.float16)}
    return D.LayerWeights(run, run)


def _time(fn, reps):
    fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        fn()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def sweep(batch, taus, reps, d=4096, H=32, F=12288, N=1024, seed=0, bucket_min=8):
    dev = torch.device("cuda", 0)
    ctx, L = _lengths(batch, seed)
    full = ctx + N
    cu_full = np.concatenate([[0], np.cumsum(full)]).astype(np.int32)
    T_full = int(cu_full[-1])
    g = torch.Generator(device=dev).manual_seed(seed + 1)
    x_full = torch.randn((T_full, d), device=dev, generator=g).to(torch.bfloat16)
    W = _weights(d, F, dev, seed + 2)
    dims = S.make_dims(d, H, d // H, F)
    i32 = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32)).to(dev)
    cu_d, ctx_d, L_d = i32(cu_full), i32(ctx), i32(L)
    flops = lambda seg, kv: float(8.0 * seg.sum() * d * d + 6.0 * seg.sum() * d * F + 4.0 * d * np.sum(seg * kv))
    out = []

    def point(tau):
        path = D.SeerPath(dims, "bf16", batch, N, T_full, S.make_params(0.0, tau_pad=tau, bucket_min=bucket_min), dev)
        path.L_star.copy_(L_d)
        path.pack(x_full, cu_d, ctx_d)
        route = path.route()
        seg = np.diff(path.cu.cpu().numpy()).astype(np.float64)
        kv = path.kv.cpu().numpy().astype(np.float64)
        ms = _time(lambda: path.layer(W), reps)
        return path, route, seg, kv, ms

    valid = flops(ctx + L, ctx + L)
    path0 = None
    for tau in taus:
        path, route, seg, kv, ms = point(tau)
        paths = [grp["path"] for grp in route["groups"]]
        out.append({"batch": batch, "tau_pad": tau, "bucket_min": bucket_min, "ms": ms, "tokens_executed": int(seg.sum()),
                    "pad_rows": route["pad_rows"], "groups": len(route["groups"]),
                    "static_groups": paths.count(0), "varlen_groups": paths.count(1), "eager_groups": paths.count(2),
                    "flops_executed_over_valid": flops(seg, kv) / valid})
        path0 = path
    # comparators on the same lengths: naive batch-max padding and the untruncated window
    xn, cun, kvn, Tn = path0.naive_pad_inputs(x_full, cu_d, ctx_d)
    yn = torch.empty((Tn, d), device=dev, dtype=torch.bfloat16)
    ms_naive = _time(lambda: path0.layer(W, x=xn, y=yn, cu=cun, kv=kvn, T_cap=Tn), reps)
    del xn, yn
    y_full = torch.empty((T_full, d), device=dev, dtype=torch.bfloat16)
    ms_pad = _time(lambda: path0.padded_forward(x_full, cu_d, W, y_full), reps)
    seg_n = np.diff(cun.cpu().numpy()).astype(np.float64)
    out.append({"batch": batch, "comparator": "naive_pad", "ms": ms_naive, "tokens_executed": int(seg_n.sum()),
                "flops_executed_over_valid": flops(seg_n, kvn.cpu().numpy().astype(np.float64)) / valid})
    out.append({"batch": batch, "comparator": "untruncated", "ms": ms_pad, "tokens_executed": T_full,
                "flops_executed_over_valid": flops(full.astype(np.float64), full.astype(np.float64)) / valid})
    return out


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--batches", default="16,32,64,128")
    ap.add_argument("--taus", default="-1,0.1,0.2,0.3,0.4,0.5,0.6,0.7,0.8,0.9")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--bucket-mins", default="8")
    args = ap.parse_args(argv)
    for bm in [int(v) for v in args.bucket_mins.split(",")]:
        for b in [int(v) for v in args.batches.split(",")]:
            for line in sweep(b, [float(t) for t in args.taus.split(",")], args.reps, bucket_min=bm):
                print(json.dumps(line), flush=True)
        assert S.seer_check_device() == 0
        torch.cuda.empty_cache()


if __name__ == "__main__":
    main()
