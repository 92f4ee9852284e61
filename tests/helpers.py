"""Shared helpers of the GPU parity tests (marshalling and tolerance checks only)."""
import numpy as np
import torch

import synth

BF16_ATOL = 1e-2
BF16_RTOL = 1e-2
F32_ATOL = 1e-4
F32_RTOL = 1e-4
COUNT_TOL_FRAC = 0.005    # near-zero counts within 0.5% of the intermediate width F


def cuda():
    return torch.device("cuda", 0)


def tdtype(dtype: str):
    return {"bf16": torch.bfloat16, "f16": torch.float16, "f32": torch.float32}[dtype]


def to_dev(a, dtype: str):
    """Upload values that are already representable in the storage type."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.to(tdtype(dtype)).to(cuda())


def i32(a):
    return torch.as_tensor(np.asarray(a, dtype=np.int32)).to(cuda())


def host(t):
    return t.detach().float().cpu().numpy().astype(np.float64)


def tol(dtype):
    return (F32_ATOL, F32_RTOL) if dtype == "f32" else (BF16_ATOL, BF16_RTOL)


def check_close(got, ref, dtype, what=""):
    """|got - ref| <= atol + rtol * |ref| element by element (the parity bar)."""
    atol, rtol = tol(dtype)
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    err = np.abs(got - ref)
    bad = err > atol + rtol * np.abs(ref)
    if bad.any() or not np.isfinite(got).all():
        idx = np.argwhere(bad)[:8]
        raise AssertionError(f"{what}: {int(bad.sum())}/{bad.size} elements outside {atol}+{rtol}|ref|; "
                             f"max err {np.nanmax(err):.4g}; first bad {idx.tolist()}; "
                             f"finite={np.isfinite(got).all()}")
    return float(err.max()) if err.size else 0.0


def check_counts(got, ref, F, what=""):
    """|got - ref| <= 0.5% of F for every token's near-zero count (the parity
    bar of the sparsity counts); returns the largest difference."""
    got = np.asarray(got, dtype=np.int64)
    ref = np.asarray(ref, dtype=np.int64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    diff = np.abs(got - ref)
    worst = int(diff.max()) if diff.size else 0
    if worst > COUNT_TOL_FRAC * F:
        idx = np.argwhere(diff > COUNT_TOL_FRAC * F)[:8]
        raise AssertionError(f"{what}: max |count - oracle| = {worst} > {COUNT_TOL_FRAC * F:g} (0.5% of F={F}) at "
                             f"{int((diff > COUNT_TOL_FRAC * F).sum())}/{diff.size} tokens; first {idx.tolist()}")
    return worst


def layer_weight_tensors(wl, w):
    """Device weights of one layer: model dtype copies plus, for a bf16 model,
    the f16 copies the layer runs on (made by the library's converter)."""
    from paper_2607_14557_gb300 import seer as S
    dt = wl.dtype
    model = {
        "w_qkv": to_dev(np.concatenate([w["wq"], w["wk"], w["wv"]], axis=0), dt),
        "w_o": to_dev(w["wo"], dt), "w_gate": to_dev(w["wg"], dt), "w_up": to_dev(w["wu"], dt),
        "w_down": to_dev(w["wd"], dt), "g_attn": to_dev(w["g_attn"], dt), "g_mlp": to_dev(w["g_mlp"], dt),
    }
    if dt == "f32":
        return model, model
    layer = {}
    for k, t in model.items():
        dst = torch.empty(t.shape, dtype=torch.float16, device=t.device)
        S.seer_convert(t, "bf16", dst, "f16", t.numel())
        layer[k] = dst
    return model, layer


def weights_struct(layer):
    from paper_2607_14557_gb300 import seer as S
    return S.make_weights(*[layer[k] for k in ("w_qkv", "w_o", "w_gate", "w_up", "w_down", "g_attn", "g_mlp")])
