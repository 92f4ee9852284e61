"""Seeded synthetic inputs shaped like the Seer workloads.

This module only *generates data*: sequence lengths, planted-boundary hidden
states and random-init layer weights.  It holds none of the method's
arithmetic (no sparsity counts, no boundary scan, no routing, no layer math),
so both the CPU oracle and the CUDA path can consume the same inputs without
sharing any computation.

Recipe (one numpy PCG64 ``SeedSequence`` per workload, seed = 1000 + index,
with independent child streams for lengths, hidden states, the suffix noise
and the weights):

* visual-prefix and prompt rows, and response rows before the planted
  boundary ``b``: i.i.d. N(0, 1);
* response rows at positions >= ``b``: one shared EOS-like vector
  ``e = 0.1 * z`` (``z ~ N(0, I)``) plus i.i.d. N(0, 0.05^2) noise, so the
  suffix sits near zero after the MLP (the activation behaviour the paper
  describes for padding tokens, Sec. 1 and Sec. 3.2);
* weights N(0, 0.02^2); RMSNorm gains 1.  Layer ``l`` of a stack draws from
  ``SeedSequence([seed, 7, l])`` so any layer can be regenerated alone.

Values are rounded once to the workload's storage type (bf16 or fp32) with
torch's converter; the float32 arrays returned here are exactly the values the
GPU receives, so input rounding is never an error source.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, Optional

import numpy as np

__all__ = [
    "Workload", "WORKLOADS", "workload", "tiny_workload", "Lengths", "lengths",
    "hidden_full", "layer_weights", "round_storage", "with_lengths",
]


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shape and planted-boundary recipe of one synthetic workload."""
    index: int
    name: str
    dtype: str            # "f32" or "bf16": storage type of every tensor
    d: int                # hidden size
    n_heads: int
    head_dim: int
    d_ff: int             # SwiGLU intermediate width F
    batch: int
    window: int           # generation window N
    n_layers: int
    act_eps: float        # absolute near-zero threshold for the sparsity count
    visual: tuple         # ("fixed", n) or ("mult", base, kmin, kmax)
    prompt: tuple         # ("fixed", n) or ("uniform", lo, hi)
    boundary: tuple       # ("fixed", b) | ("uniform", lo, hi) | ("loguniform", lo, hi) | ("pareto", alpha, scale, lo, hi)
    steps: int = 1        # denoising steps timed (stack workload)
    seed_offset: int = 1000

    @property
    def seed(self) -> int:
        return self.seed_offset + self.index


WORKLOADS: Dict[int, Workload] = {
    0: Workload(0, "tiny-f32", "f32", 256, 4, 64, 768, 1, 128, 1, 3e-4,
                ("fixed", 64), ("fixed", 16), ("fixed", 40)),
    1: Workload(1, "llada8b-layer-b1", "bf16", 4096, 32, 128, 12288, 1, 256, 1, 5e-3,
                ("fixed", 729), ("fixed", 64), ("fixed", 48)),
    2: Workload(2, "llada8b-layer-ragged-b16", "bf16", 4096, 32, 128, 12288, 16, 1024, 1, 5e-3,
                ("mult", 729, 1, 5), ("uniform", 32, 128), ("uniform", 16, 400)),
    3: Workload(3, "llada8b-stack32-b8", "bf16", 4096, 32, 128, 12288, 8, 512, 32, 5e-3,
                ("fixed", 2916), ("fixed", 96), ("loguniform", 24, 480), steps=64),
    4: Workload(4, "video-layer-b4", "bf16", 4096, 32, 128, 12288, 4, 2048, 1, 5e-3,
                ("fixed", 11664), ("fixed", 128), ("pareto", 1.5, 32, 32, 1800)),
}


def workload(index: int) -> Workload:
    return WORKLOADS[index]


def tiny_workload(name: str = "tiny-bf16", *, dtype: str = "bf16", d: int = 256, n_heads: int = 2,
                  head_dim: int = 128, d_ff: int = 768, batch: int = 3, window: int = 160,
                  visual=("mult", 96, 1, 3), prompt=("uniform", 5, 40), boundary=("uniform", 10, 150),
                  act_eps: Optional[float] = None, seed: int = 7, n_layers: int = 1) -> Workload:
    """A small workload for parity tests: several tiles and ragged tails."""
    if act_eps is None:
        act_eps = 3e-4 if d <= 512 else 5e-3
    return Workload(seed, name, dtype, d, n_heads, head_dim, d_ff, batch, window, n_layers, act_eps,
                    visual, prompt, boundary, seed_offset=0)


@dataclasses.dataclass
class Lengths:
    visual: np.ndarray    # int64 [B]
    prompt: np.ndarray    # int64 [B]
    boundary: np.ndarray  # int64 [B]: first planted suffix position (0-based) in the window
    window: int

    @property
    def ctx(self) -> np.ndarray:
        return self.visual + self.prompt

    @property
    def full(self) -> np.ndarray:
        return self.ctx + self.window


def _streams(wl: Workload):
    ss = np.random.SeedSequence(wl.seed)
    lens, hid, noise = ss.spawn(3)
    return (np.random.Generator(np.random.PCG64(lens)), np.random.Generator(np.random.PCG64(hid)),
            np.random.Generator(np.random.PCG64(noise)))


def _draw(spec, rng, B):
    kind = spec[0]
    if kind == "fixed":
        return np.full(B, spec[1], dtype=np.int64)
    if kind == "mult":
        _, base, kmin, kmax = spec
        return base * rng.integers(kmin, kmax + 1, size=B)
    if kind == "uniform":
        _, lo, hi = spec
        return rng.integers(lo, hi + 1, size=B).astype(np.int64)
    if kind == "loguniform":
        _, lo, hi = spec
        return np.floor(np.exp(rng.uniform(np.log(lo), np.log(hi), size=B))).astype(np.int64)
    if kind == "pareto":
        _, alpha, scale, lo, hi = spec
        return np.clip(np.floor(scale * (1.0 + rng.pareto(alpha, size=B))), lo, hi).astype(np.int64)
    raise ValueError(spec)


def lengths(wl: Workload) -> Lengths:
    rl, _, _ = _streams(wl)
    B = wl.batch
    return Lengths(_draw(wl.visual, rl, B), _draw(wl.prompt, rl, B), _draw(wl.boundary, rl, B), wl.window)


def with_lengths(wl: Workload, lens: Lengths, **changes) -> Lengths:
    """Copy of ``lens`` with some fields replaced (used by edge-case tests)."""
    out = Lengths(lens.visual.copy(), lens.prompt.copy(), lens.boundary.copy(), lens.window)
    for k, v in changes.items():
        setattr(out, k, np.asarray(v, dtype=np.int64) if k != "window" else int(v))
    return out


def round_storage(a: np.ndarray, dtype: str) -> np.ndarray:
    """Round to the storage type and return float32 holding exactly those values."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    if dtype == "f32":
        return a
    import torch
    return torch.from_numpy(a).to(torch.bfloat16).to(torch.float32).numpy()


def hidden_full(wl: Workload, lens: Optional[Lengths] = None):
    """Full-window stack input, packed over sequences.

    Returns ``(x_full, cu_full, resp_start)``: ``x_full`` float32 [sum(ctx_i+N), d]
    with rows ``[visual | prompt | window]`` per sequence, ``cu_full`` int32 [B+1]
    row offsets, and ``resp_start`` int32 [B] = row of each window's first token.
    """
    if lens is None:
        lens = lengths(wl)
    _, rh, rn = _streams(wl)
    d, N = wl.d, lens.window
    full = lens.full
    cu = np.zeros(len(full) + 1, dtype=np.int64)
    cu[1:] = np.cumsum(full)
    x = rh.standard_normal((int(cu[-1]), d), dtype=np.float32)
    eos = (0.1 * rn.standard_normal(d, dtype=np.float32)).astype(np.float32)
    resp = (cu[:-1] + lens.ctx).astype(np.int64)
    for i in range(len(full)):
        b = int(lens.boundary[i])
        if b < N:
            rows = slice(int(resp[i]) + b, int(resp[i]) + N)
            x[rows] = eos[None, :] + 0.05 * rn.standard_normal((N - b, d), dtype=np.float32)
    x = round_storage(x, wl.dtype)
    return x, cu.astype(np.int32), resp.astype(np.int32)


def _bf16_bits_of_layer(args):
    wl, layer = args
    w = layer_weights(wl, layer)
    return layer, {k: (np.ascontiguousarray(v).view(np.uint32) >> 16).astype(np.uint16) for k, v in w.items()}


def stack_weights_bf16_bits(wl: Workload, layers, workers: Optional[int] = None):
    """Yield ``(layer, {name: uint16 bf16 bit patterns})`` for the given layers,
    generated in a spawn-started process pool (each layer has its own seeded
    stream, so the values equal :func:`layer_weights`).  bf16 workloads only."""
    import concurrent.futures
    import multiprocessing
    import os
    assert wl.dtype == "bf16"
    layers = list(layers)
    n = workers or max(1, min(len(layers), (os.cpu_count() or 2) // 2, 16))
    ctx = multiprocessing.get_context("spawn")
    with concurrent.futures.ProcessPoolExecutor(max_workers=n, mp_context=ctx) as ex:
        for item in ex.map(_bf16_bits_of_layer, [(wl, l) for l in layers]):
            yield item


def layer_weights(wl: Workload, layer: int = 0) -> Dict[str, np.ndarray]:
    """Random-init weights of one block, nn.Linear layout [out, in]."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence([wl.seed, 7, layer])))
    d, F = wl.d, wl.d_ff

    def w(o, i):
        return round_storage(0.02 * rng.standard_normal((o, i), dtype=np.float32), wl.dtype)

    out = {"wq": w(d, d), "wk": w(d, d), "wv": w(d, d), "wo": w(d, d),
           "wg": w(F, d), "wu": w(F, d), "wd": w(d, F)}
    out["g_attn"] = np.ones(d, dtype=np.float32)
    out["g_mlp"] = np.ones(d, dtype=np.float32)
    return out
