"""fp64 numpy oracle of the Seer hot path.  Test infrastructure only.

Readings of the paper that this file takes:

* The "MLP activation" whose sparsity is measured is the SwiGLU intermediate
  ``a = SiLU(x Wg^T) * (x Wu^T)`` (the input of the down projection); a value
  is "near zero" when ``|a| < eps`` (strict), ``eps`` an absolute threshold
  the paper does not print (Sec. 1, Sec. 3.2).
* The sparsity array ``S`` is 0-based here.  Window ``W_i = s_i .. s_{i+w-1}``
  is tested against ``s_{i-1}`` for ``i = 1 .. N-w``; the first (smallest)
  ``i`` that passes is ``i*``; ``L* = i* + 1``; no hit keeps the whole window
  (``L* = N``) (Sec. 3.3).
* ``s_i = c_i / F`` and the two tests are evaluated in IEEE fp64 in exactly
  this order: ``jump = min(W) - s_{i-1}``, ``noise = max(W) - min(W)``,
  ``jump >= tau_jump`` and ``noise <= gamma * jump``.
* Micro-buckets are the powers of two from 8 below ``N`` plus ``N`` itself;
  a sequence joins the smallest bucket ``>= L*``; a group is the set of
  sequences sharing a bucket (Sec. 3.4).
* The block is a pre-norm LLaMA-style layer (RMSNorm, eps 1e-5; MHA without
  bias; SwiGLU MLP), attention scaled by ``1/sqrt(head_dim)`` (Eq. 7 prints
  ``sqrt(d)``, read as the per-head width).  The paper names no positional
  scheme; a rotary embedding of queries and keys is optional (off unless
  ``rope_theta > 0``), positions restarting at 0 in every sequence.
* A "BF16 layer" stores every tensor that crosses an op boundary in bf16:
  ``xn, q, k, v, o, h, hn, a, y`` are rounded to the storage type after being
  computed exactly (fp64) from already-rounded inputs.
"""
from __future__ import annotations

import math
from typing import Callable, Dict, List, Optional, Sequence

import numpy as np

__all__ = [
    "round_bf16", "round_f32", "rounding_for", "silu", "swiglu_activation", "sparsity_counts",
    "snr_boundary", "snr_boundaries", "bucket_set", "bucket_of", "padding_waste_ratio", "route",
    "segment_layout", "pack_rows", "rmsnorm", "rope", "attention_weights", "attention", "layer_forward_segment",
    "layer_forward_packed", "layer_forward_rows", "kv_prefill", "layer_forward_cached", "PATH_STATIC", "PATH_VARLEN",
    "PATH_EAGER",
]


# --------------------------------------------------------------------------
# storage rounding
# --------------------------------------------------------------------------
def round_bf16(x) -> np.ndarray:
    """Round fp64 values to the nearest bf16 value (ties to even), in fp64.

    bf16 keeps 8 significant bits and fp32's exponent range; below the
    smallest normal (2^-126) the spacing is fixed at 2^-133.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.empty_like(x)
    finite = np.isfinite(x)
    out[~finite] = x[~finite]
    xf = x[finite]
    m, e = np.frexp(xf)                      # xf = m * 2^e, 0.5 <= |m| < 1
    normal = np.abs(xf) >= 2.0 ** -126
    q = np.where(normal, np.ldexp(np.rint(np.ldexp(m, 8)), e - 8),
                 np.rint(xf / 2.0 ** -133) * 2.0 ** -133)
    # values that round past the largest finite bf16 become infinity
    big = np.abs(q) > 3.3895313892515355e38
    q = np.where(big, np.copysign(np.inf, xf), q)
    out[finite] = q
    return out


def round_f32(x) -> np.ndarray:
    return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)


def rounding_for(dtype: Optional[str]) -> Callable[[np.ndarray], np.ndarray]:
    if dtype == "bf16":
        return round_bf16
    if dtype == "f32":
        return round_f32
    return lambda a: np.asarray(a, dtype=np.float64)


# --------------------------------------------------------------------------
# Sec. 3.2 / Sec. 3.3: step-0 MLP sparsity and the SNR boundary criterion
# --------------------------------------------------------------------------
def silu(x):
    x = np.asarray(x, dtype=np.float64)
    return x / (1.0 + np.exp(-x))


def swiglu_activation(x, wg, wu) -> np.ndarray:
    """SwiGLU intermediate a = SiLU(x Wg^T) * (x Wu^T) for rows of x (Sec. 3.2)."""
    x = np.asarray(x, dtype=np.float64)
    g = x @ np.asarray(wg, dtype=np.float64).T
    u = x @ np.asarray(wu, dtype=np.float64).T
    return silu(g) * u


def sparsity_counts(x, wg, wu, eps: float) -> np.ndarray:
    """Per row, the number of SwiGLU activations with |a| < eps (Sec. 1, Sec. 3.2)."""
    a = swiglu_activation(x, wg, wu)
    return (np.abs(a) < eps).sum(axis=-1).astype(np.int64)


def snr_boundary(counts: Sequence[int], F: int, tau_jump: float = 0.03, gamma: float = 0.6,
                 window: int = 3):
    """SNR-aware boundary detection over one sparsity array (Sec. 3.3).

    ``counts[i]`` near-zero activations of response token i out of ``F``.
    Returns ``(i_star, L_star)``; ``i_star = -1`` and ``L_star = N`` when no
    position passes both the signal test and the plateau (SNR) test.
    """
    s = [float(c) / float(F) for c in counts]
    N = len(s)
    for i in range(1, N - window + 1):
        w = s[i:i + window]
        lo, hi = min(w), max(w)
        jump = lo - s[i - 1]
        noise = hi - lo
        if jump >= tau_jump and noise <= gamma * jump:
            return i, i + 1
    return -1, N


def snr_boundaries(counts2d, F: int, tau_jump: float = 0.03, gamma: float = 0.6, window: int = 3):
    res = [snr_boundary(row, F, tau_jump, gamma, window) for row in np.asarray(counts2d)]
    return (np.array([r[0] for r in res], dtype=np.int64), np.array([r[1] for r in res], dtype=np.int64))


# --------------------------------------------------------------------------
# Sec. 3.4: static micro-buckets, padding waste ratio, three execution paths
# --------------------------------------------------------------------------
PATH_STATIC, PATH_VARLEN, PATH_EAGER = 0, 1, 2


def bucket_set(n_max: int, b_min: int = 8) -> List[int]:
    """Static micro-buckets {8, 16, 32, ..., N_max} (Sec. 3.4); ``b_min`` is
    the smallest bucket (the paper's set starts at 8), each next one doubles."""
    out, b = [], int(b_min)
    while b < n_max:
        out.append(b)
        b *= 2
    out.append(n_max)
    return out


def bucket_of(L: int, n_max: int, b_min: int = 8) -> int:
    for b in bucket_set(n_max, b_min):
        if L <= b:
            return b
    raise ValueError(f"L*={L} exceeds the window {n_max}")


def padding_waste_ratio(L_stars: Sequence[int], B_G: int) -> float:
    """Eq. 4: rho = 1 - sum_i L*_i / (|G| * B_G)."""
    return 1.0 - float(sum(int(v) for v in L_stars)) / float(len(L_stars) * B_G)


def route(L_star: Sequence[int], n_max: int, tau_pad: float = 0.2, eager_max_bucket: int = 4, bucket_min: int = 8):
    """Group sequences by micro-bucket and pick each group's path (Sec. 3.4).

    Returns a list of dicts (ascending bucket) with keys ``bucket``,
    ``members`` (sequence indices), ``rho`` and ``path`` (0 static-graph,
    1 bucket-varlen-graph, 2 bucket-varlen-eager).
    """
    groups: Dict[int, List[int]] = {}
    for i, L in enumerate(L_star):
        groups.setdefault(bucket_of(int(L), n_max, bucket_min), []).append(i)
    out = []
    for b in sorted(groups):
        mem = groups[b]
        rho = padding_waste_ratio([L_star[i] for i in mem], b)
        if b <= eager_max_bucket or len(mem) == 1:
            path = PATH_EAGER
        elif rho <= tau_pad:
            path = PATH_STATIC
        else:
            path = PATH_VARLEN
        out.append({"bucket": b, "members": mem, "rho": rho, "path": path})
    return out


# --------------------------------------------------------------------------
# Sec. 3.5: compaction layout
# --------------------------------------------------------------------------
def segment_layout(ctx_len, L_star, n_max: int, tau_pad: float = 0.2, eager_max_bucket: int = 4, bucket_min: int = 8):
    """Rows kept per sequence after truncation and routing (Sec. 3.4-3.5).

    A static-graph group pads each response to the group's bucket (those rows
    are computed but masked as keys); the other paths keep exactly
    ``ctx_i + L*_i`` rows.  Returns ``(seg_len, kv_len, cu)``.
    """
    ctx_len = np.asarray(ctx_len, dtype=np.int64)
    L_star = np.asarray(L_star, dtype=np.int64)
    seg = ctx_len + L_star
    for g in route(L_star, n_max, tau_pad, eager_max_bucket, bucket_min):
        if g["path"] == PATH_STATIC:
            for i in g["members"]:
                seg[i] = ctx_len[i] + g["bucket"]
    kv = ctx_len + L_star
    cu = np.zeros(len(seg) + 1, dtype=np.int64)
    cu[1:] = np.cumsum(seg)
    return seg, kv, cu


def pack_rows(x_full, cu_full, seg_len) -> np.ndarray:
    """Keep the first seg_len[i] rows of each sequence, back to back (Sec. 3.5)."""
    parts = [np.asarray(x_full)[int(cu_full[i]):int(cu_full[i]) + int(seg_len[i])]
             for i in range(len(seg_len))]
    return np.concatenate(parts, axis=0) if parts else np.zeros((0, np.asarray(x_full).shape[1]))


# --------------------------------------------------------------------------
# Sec. 3.1 / Sec. 3.6: the denoising layer over the retained context
# --------------------------------------------------------------------------
def rmsnorm(x, g, eps: float = 1e-5) -> np.ndarray:
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(g, dtype=np.float64)


def rope(x, positions, n_heads: int, theta: float) -> np.ndarray:
    """Rotary position embedding of every head of ``x`` [L, H*dh].

    Not from the paper (which names no positional scheme): the rotation of
    RoFormer (Su et al., 2021) in the half-split layout of LLaMA checkpoints.
    Pair ``i < dh/2`` of a head is ``(x_i, x_{i+dh/2})``; it is rotated by
    the angle ``pos * theta^(-2i/dh)``.  ``theta <= 0`` leaves ``x`` as is.
    """
    x = np.asarray(x, dtype=np.float64)
    if theta <= 0:
        return x.copy()
    dh = x.shape[1] // n_heads
    half = dh // 2
    ang = np.asarray(positions, dtype=np.float64)[:, None] * float(theta) ** (-2.0 * np.arange(half) / dh)
    c, s = np.cos(ang), np.sin(ang)
    out = np.empty_like(x)
    for h in range(n_heads):
        a = x[:, h * dh:h * dh + half]
        b = x[:, h * dh + half:(h + 1) * dh]
        out[:, h * dh:h * dh + half] = a * c - b * s
        out[:, h * dh + half:(h + 1) * dh] = b * c + a * s
    return out


def attention_weights(q, k) -> np.ndarray:
    """Eqs. 6-7: A[i, j] = exp(e_ij) / sum_u exp(e_iu), e_ij = q_i . k_j / sqrt(dh).

    Bidirectional: every query sees every key of the sequence.
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    e = (q @ k.T) / math.sqrt(q.shape[-1])
    e = e - e.max(axis=-1, keepdims=True)
    p = np.exp(e)
    return p / p.sum(axis=-1, keepdims=True)


def attention(q, k, v, n_heads: int) -> np.ndarray:
    """Multi-head bidirectional attention; q [Lq, H*dh], k/v [Lk, H*dh]."""
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    dh = q.shape[1] // n_heads
    out = np.empty((q.shape[0], n_heads * dh))
    for h in range(n_heads):
        c = slice(h * dh, (h + 1) * dh)
        out[:, c] = attention_weights(q[:, c], k[:, c]) @ v[:, c]
    return out


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def layer_forward_segment(x, w: Dict[str, np.ndarray], n_heads: int, *, kv_len: Optional[int] = None,
                          dtype: Optional[str] = None, rms_eps: float = 1e-5, count_rows=None,
                          act_eps: float = 0.0, return_parts: bool = False, rope_theta: float = 0.0):
    """One pre-norm block over one sequence (Eq. 9-10: keys = retained rows).

    ``x`` [L, d] rows of one sequence.  Only the first ``kv_len`` rows serve
    as keys/values (the rest are bucket padding); every row is a query.
    ``count_rows``: optional row indices whose SwiGLU activations are counted
    against ``act_eps`` (the step-0 detection hook).  ``rope_theta > 0``
    rotates q and k (:func:`rope`) at their row positions in the sequence.
    """
    R = rounding_for(dtype)
    x = _f64(x)
    L = x.shape[0]
    kv = L if kv_len is None else int(kv_len)
    xn = R(rmsnorm(x, w["g_attn"], rms_eps))
    q = R(rope(xn @ _f64(w["wq"]).T, np.arange(L), n_heads, rope_theta))
    k = R(rope(xn[:kv] @ _f64(w["wk"]).T, np.arange(kv), n_heads, rope_theta))
    v = R(xn[:kv] @ _f64(w["wv"]).T)
    o = R(attention(q, k, v, n_heads))
    h = R(x + o @ _f64(w["wo"]).T)
    hn = R(rmsnorm(h, w["g_mlp"], rms_eps))
    a_exact = swiglu_activation(hn, w["wg"], w["wu"])
    a = R(a_exact)
    y = R(h + a @ _f64(w["wd"]).T)
    counts = None
    if count_rows is not None:
        counts = (np.abs(a_exact[np.asarray(count_rows, dtype=np.int64)]) < act_eps).sum(-1).astype(np.int64)
    if return_parts:
        return {"xn": xn, "q": q, "k": k, "v": v, "o": o, "h": h, "hn": hn, "a": a, "y": y, "counts": counts}
    return (y, counts) if count_rows is not None else y


def layer_forward_packed(x_packed, cu, w, n_heads: int, *, kv_len=None, dtype=None, rms_eps=1e-5,
                         rope_theta: float = 0.0):
    """Apply :func:`layer_forward_segment` to each packed segment independently."""
    x_packed = _f64(x_packed)
    y = np.empty_like(x_packed)
    for i in range(len(cu) - 1):
        a, b = int(cu[i]), int(cu[i + 1])
        if b > a:
            y[a:b] = layer_forward_segment(x_packed[a:b], w, n_heads, dtype=dtype, rms_eps=rms_eps,
                                           kv_len=None if kv_len is None else int(kv_len[i]), rope_theta=rope_theta)
    return y


def layer_forward_rows(x_seg, w, n_heads: int, rows, *, kv_len=None, dtype=None, rms_eps=1e-5, act_eps=None,
                       rope_theta: float = 0.0):
    """Outputs of selected rows of one segment (keys/values from all kept rows).

    Same arithmetic as :func:`layer_forward_segment`, restricted to the query
    rows ``rows``; used where the full segment is too large for the oracle.
    With ``act_eps`` set, also returns the near-zero SwiGLU counts of those
    rows (the step-0 detection hook): ``(y_rows, counts)``.
    """
    R = rounding_for(dtype)
    x = _f64(x_seg)
    kv = x.shape[0] if kv_len is None else int(kv_len)
    rows = np.asarray(rows, dtype=np.int64)
    xn_kv = R(rmsnorm(x[:kv], w["g_attn"], rms_eps))
    k = R(rope(xn_kv @ _f64(w["wk"]).T, np.arange(kv), n_heads, rope_theta))
    v = R(xn_kv @ _f64(w["wv"]).T)
    xr = x[rows]
    xn = R(rmsnorm(xr, w["g_attn"], rms_eps))
    q = R(rope(xn @ _f64(w["wq"]).T, rows, n_heads, rope_theta))
    o = R(attention(q, k, v, n_heads))
    h = R(xr + o @ _f64(w["wo"]).T)
    hn = R(rmsnorm(h, w["g_mlp"], rms_eps))
    a_exact = swiglu_activation(hn, w["wg"], w["wu"])
    y = R(h + R(a_exact) @ _f64(w["wd"]).T)
    if act_eps is None:
        return y
    return y, (np.abs(a_exact) < act_eps).sum(-1).astype(np.int64)


# --------------------------------------------------------------------------
# Prefix key/value caching combined with truncation (Sec. 4, Table 7: Seer
# composes with KV caching of the visual + prompt prefix)
# --------------------------------------------------------------------------
def kv_prefill(x_prefix, w, n_heads: int, *, dtype=None, rms_eps=1e-5):
    """Keys and values of a sequence's prefix rows for one layer (the cache):
    the same normalisation and projections as the block, applied to the
    prefix rows only.  Returns ``(k, v)``, each [ctx, H*dh]."""
    R = rounding_for(dtype)
    xn = R(rmsnorm(_f64(x_prefix), w["g_attn"], rms_eps))
    return R(xn @ _f64(w["wk"]).T), R(xn @ _f64(w["wv"]).T)


def layer_forward_cached(x_resp, k_prefix, v_prefix, w, n_heads: int, *, kv_valid=None, dtype=None, rms_eps=1e-5):
    """The block over a sequence's response rows only, with the prefix keys and
    values taken from a cache: queries are the response rows; keys/values are
    the cached prefix rows followed by the response rows' own (the first
    ``kv_valid`` response rows when given: bucket padding is never a key)."""
    R = rounding_for(dtype)
    x = _f64(x_resp)
    nv = x.shape[0] if kv_valid is None else int(kv_valid)
    xn = R(rmsnorm(x, w["g_attn"], rms_eps))
    q = R(xn @ _f64(w["wq"]).T)
    k = np.concatenate([_f64(k_prefix), R(xn[:nv] @ _f64(w["wk"]).T)])
    v = np.concatenate([_f64(v_prefix), R(xn[:nv] @ _f64(w["wv"]).T)])
    o = R(attention(q, k, v, n_heads))
    h = R(x + o @ _f64(w["wo"]).T)
    hn = R(rmsnorm(h, w["g_mlp"], rms_eps))
    return R(h + R(swiglu_activation(hn, w["wg"], w["wu"])) @ _f64(w["wd"]).T)
