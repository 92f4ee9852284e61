"""Thin ctypes binding of libseer (include/seer.h).

Argument marshalling only: every function has the name of its C entry point,
takes torch tensors (or raw integer device pointers), passes their addresses
and the current CUDA stream, and raises :class:`SeerError` on a non-zero
status.  All arithmetic happens in the library's CUDA kernels; there is no
host fallback, and importing this module fails loudly when libseer.so has not
been built.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch  # noqa: F401  (loads the CUDA runtime the library shares)

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libseer.so")

SEER_F32, SEER_BF16, SEER_F16 = 0, 1, 2
PATH_STATIC, PATH_VARLEN, PATH_EAGER = 0, 1, 2
MAX_GROUPS = 32
CTRL_WORDS = 8 + 4 * MAX_GROUPS
N_PHASES = 11
PHASES = ("detect_gemm", "snr_scan", "pack", "norm1", "qkv", "attention", "o_proj", "norm2", "gate_up", "down",
          "kv_cache")

_STATUS = {0: "SEER_OK", 1: "SEER_ERR_INVALID_ARG", 2: "SEER_ERR_UNSUPPORTED", 3: "SEER_ERR_WORKSPACE",
           4: "SEER_ERR_CUDA", 5: "SEER_ERR_TIMEOUT", 6: "SEER_ERR_DEVICE"}


class SeerError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


class seer_dims(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int), ("n_heads", ctypes.c_int), ("head_dim", ctypes.c_int),
                ("d_ff", ctypes.c_int), ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float)]


class seer_params(ctypes.Structure):
    _fields_ = [("act_eps", ctypes.c_float), ("tau_jump", ctypes.c_double), ("gamma", ctypes.c_double),
                ("window", ctypes.c_int), ("tau_pad", ctypes.c_double), ("eager_max_bucket", ctypes.c_int),
                ("bucket_min", ctypes.c_int)]


class seer_layer_weights(ctypes.Structure):
    _fields_ = [("w_qkv", ctypes.c_void_p), ("w_o", ctypes.c_void_p), ("w_gate", ctypes.c_void_p),
                ("w_up", ctypes.c_void_p), ("w_down", ctypes.c_void_p), ("g_attn", ctypes.c_void_p),
                ("g_mlp", ctypes.c_void_p)]


_lib = None


def lib() -> ctypes.CDLL:
    """Load libseer.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libseer.so not found at {LIB_PATH}; build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        sigs = {
            "seer_detect_boundary": [vp, i32, i32, vp, i32, i32, vp, vp, ctypes.POINTER(seer_dims),
                                     ctypes.POINTER(seer_params), vp, vp, vp, vp],
            "seer_pack_ragged": [vp, i32, vp, vp, vp, i32, i32, i32, i32, ctypes.POINTER(seer_params), vp, vp, vp,
                                 vp, vp, ctypes.c_int32, vp],
            "seer_poll_ctrl": [vp, ctypes.c_int32, i32, vp],
            "seer_sparsity_counts": [vp, i32, i32, vp, i32, i32, vp, vp, ctypes.POINTER(seer_dims), ctypes.c_float,
                                     i32, vp, vp],
            "seer_kv_prefill": [ctypes.POINTER(seer_layer_weights), ctypes.POINTER(seer_dims), i32, vp, vp, vp, i32, i32,
                                vp, vp, i32, vp, sz, vp],
            "seer_layer_forward_cached": [ctypes.POINTER(seer_layer_weights), ctypes.POINTER(seer_dims), i32, vp, vp,
                                          vp, vp, i32, i32, vp, vp, vp, i32, vp, sz, vp],
            "seer_gather_response": [vp, i32, vp, vp, i32, i32, i32, vp, vp, vp],
            "seer_snr_scan": [vp, i32, i32, i32, ctypes.POINTER(seer_params), vp, vp, vp],
            "seer_layer_forward": [ctypes.POINTER(seer_layer_weights), ctypes.POINTER(seer_dims), i32, vp, vp, vp, vp,
                                   i32, i32, vp, i32, ctypes.c_float, vp, vp, sz, vp],
            "seer_layer_workspace_size": [ctypes.POINTER(seer_dims), i32, i32, i32, ctypes.POINTER(sz)],
            "seer_rmsnorm": [vp, i32, vp, vp, i32, i32, vp, i32, ctypes.c_float, vp],
            "seer_linear": [vp, vp, i32, vp, i32, vp, i32, i32, vp, i32, i32, vp],
            "seer_rope": [vp, i32, vp, i32, i32, i32, i32, ctypes.c_float, vp],
            "seer_swiglu": [vp, vp, vp, i32, vp, i32, i32, vp, i32, i32, vp, i32, vp, i32, ctypes.c_float, vp, vp],
            "seer_convert": [vp, i32, vp, i32, sz, vp],
            "seer_attention": [vp, vp, i32, vp, vp, i32, i32, i32, i32, vp, sz, vp],
            "seer_attention_noalloc": [vp, vp, i32, vp, vp, i32, i32, i32, i32, vp],
            "seer_check_device": [ctypes.POINTER(ctypes.c_int)],
            "seer_selftest_wait_timeout": [i32, vp],
            "seer_profile_enable": [i32],
            "seer_profile_reset": [],
            "seer_profile_select": [ctypes.c_uint32],
            "seer_profile_read": [vp, vp],
        }
        for name, args in sigs.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        L.seer_last_error.restype = ctypes.c_char_p
        L.seer_last_error.argtypes = []
        L.seer_version.restype = ctypes.c_char_p
        L.seer_num_sms.restype = ctypes.c_int
        L.seer_set_launch_overlap.restype = ctypes.c_int
        L.seer_set_launch_overlap.argtypes = [ctypes.c_int]
        _lib = L
    return _lib


def _check(status: int):
    if status != 0:
        raise SeerError(status, lib().seer_last_error().decode())


def _p(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _dt(dt) -> int:
    if dt in (SEER_F32, SEER_BF16, SEER_F16):
        return dt
    if dt in ("bf16", torch.bfloat16):
        return SEER_BF16
    if dt in ("f16", torch.float16):
        return SEER_F16
    if dt in ("f32", torch.float32):
        return SEER_F32
    raise ValueError(f"unsupported dtype {dt!r}")


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_dims(d_model, n_heads, head_dim, d_ff, rms_eps=1e-5, rope_theta=0.0) -> seer_dims:
    return seer_dims(d_model, n_heads, head_dim, d_ff, rms_eps, rope_theta)


def make_params(act_eps, tau_jump=0.03, gamma=0.6, window=3, tau_pad=0.2, eager_max_bucket=4,
                bucket_min=8) -> seer_params:
    return seer_params(act_eps, tau_jump, gamma, window, tau_pad, eager_max_bucket, bucket_min)


def make_weights(w_qkv, w_o, w_gate, w_up, w_down, g_attn, g_mlp) -> seer_layer_weights:
    return seer_layer_weights(*[_p(t) for t in (w_qkv, w_o, w_gate, w_up, w_down, g_attn, g_mlp)])


# ----------------------------------------------------------------- entry points
def seer_detect_boundary(x, dt, T_rows, resp_start, B, N, w_gate, w_up, dims, params, counts_out, L_star_out,
                         i_star_out=None, stream=None):
    _check(lib().seer_detect_boundary(_p(x), _dt(dt), T_rows, _p(resp_start), B, N, _p(w_gate), _p(w_up),
                                      ctypes.byref(dims), ctypes.byref(params), _p(counts_out), _p(L_star_out),
                                      _p(i_star_out), _stream(stream)))


def seer_pack_ragged(x_full, dt, cu_full, ctx_len, L_star, B, d, N, T_capacity, params, x_packed, cu_out, kv_len_out,
                     meta_out, host_ctrl=None, epoch=1, stream=None):
    _check(lib().seer_pack_ragged(_p(x_full), _dt(dt), _p(cu_full), _p(ctx_len), _p(L_star), B, d, N, T_capacity,
                                  ctypes.byref(params), _p(x_packed), _p(cu_out), _p(kv_len_out), _p(meta_out),
                                  _p(host_ctrl), epoch, _stream(stream)))


def seer_sparsity_counts(x, dt, T_rows, resp_start, B, N, w_gate, w_up, dims, act_eps, counts_inout, accumulate=False,
                         stream=None):
    _check(lib().seer_sparsity_counts(_p(x), _dt(dt), T_rows, _p(resp_start), B, N, _p(w_gate), _p(w_up),
                                      ctypes.byref(dims), act_eps, 1 if accumulate else 0, _p(counts_inout),
                                      _stream(stream)))


def seer_kv_prefill(w, dims, dt, x, cu_x, ctx_len, B, T_x_cap, kv_cache, cu_kv, T_kv_cap, ws, ws_bytes, stream=None):
    _check(lib().seer_kv_prefill(ctypes.byref(w), ctypes.byref(dims), _dt(dt), _p(x), _p(cu_x), _p(ctx_len), B, T_x_cap,
                                 _p(kv_cache), _p(cu_kv), T_kv_cap, _p(ws), ws_bytes, _stream(stream)))


def seer_layer_forward_cached(w, dims, dt, x_resp, y_resp, cu_resp, ctx_len, B, T_resp_cap, kv_cache, cu_kv, kv_len,
                              T_kv_cap, ws, ws_bytes, stream=None):
    _check(lib().seer_layer_forward_cached(ctypes.byref(w), ctypes.byref(dims), _dt(dt), _p(x_resp), _p(y_resp),
                                           _p(cu_resp), _p(ctx_len), B, T_resp_cap, _p(kv_cache), _p(cu_kv),
                                           _p(kv_len), T_kv_cap, _p(ws), ws_bytes, _stream(stream)))


def seer_gather_response(x_packed, dt, cu, ctx_len, B, d, T_cap, x_resp, cu_resp_out, stream=None):
    _check(lib().seer_gather_response(_p(x_packed), _dt(dt), _p(cu), _p(ctx_len), B, d, T_cap, _p(x_resp),
                                      _p(cu_resp_out), _stream(stream)))


def seer_snr_scan(counts, B, N, F, params, L_star_out, i_star_out=None, stream=None):
    _check(lib().seer_snr_scan(_p(counts), B, N, F, ctypes.byref(params), _p(L_star_out), _p(i_star_out),
                               _stream(stream)))


def seer_poll_ctrl(host_ctrl, epoch, timeout_us, ctrl_copy=None):
    _check(lib().seer_poll_ctrl(_p(host_ctrl), epoch, timeout_us, _p(ctrl_copy)))


def seer_layer_forward(w, dims, dt, x, y, cu_seqlens, kv_len, B, T_capacity, count_resp_start, N, act_eps, counts_out,
                       ws, ws_bytes, stream=None):
    _check(lib().seer_layer_forward(ctypes.byref(w), ctypes.byref(dims), _dt(dt), _p(x), _p(y), _p(cu_seqlens),
                                    _p(kv_len), B, T_capacity, _p(count_resp_start), N, act_eps, _p(counts_out),
                                    _p(ws), ws_bytes, _stream(stream)))


def seer_layer_workspace_size(dims, dt, T_capacity, B) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().seer_layer_workspace_size(ctypes.byref(dims), _dt(dt), T_capacity, B, ctypes.byref(out)))
    return out.value


def seer_rmsnorm(x, x_dt, g, y, y_dt, M_cap, M_dev, d, eps, stream=None):
    _check(lib().seer_rmsnorm(_p(x), _dt(x_dt), _p(g), _p(y), _dt(y_dt), M_cap, _p(M_dev), d, eps, _stream(stream)))


def seer_linear(a, w, op_dt, r, r_dt, c, c_dt, M_cap, M_dev, N, K, stream=None):
    _check(lib().seer_linear(_p(a), _p(w), _dt(op_dt), _p(r), _dt(r_dt), _p(c), _dt(c_dt), M_cap, _p(M_dev), N, K,
                             _stream(stream)))


def seer_rope(qkv, dt, cu_seqlens, B, T_capacity, n_heads, head_dim, theta, stream=None):
    _check(lib().seer_rope(_p(qkv), _dt(dt), _p(cu_seqlens), B, T_capacity, n_heads, head_dim, theta, _stream(stream)))


def seer_swiglu(a, w_gate, w_up, op_dt, act, act_dt, M_cap, M_dev, F, K, cu_seqlens=None, B=0, count_resp_start=None,
                N=0, act_eps=0.0, counts_out=None, stream=None):
    _check(lib().seer_swiglu(_p(a), _p(w_gate), _p(w_up), _dt(op_dt), _p(act), _dt(act_dt), M_cap, _p(M_dev), F, K,
                             _p(cu_seqlens), B, _p(count_resp_start), N, act_eps, _p(counts_out), _stream(stream)))


def seer_convert(src, src_dt, dst, dst_dt, n, stream=None):
    _check(lib().seer_convert(_p(src), _dt(src_dt), _p(dst), _dt(dst_dt), n, _stream(stream)))


def seer_attention(qkv, o, dt, cu_seqlens, kv_len, B, T_capacity, n_heads, head_dim, ws=None, ws_bytes=0,
                   stream=None):
    _check(lib().seer_attention(_p(qkv), _p(o), _dt(dt), _p(cu_seqlens), _p(kv_len), B, T_capacity, n_heads,
                                head_dim, _p(ws), ws_bytes, _stream(stream)))


def seer_attention_noalloc(qkv, o, dt, cu_seqlens, kv_len, B, T_capacity, n_heads, head_dim, stream=None):
    _check(lib().seer_attention_noalloc(_p(qkv), _p(o), _dt(dt), _p(cu_seqlens), _p(kv_len), B, T_capacity, n_heads,
                                        head_dim, _stream(stream)))


def seer_check_device() -> int:
    code = ctypes.c_int(0)
    st = lib().seer_check_device(ctypes.byref(code))
    if st not in (0, 6):
        _check(st)
    return code.value


def seer_profile_enable(on: bool = True):
    _check(lib().seer_profile_enable(1 if on else 0))


def seer_profile_select(phases=None):
    """Record only the named phases (names from PHASES; None = all)."""
    mask = 0xFFFFFFFF if phases is None else sum(1 << PHASES.index(n) for n in phases)
    _check(lib().seer_profile_select(mask))


def seer_profile_reset():
    _check(lib().seer_profile_reset())


def seer_profile_read():
    ms = (ctypes.c_float * N_PHASES)()
    n = (ctypes.c_int32 * N_PHASES)()
    _check(lib().seer_profile_read(ctypes.addressof(ms), ctypes.addressof(n)))
    return {PHASES[i]: (float(ms[i]), int(n[i])) for i in range(N_PHASES)}


def seer_set_launch_overlap(on: bool) -> bool:
    """Turns programmatic dependent launch of the library's kernels on or off
    (process-wide); returns the previous setting."""
    return bool(lib().seer_set_launch_overlap(1 if on else 0))


def seer_num_sms() -> int:
    return int(lib().seer_num_sms())


def seer_version() -> str:
    return lib().seer_version().decode()


def seer_selftest_wait_timeout(limit_us: int, stream=None):
    _check(lib().seer_selftest_wait_timeout(limit_us, _stream(stream)))
