"""Device-side input checks, through the C ABI: inconsistent device data is
recorded in the library's device error word (read and cleared by
seer_check_device) and clamped so that no kernel reads or writes outside the
buffers it was given.

Every output buffer here is allocated larger than the capacity passed to the
library and the margin is filled with a sentinel: the checks must leave it
untouched.  The inputs are ones the kernels' own checks turn into an error
code; none faults the GPU.
"""
import numpy as np
import pytest
import torch

import oracle
from tests.helpers import cuda, host, i32

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")

ERR_ROWS, ERR_LAYOUT, ERR_BOUNDARY, ERR_CAPACITY = 1, 2, 4, 5
SENTINEL = 13.0


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    assert S.seer_check_device() == 0
    yield
    assert S.seer_check_device() == 0


def _pack_inputs(B=3, N=64, d=256, seed=0):
    rng = np.random.default_rng(seed)
    ctx = rng.integers(20, 90, B)
    full = ctx + N
    cu_full = np.concatenate([[0], np.cumsum(full)]).astype(np.int32)
    x = torch.randn((int(cu_full[-1]), d), device=cuda(), dtype=torch.float32).to(torch.bfloat16)
    return ctx, cu_full, x


def test_boundary_out_of_range_is_recorded_and_clamped():
    B, N, d = 3, 64, 256
    ctx, cu_full, x = _pack_inputs(B, N, d)
    L = np.array([N + 5, 0, 17], dtype=np.int32)          # above N, below 1, valid
    T_cap = int(cu_full[-1])
    xp = torch.full((T_cap + 64, d), SENTINEL, dtype=torch.bfloat16, device=cuda())
    cu = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    kv = torch.empty(B, dtype=torch.int32, device=cuda())
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=cuda())
    params = S.make_params(0.0, tau_pad=-1.0)              # every segment keeps exactly ctx + L*
    S.seer_pack_ragged(x, "bf16", i32(cu_full), i32(ctx), i32(L), B, d, N, T_cap, params, xp, cu, kv, meta)
    torch.cuda.synchronize()
    assert S.seer_check_device() == ERR_BOUNDARY
    L_clamped = np.clip(L, 1, N)
    seg, kv_ref, cu_ref = oracle.segment_layout(ctx, L_clamped, N, -1.0)
    np.testing.assert_array_equal(cu.cpu().numpy(), cu_ref)
    np.testing.assert_array_equal(kv.cpu().numpy(), kv_ref)
    T = int(cu_ref[-1])
    np.testing.assert_array_equal(host(xp)[:T], oracle.pack_rows(host(x), cu_full, seg))
    assert (host(xp)[T:] == SENTINEL).all()


def test_packed_rows_beyond_capacity_are_recorded_and_not_written():
    B, N, d = 3, 64, 256
    ctx, cu_full, x = _pack_inputs(B, N, d, seed=1)
    L = np.array([40, 50, 60], dtype=np.int32)
    total = int((ctx + L).sum())
    T_cap = total - 37                                     # too small for the packed rows
    xp = torch.full((T_cap + 128, d), SENTINEL, dtype=torch.bfloat16, device=cuda())
    cu = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    kv = torch.empty(B, dtype=torch.int32, device=cuda())
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=cuda())
    params = S.make_params(0.0, tau_pad=-1.0)
    S.seer_pack_ragged(x, "bf16", i32(cu_full), i32(ctx), i32(L), B, d, N, T_cap, params, xp, cu, kv, meta)
    torch.cuda.synchronize()
    assert S.seer_check_device() == ERR_CAPACITY
    seg, _, _ = oracle.segment_layout(ctx, L, N, -1.0)
    np.testing.assert_array_equal(host(xp)[:T_cap], oracle.pack_rows(host(x), cu_full, seg)[:T_cap])
    assert (host(xp)[T_cap:] == SENTINEL).all()


def test_device_row_count_above_capacity_is_recorded_and_clamped():
    M_cap, N, K = 200, 256, 256
    a = torch.randn((M_cap, K), device=cuda()).half()
    w = (0.02 * torch.randn((N, K), device=cuda())).half()
    c = torch.full((M_cap + 64, N), SENTINEL, dtype=torch.float16, device=cuda())
    M_dev = torch.tensor([M_cap + 100], dtype=torch.int32, device=cuda())
    S.seer_linear(a, w, "f16", None, "f16", c, "f16", M_cap, M_dev, N, K)
    torch.cuda.synchronize()
    assert S.seer_check_device() == ERR_ROWS
    ref = a.double() @ w.double().T
    got = c[:M_cap].double()
    assert ((got - ref).abs() <= 1e-2 + 1e-2 * ref.abs()).all()
    assert (host(c)[M_cap:] == SENTINEL).all()


def test_attention_segment_past_capacity_is_recorded_and_skipped():
    H, dh = 2, 128
    D = H * dh
    T_cap = 300
    qkv = torch.randn((T_cap, 3 * D), device=cuda()).half()
    o = torch.full((T_cap + 32, D), SENTINEL, dtype=torch.float16, device=cuda())
    cu = np.array([0, 120, T_cap + 40], dtype=np.int32)    # the second segment runs past T_cap
    ws_bytes = S.seer_layer_workspace_size(S.make_dims(D, H, dh, 256), "f16", T_cap, 2)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_attention(qkv, o, "f16", i32(cu), None, 2, T_cap, H, dh, ws, ws_bytes)
    torch.cuda.synchronize()
    assert S.seer_check_device() == ERR_LAYOUT
    q = host(qkv)[:120].astype(np.float64)
    ref = oracle.attention(q[:, :D], q[:, D:2 * D], q[:, 2 * D:], H)
    got = host(o)[:120].astype(np.float64)
    assert (np.abs(got - ref) <= 1e-2 + 1e-2 * np.abs(ref)).all()     # the valid segment still runs
    assert (host(o)[120:] == SENTINEL).all()                            # the bad one is skipped


# ---------------------------------------------------------------- f16 range guard
ERR_RANGE = 6


def test_swiglu_intermediate_beyond_f16_range_is_recorded():
    # a = SiLU(x Wg^T) * (x Wu^T) with x = 4 and weights 0.5 over K = 256: g = u = 512
    # and a ~ 2.6e5, beyond f16's largest finite value 65504; the stored f16 `a` is
    # infinite and the epilogue's range guard records the code.  The same call with
    # x = 0.25 (a ~ 1024) stays finite and records nothing.
    M, F, K = 256, 256, 256
    wg = torch.full((F, K), 0.5, dtype=torch.float16, device=cuda())
    wu = torch.full((F, K), 0.5, dtype=torch.float16, device=cuda())
    act = torch.empty((M, F), dtype=torch.float16, device=cuda())
    small = torch.full((M, K), 0.25, dtype=torch.float16, device=cuda())
    S.seer_swiglu(small, wg, wu, "f16", act, "f16", M, None, F, K)
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
    assert torch.isfinite(act.float()).all()
    big = torch.full((M, K), 4.0, dtype=torch.float16, device=cuda())
    S.seer_swiglu(big, wg, wu, "f16", act, "f16", M, None, F, K)
    torch.cuda.synchronize()
    assert S.seer_check_device() == ERR_RANGE
    assert torch.isinf(act.float()).all()


def test_layer_residual_beyond_f16_range_is_recorded():
    # a bf16 layer whose input rows hold 1e5 (finite in bf16): the f16 residual
    # stream h = x + o Wo^T overflows, and the O-projection epilogue records the
    # code; the same layer on N(0, 1) rows records nothing
    from tests.helpers import layer_weight_tensors, to_dev, weights_struct
    import synth
    wl = synth.tiny_workload(dtype="bf16", seed=410, d=256, n_heads=2, head_dim=128, d_ff=768, batch=2, window=64)
    w = synth.layer_weights(wl, 0)
    _, WL = layer_weight_tensors(wl, w)
    dims = S.make_dims(wl.d, wl.n_heads, wl.head_dim, wl.d_ff)
    T = 300
    cu = i32([0, 140, T])
    ws_bytes = S.seer_layer_workspace_size(dims, "bf16", T, 2)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    y = torch.empty((T, wl.d), dtype=torch.bfloat16, device=cuda())
    x = to_dev(np.random.default_rng(0).standard_normal((T, wl.d)), "bf16")
    S.seer_layer_forward(weights_struct(WL), dims, "bf16", x, y, cu, None, 2, T, None, 0, 0.0, None, ws, ws_bytes)
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
    x_big = torch.full((T, wl.d), 1e5, dtype=torch.bfloat16, device=cuda())
    S.seer_layer_forward(weights_struct(WL), dims, "bf16", x_big, y, cu, None, 2, T, None, 0, 0.0, None, ws, ws_bytes)
    torch.cuda.synchronize()
    assert S.seer_check_device() == ERR_RANGE


def test_convert_beyond_f16_range_is_recorded():
    # bf16 -> f16 of 1e5 (finite in bf16, beyond f16) gives infinity and the code
    src = torch.full((64,), 1e5, dtype=torch.bfloat16, device=cuda())
    dst = torch.empty((64,), dtype=torch.float16, device=cuda())
    S.seer_convert(src, "bf16", dst, "f16", 64)
    torch.cuda.synchronize()
    assert S.seer_check_device() == ERR_RANGE
    S.seer_convert(src / 4, "bf16", dst, "f16", 64)      # 25000: finite in f16
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
