"""Seeded fuzzing of the whole path (detect -> route/pack -> truncated layer)
through the C ABI against the oracle: batch sizes, windows, prefix lengths,
boundaries near both ends of the window, tau_pad and the smallest bucket drawn
at random per case; a second family at 4-6 heads and F up to 2048, with the
rotary embedding on or off."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import check_close, cuda, host, i32, layer_weight_tensors, to_dev, weights_struct

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    assert S.seer_check_device() == 0


def _case(seed):
    r = np.random.default_rng(1000 + seed)
    B = int(r.integers(1, 7))
    N = int(r.integers(16, 300))
    wl = synth.tiny_workload(dtype="bf16", seed=500 + seed, d=256, n_heads=2, head_dim=128, d_ff=768, batch=B,
                             window=N, visual=("mult", int(r.integers(1, 200)), 0, 2),
                             prompt=("uniform", 1, int(r.integers(2, 60))), boundary=("uniform", 1, N - 5))
    return wl, float(r.choice([-1.0, 0.1, 0.2, 0.5, 0.9])), int(r.choice([1, 8, 16, 64]))


@pytest.mark.parametrize("seed", range(12))
def test_fuzz_full_path(seed):
    wl, tau_pad, bucket_min = _case(seed)
    lens = synth.lengths(wl)
    x, cu_full, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    B, N, F, d = wl.batch, wl.window, wl.d_ff, wl.d
    dims = S.make_dims(d, wl.n_heads, wl.head_dim, F)
    params = S.make_params(wl.act_eps, tau_pad=tau_pad, bucket_min=bucket_min)
    W, WL = layer_weight_tensors(wl, w)
    xd = to_dev(x, "bf16")
    counts = torch.empty(B * N, dtype=torch.int32, device=cuda())
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_detect_boundary(xd, "bf16", x.shape[0], i32(resp), B, N, W["w_gate"], W["w_up"], dims, params, counts, L)
    T_cap = int(cu_full[-1]) + 17
    xp = torch.zeros((T_cap, d), dtype=torch.bfloat16, device=cuda())
    cu = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    kv = torch.empty(B, dtype=torch.int32, device=cuda())
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=cuda())
    S.seer_pack_ragged(xd, "bf16", i32(cu_full), i32(lens.ctx), L, B, d, N, T_cap, params, xp, cu, kv, meta)
    y = torch.full((T_cap, d), 9.0, dtype=torch.bfloat16, device=cuda())
    ws_bytes = S.seer_layer_workspace_size(dims, "bf16", T_cap, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_layer_forward(weights_struct(WL), dims, "bf16", xp, y, cu, kv, B, T_cap, None, 0, 0.0, None, ws, ws_bytes)
    torch.cuda.synchronize()
    # detection: the planted boundary, and the counts within 0.5% of F
    L_h = L.cpu().numpy()
    np.testing.assert_array_equal(L_h, lens.boundary + 1)
    got = counts.cpu().numpy().reshape(B, N)
    for b in range(B):
        ref = oracle.sparsity_counts(x[resp[b]:resp[b] + N], w["wg"], w["wu"], wl.act_eps)
        assert np.abs(got[b] - ref).max() <= 0.005 * F
    # routing and compaction: bit exact
    seg, kv_ref, cu_ref = oracle.segment_layout(lens.ctx, L_h, N, tau_pad, bucket_min=bucket_min)
    np.testing.assert_array_equal(cu.cpu().numpy(), cu_ref)
    np.testing.assert_array_equal(kv.cpu().numpy(), kv_ref)
    T = int(cu_ref[-1])
    np.testing.assert_array_equal(host(xp)[:T], oracle.pack_rows(x, cu_full, seg))
    # the layer against the exact definition; nothing written past the packed rows
    ref = oracle.layer_forward_packed(host(xp)[:T], cu_ref, w, wl.n_heads, kv_len=kv_ref)
    check_close(host(y)[:T], ref, "bf16", f"fuzz case {seed}")
    assert (host(y)[T:] == 9.0).all()


def _wide_case(seed):
    r = np.random.default_rng(2000 + seed)
    d = int(r.choice([512, 768]))
    B = int(r.integers(1, 5))
    N = int(r.integers(32, 260))
    F = int(r.choice([1536, 2048]))
    wl = synth.tiny_workload(dtype="bf16", seed=700 + seed, d=d, n_heads=d // 128, head_dim=128, d_ff=F, batch=B,
                             window=N, visual=("mult", int(r.integers(1, 150)), 0, 2), prompt=("uniform", 1, 40),
                             boundary=("uniform", 1, N - 5))
    return wl, float(r.choice([-1.0, 0.2, 0.9])), float(r.choice([0.0, 1e4]))


@pytest.mark.parametrize("seed", range(10))
def test_fuzz_full_path_wide(seed):
    # 4 or 6 heads, F 1536 or 2048 (several GEMM n-tiles, ragged m-tiles), rotary on or off
    wl, tau_pad, theta = _wide_case(seed)
    lens = synth.lengths(wl)
    x, cu_full, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    B, N, F, d = wl.batch, wl.window, wl.d_ff, wl.d
    dims = S.make_dims(d, wl.n_heads, wl.head_dim, F, rope_theta=theta)
    params = S.make_params(wl.act_eps, tau_pad=tau_pad)
    W, WL = layer_weight_tensors(wl, w)
    xd = to_dev(x, "bf16")
    counts = torch.empty(B * N, dtype=torch.int32, device=cuda())
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_detect_boundary(xd, "bf16", x.shape[0], i32(resp), B, N, W["w_gate"], W["w_up"], dims, params, counts, L)
    T_cap = int(cu_full[-1]) + 5
    xp = torch.zeros((T_cap, d), dtype=torch.bfloat16, device=cuda())
    cu = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    kv = torch.empty(B, dtype=torch.int32, device=cuda())
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=cuda())
    S.seer_pack_ragged(xd, "bf16", i32(cu_full), i32(lens.ctx), L, B, d, N, T_cap, params, xp, cu, kv, meta)
    y = torch.full((T_cap, d), 9.0, dtype=torch.bfloat16, device=cuda())
    ws_bytes = S.seer_layer_workspace_size(dims, "bf16", T_cap, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_layer_forward(weights_struct(WL), dims, "bf16", xp, y, cu, kv, B, T_cap, None, 0, 0.0, None, ws, ws_bytes)
    torch.cuda.synchronize()
    L_h = L.cpu().numpy()
    np.testing.assert_array_equal(L_h, lens.boundary + 1)
    got = counts.cpu().numpy().reshape(B, N)
    for b in range(B):
        ref = oracle.sparsity_counts(x[resp[b]:resp[b] + N], w["wg"], w["wu"], wl.act_eps)
        assert np.abs(got[b] - ref).max() <= 0.005 * F
    seg, kv_ref, cu_ref = oracle.segment_layout(lens.ctx, L_h, N, tau_pad)
    np.testing.assert_array_equal(cu.cpu().numpy(), cu_ref)
    np.testing.assert_array_equal(kv.cpu().numpy(), kv_ref)
    T = int(cu_ref[-1])
    np.testing.assert_array_equal(host(xp)[:T], oracle.pack_rows(x, cu_full, seg))
    ref = oracle.layer_forward_packed(host(xp)[:T], cu_ref, w, wl.n_heads, kv_len=kv_ref, rope_theta=theta)
    check_close(host(y)[:T], ref, "bf16", f"wide fuzz case {seed}")
    assert (host(y)[T:] == 9.0).all()
