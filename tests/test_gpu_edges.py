"""Degenerate and boundary cases of the hot path, through the C ABI, against the
oracle: tile and tile-pair boundaries of the attention schedule, empty
segments, empty calls, extreme boundaries (L* = 1 everywhere, a scan window of
one candidate, all-zero counts) and an empty prefix on the K/V-cache path."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import check_close, cuda, host, i32, to_dev
from tests.test_gpu_ops import _attention_case, _pack_case

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    assert S.seer_check_device() == 0


@pytest.mark.parametrize("dt", ["f16", "bf16"])
def test_attention_query_tile_pair_boundaries(dt):
    # a CTA takes two 128-query tiles: lengths around 256 and 384 leave the
    # second tile full, partial or absent
    lens = [255, 256, 257, 383, 384, 385, 2]
    _attention_case(dt, 2, 128, lens, lens, 1.0, 21)


@pytest.mark.parametrize("dt", ["f16", "bf16"])
def test_attention_probability_half_boundaries(dt):
    # a round's PV is issued in two halves of 64 keys as the softmax releases
    # them: last key tiles with 63, 64 and 65 valid keys (the second half empty,
    # exactly full, or holding one key), and a kv_len short of the segment
    lens = [64, 63, 65, 192, 191, 193, 300]
    kv = [64, 63, 65, 192, 191, 193, 129]
    _attention_case(dt, 2, 128, lens, kv, 1.0, 27)


def test_attention_single_key_and_single_query_segments():
    lens = [1, 1, 129, 1]
    _attention_case("f16", 2, 128, lens, [1, 1, 1, 1], 1.0, 22)


def test_attention_empty_segments_are_skipped():
    rng = np.random.default_rng(23)
    H, dh = 2, 128
    D = H * dh
    lens = [0, 70, 0, 256]
    cu = np.concatenate([[0], np.cumsum(lens)])
    T = int(cu[-1])
    qkv = synth.round_storage(rng.standard_normal((T, 3 * D)), "bf16")
    out = torch.full((T, D), 3.0, dtype=torch.bfloat16, device=cuda())
    ws_bytes = H * ((T + 127) // 128 + len(lens)) * 16 + 4096
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_attention(to_dev(qkv, "bf16"), out, "bf16", i32(cu), i32(lens), len(lens), T, H, dh, ws, ws_bytes)
    got = host(out)
    for b in range(len(lens)):
        s0, s1 = cu[b], cu[b + 1]
        if s1 > s0:
            ref = oracle.attention(qkv[s0:s1, :D], qkv[s0:s1, D:2 * D], qkv[s0:s1, 2 * D:], H)
            check_close(got[s0:s1], ref, "bf16", f"segment {b}")


def test_empty_calls_launch_nothing_and_succeed():
    x = torch.full((4, 256), 5.0, dtype=torch.float16, device=cuda())
    w = torch.zeros((256, 256), dtype=torch.float16, device=cuda())
    S.seer_linear(x, w, "f16", None, "f16", x, "f16", 0, None, 256, 256)
    ws = torch.empty(1 << 16, dtype=torch.uint8, device=cuda())
    S.seer_attention(x, x, "f16", i32([0, 0]), None, 1, 0, 2, 128, ws, 1 << 16)
    torch.cuda.synchronize()
    assert (host(x) == 5.0).all()


def test_pack_every_boundary_at_one_token():
    # L* = 1 everywhere: every sequence falls in the smallest bucket
    ctx = [33, 70, 12, 128, 5]
    _pack_case("bf16", ctx, [1] * len(ctx), 512, 256, seed=24)


def test_pack_mixed_extremes():
    ctx = [64, 1, 200, 7]
    _pack_case("bf16", ctx, [1, 512, 512, 2], 512, 256, seed=25)


def test_snr_scan_degenerate_windows():
    # N = w + 1 leaves a single candidate i = 1; all-zero counts never hit
    p = S.make_params(0.0, 0.03, 0.6, 3)
    counts = np.array([[0, 50, 50, 50], [0, 0, 0, 0], [10, 10, 10, 10]])
    B, N = counts.shape
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    I = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_snr_scan(i32(counts.ravel()), B, N, 100, p, L, I)
    i_ref, L_ref = oracle.snr_boundaries(counts, 100)
    np.testing.assert_array_equal(I.cpu().numpy(), i_ref)
    np.testing.assert_array_equal(L.cpu().numpy(), L_ref)
    assert list(L_ref) == [2, 4, 4]


def test_cached_layer_with_an_empty_prefix():
    # ctx = 0 for one sequence: its keys are its response rows alone
    from paper_2607_14557_gb300 import driver as D
    wl = synth.tiny_workload(dtype="bf16", seed=380, d=256, n_heads=2, head_dim=128, d_ff=768, batch=2, window=128)
    w = synth.layer_weights(wl, 0)
    d, H, B = wl.d, wl.n_heads, 2
    rng = np.random.default_rng(26)
    ctx = np.array([0, 150])
    resp = np.array([40, 60])
    seg = ctx + resp
    cu = np.concatenate([[0], np.cumsum(seg)]).astype(np.int32)
    T = int(cu[-1])
    x = synth.round_storage(rng.standard_normal((T, d)), "bf16")
    dims = S.make_dims(d, H, wl.head_dim, wl.d_ff)
    W = D.LayerWeights.from_host(w, "bf16")
    ws_bytes = S.seer_layer_workspace_size(dims, "bf16", T, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    cache = torch.zeros((T, 2 * d), dtype=torch.float16, device=cuda())
    xd = to_dev(x, "bf16")
    S.seer_kv_prefill(W.struct(), dims, "bf16", xd, i32(cu), i32(ctx), B, T, cache, i32(cu), T, ws, ws_bytes)
    xr = torch.zeros((T, d), dtype=torch.bfloat16, device=cuda())
    cu_r = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    S.seer_gather_response(xd, "bf16", i32(cu), i32(ctx), B, d, T, xr, cu_r)
    yr = torch.full_like(xr, 9.0)
    S.seer_layer_forward_cached(W.struct(), dims, "bf16", xr, yr, cu_r, i32(ctx), B, T, cache, i32(cu), None, T, ws,
                                ws_bytes)
    torch.cuda.synchronize()
    cr = cu_r.cpu().numpy()
    np.testing.assert_array_equal(cr, [0, 40, 100])
    yh = host(yr)
    for b in range(B):
        xs = x[cu[b]:cu[b + 1]]
        k, v = oracle.kv_prefill(xs[:ctx[b]], w, H)
        ref = oracle.layer_forward_cached(xs[ctx[b]:], k, v, w, H)
        check_close(yh[cr[b]:cr[b + 1]], ref, "bf16", f"cached segment {b}")
    assert (yh[cr[-1]:] == 9.0).all()
