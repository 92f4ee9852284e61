"""GPU parity of prefix key/value caching combined with truncation (Table 7's
composition): prefill of the prefix K/V, response-row gather, and the block
over response rows with cached prefix keys, through the C ABI, against the
oracle; and exactness against the uncached truncated layer on the same input."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import check_close, cuda, host, i32, to_dev

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    assert S.seer_check_device() == 0


def _workload(dtype):
    if dtype == "f32":
        return synth.workload(0)
    return synth.tiny_workload(dtype="bf16", seed=370, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4, window=200,
                               boundary=("uniform", 8, 190), visual=("mult", 96, 1, 3))


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_cached_layer_matches_oracle_and_uncached_rows(dtype):
    from paper_2607_14557_gb300 import driver as D
    wl = _workload(dtype)
    lens = synth.lengths(wl)
    x, cu_full, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    B, N, d, H = wl.batch, wl.window, wl.d, wl.n_heads
    dims = S.make_dims(d, H, wl.head_dim, wl.d_ff)
    W = D.LayerWeights.from_host(w, dtype)
    T_full = x.shape[0]
    path = D.SeerPath(dims, dtype, B, N, T_full, S.make_params(wl.act_eps))
    ctx = i32(lens.ctx)
    path.step(to_dev(x, dtype), i32(cu_full), i32(resp), ctx, W)         # detect, pack, uncached truncated layer
    it = torch.float32 if dtype == "f32" else torch.float16
    cache = torch.full((T_full, 2 * d), 7.0, dtype=it, device=cuda())
    S.seer_kv_prefill(W.struct(), dims, dtype, path.x_packed, path.cu, ctx, B, T_full, cache, path.cu, T_full, path.ws,
                      path.ws_bytes)
    xr = torch.zeros_like(path.x_packed)
    cu_r = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    S.seer_gather_response(path.x_packed, dtype, path.cu, ctx, B, d, T_full, xr, cu_r)
    yr = torch.full_like(xr, 9.0)
    S.seer_layer_forward_cached(W.struct(), dims, dtype, xr, yr, cu_r, ctx, B, T_full, cache, path.cu, path.kv, T_full,
                                path.ws, path.ws_bytes)
    torch.cuda.synchronize()
    cu, kv, c = path.cu.cpu().numpy(), path.kv.cpu().numpy(), lens.ctx
    np.testing.assert_array_equal(path.L_star.cpu().numpy(), lens.boundary + 1)
    np.testing.assert_array_equal(cu_r.cpu().numpy(), cu - np.concatenate([[0], np.cumsum(c)]))
    cr = cu_r.cpu().numpy()
    xp, xrh, yrh, yfull, ch = host(path.x_packed), host(xr), host(yr), host(path.y), host(cache)
    for b in range(B):
        seg = xp[cu[b]:cu[b + 1]]
        np.testing.assert_array_equal(xrh[cr[b]:cr[b + 1]], seg[c[b]:])                 # gather is exact
        # the cached block reproduces the uncached truncated layer's response rows bit for bit
        np.testing.assert_array_equal(yrh[cr[b]:cr[b + 1]], yfull[cu[b] + c[b]:cu[b + 1]])
        k, v = oracle.kv_prefill(seg[:c[b]], w, H)
        check_close(ch[cu[b]:cu[b] + c[b]], np.concatenate([k, v], axis=1), dtype, f"prefix K/V {b}")
        ref = oracle.layer_forward_cached(seg[c[b]:], k, v, w, H, kv_valid=int(kv[b] - c[b]))
        check_close(yrh[cr[b]:cr[b + 1]], ref, dtype, f"cached block segment {b}")
    assert (yrh[cr[-1]:] == 9.0).all()                                                 # zero work past the rows


def test_cache_entry_points_reject_bad_arguments():
    x = torch.zeros((8, 256), dtype=torch.bfloat16, device=cuda())
    cu = i32([0, 8])
    with pytest.raises(RuntimeError):
        S.seer_gather_response(x, "bf16", cu, None, 1, 256, 8, x, cu)
    dims = S.make_dims(256, 2, 128, 768, rope_theta=1e4)
    w = S.seer_layer_weights()
    with pytest.raises(RuntimeError):
        S.seer_layer_forward_cached(w, dims, "bf16", x, x, cu, cu, 1, 8, x, cu, None, 8, x, 0)
