"""Pins of the oracle's layer (Sec. 3.1 Eq. 2; Sec. 3.6 Eqs. 6-7, 9-11)."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as TF

import oracle
import synth


def t(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float64))


def test_round_bf16_matches_torch_converter():
    rng = np.random.default_rng(0)
    vals = np.concatenate([
        rng.standard_normal(20000).astype(np.float32),
        (rng.standard_normal(2000) * 1e-38).astype(np.float32),      # subnormal range
        (rng.standard_normal(2000) * 1e30).astype(np.float32),
    ])
    # exact halfway points between neighbouring bf16 values (ties to even)
    base = torch.from_numpy(rng.standard_normal(2000).astype(np.float32)).to(torch.bfloat16).float().numpy()
    bits = base.view(np.uint32) | np.uint32(0x8000)
    vals = np.concatenate([vals, bits.view(np.float32), np.float32([0.0, -0.0, 1.0, -3.5])])
    ref = torch.from_numpy(vals).to(torch.bfloat16).to(torch.float64).numpy()
    got = oracle.round_bf16(vals.astype(np.float64))
    np.testing.assert_array_equal(got, ref)


def test_rmsnorm_matches_torch():
    rng = np.random.default_rng(1)
    x, g = rng.standard_normal((9, 33)), rng.standard_normal(33)
    ref = TF.rms_norm(t(x), (33,), weight=t(g), eps=1e-5).numpy()
    np.testing.assert_allclose(oracle.rmsnorm(x, g, 1e-5), ref, rtol=1e-13, atol=1e-14)
    y = oracle.rmsnorm(x * 1e3, np.ones(33), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=1)), 1.0, rtol=1e-12)


def test_attention_identical_keys_average_values():
    rng = np.random.default_rng(2)
    q = rng.standard_normal((4, 8))
    k = np.tile(rng.standard_normal((1, 8)), (6, 1))
    v = rng.standard_normal((6, 8))
    np.testing.assert_allclose(oracle.attention(q, k, v, 1), np.tile(v.mean(0), (4, 1)), rtol=1e-12)


def test_attention_single_key_returns_value():
    rng = np.random.default_rng(3)
    q, k, v = rng.standard_normal((5, 16)), rng.standard_normal((1, 16)), rng.standard_normal((1, 16))
    np.testing.assert_allclose(oracle.attention(q, k, v, 2), np.tile(v, (5, 1)), rtol=1e-12)


def test_attention_rows_sum_to_one_eq11():
    rng = np.random.default_rng(4)
    A = oracle.attention_weights(rng.standard_normal((7, 16)) * 5, rng.standard_normal((30, 16)) * 5)
    np.testing.assert_allclose(A.sum(1), 1.0, rtol=1e-13)
    assert (A >= 0).all()


def test_attention_matches_torch_sdpa_bidirectional():
    rng = np.random.default_rng(5)
    H, dh, Lq, Lk = 3, 16, 9, 13
    q, k, v = (rng.standard_normal((L, H * dh)) for L in (Lq, Lk, Lk))
    got = oracle.attention(q, k, v, H)
    th = lambda a: t(a).view(a.shape[0], H, dh).transpose(0, 1)
    ref = TF.scaled_dot_product_attention(th(q), th(k), th(v), is_causal=False)
    np.testing.assert_allclose(got, ref.transpose(0, 1).reshape(Lq, H * dh).numpy(), rtol=1e-11, atol=1e-12)


def test_attention_key_permutation_invariance():
    rng = np.random.default_rng(6)
    q, k, v = rng.standard_normal((3, 8)), rng.standard_normal((10, 8)), rng.standard_normal((10, 8))
    p = rng.permutation(10)
    np.testing.assert_allclose(oracle.attention(q, k, v, 2), oracle.attention(q, k[p], v[p], 2), rtol=1e-12)


def _torch_layer(x, w, H, kv=None, dtype=None):
    """The same block through torch library ops (fp64), rounding at the same storage points."""
    R = (lambda a: a.to(torch.bfloat16).to(torch.float64)) if dtype == "bf16" else (lambda a: a)
    x = t(x)
    L, d = x.shape
    kv = L if kv is None else kv
    W = {k_: t(v_) for k_, v_ in w.items()}
    xn = R(TF.rms_norm(x, (d,), weight=W["g_attn"], eps=1e-5))
    q, k, v = R(TF.linear(xn, W["wq"])), R(TF.linear(xn[:kv], W["wk"])), R(TF.linear(xn[:kv], W["wv"]))
    dh = d // H
    sh = lambda a: a.view(a.shape[0], H, dh).transpose(0, 1)
    o = R(TF.scaled_dot_product_attention(sh(q), sh(k), sh(v)).transpose(0, 1).reshape(L, d))
    h = R(x + TF.linear(o, W["wo"]))
    hn = R(TF.rms_norm(h, (d,), weight=W["g_mlp"], eps=1e-5))
    a = R(TF.silu(TF.linear(hn, W["wg"])) * TF.linear(hn, W["wu"]))
    return R(h + TF.linear(a, W["wd"])).numpy()


def _tiny(dtype="f32", d=32, H=4, F=48, seed=0):
    wl = synth.tiny_workload(dtype=dtype, d=d, n_heads=H, head_dim=d // H, d_ff=F, seed=seed)
    w = synth.layer_weights(wl, 0)
    rng = np.random.default_rng(seed)
    w["g_attn"] = (1 + 0.1 * rng.standard_normal(d)).astype(np.float32)
    w["g_mlp"] = (1 + 0.1 * rng.standard_normal(d)).astype(np.float32)
    return wl, w


@pytest.mark.parametrize("kv", [None, 9])
def test_layer_matches_torch_fp64(kv):
    wl, w = _tiny()
    x = np.random.default_rng(7).standard_normal((13, 32))
    np.testing.assert_allclose(oracle.layer_forward_segment(x, w, 4, kv_len=kv), _torch_layer(x, w, 4, kv),
                               rtol=1e-11, atol=1e-12)


def test_layer_bf16_storage_points_match_torch():
    wl, w = _tiny("bf16", d=64, H=2, F=96, seed=3)
    x = synth.round_storage(np.random.default_rng(8).standard_normal((21, 64)), "bf16")
    got = oracle.layer_forward_segment(x, w, 2, dtype="bf16")
    ref = _torch_layer(x, w, 2, dtype="bf16")
    # torch narrows fp64 -> fp32 -> bf16 (double rounding); allow one bf16 ulp on rare ties
    assert np.mean(got == ref) > 0.99
    np.testing.assert_allclose(got, ref, rtol=2 ** -7, atol=1e-6)


def test_layer_zero_projections_reduce_to_identity():
    wl, w = _tiny(seed=1)
    x = np.random.default_rng(9).standard_normal((6, 32))
    w0 = dict(w, wo=np.zeros_like(w["wo"]), wd=np.zeros_like(w["wd"]))
    np.testing.assert_array_equal(oracle.layer_forward_segment(x, w0, 4), x)


def test_segments_are_independent_and_permutable():
    wl, w = _tiny(seed=2)
    rng = np.random.default_rng(10)
    segs = [rng.standard_normal((n, 32)) for n in (5, 11, 3)]
    cu = np.concatenate([[0], np.cumsum([len(s) for s in segs])])
    y = oracle.layer_forward_packed(np.concatenate(segs), cu, w, 4)
    for i, s in enumerate(segs):
        np.testing.assert_allclose(y[cu[i]:cu[i + 1]], oracle.layer_forward_segment(s, w, 4), rtol=0, atol=0)
    order = [2, 0, 1]
    cu2 = np.concatenate([[0], np.cumsum([len(segs[i]) for i in order])])
    y2 = oracle.layer_forward_packed(np.concatenate([segs[i] for i in order]), cu2, w, 4)
    for j, i in enumerate(order):
        np.testing.assert_array_equal(y2[cu2[j]:cu2[j + 1]], y[cu[i]:cu[i + 1]])


def test_untruncated_equals_padded_forward_with_key_mask():
    # padding rows appended after kv_len never change the valid rows (Eq. 9-10 vs Eq. 6-7)
    wl, w = _tiny(seed=4)
    rng = np.random.default_rng(11)
    x = rng.standard_normal((10, 32))
    junk = 1e3 * rng.standard_normal((6, 32))
    y = oracle.layer_forward_segment(x, w, 4)
    y_pad = oracle.layer_forward_segment(np.concatenate([x, junk]), w, 4, kv_len=10)
    np.testing.assert_allclose(y_pad[:10], y, rtol=1e-12, atol=1e-12)


def test_truncation_changes_outputs_only_through_removed_keys():
    wl, w = _tiny(seed=5)
    x = np.random.default_rng(12).standard_normal((12, 32))
    full = oracle.layer_forward_segment(x, w, 4)
    trunc = oracle.layer_forward_segment(x[:8], w, 4)
    assert not np.allclose(full[:8], trunc)        # the suffix did leak into the prefix (Eq. 6)
    np.testing.assert_allclose(oracle.layer_forward_segment(x, w, 4, kv_len=8)[:8], trunc, rtol=1e-12)


def test_rows_variant_matches_full_segment():
    for dtype in (None, "bf16"):
        wl, w = _tiny("bf16" if dtype else "f32", d=64, H=2, F=96, seed=6)
        x = synth.round_storage(np.random.default_rng(13).standard_normal((17, 64)), "bf16")
        full = oracle.layer_forward_segment(x, w, 2, kv_len=14, dtype=dtype)
        rows = [0, 5, 13, 16]
        got = oracle.layer_forward_rows(x, w, 2, rows, kv_len=14, dtype=dtype)
        # BLAS may sum in another order for a different row count: 1 ulp of fp64,
        # which a bf16 rounding step can turn into one bf16 ulp on a rare tie
        np.testing.assert_allclose(got, full[rows], rtol=1e-12 if dtype is None else 2 ** -7, atol=1e-12)
        assert np.mean(got == full[rows]) > 0.9


def test_count_hook_equals_detector_on_mlp_input():
    wl, w = _tiny(seed=7)
    x = np.random.default_rng(14).standard_normal((9, 32))
    parts = oracle.layer_forward_segment(x, w, 4, return_parts=True, count_rows=[2, 3, 8], act_eps=0.05)
    ref = oracle.sparsity_counts(parts["hn"][[2, 3, 8]], w["wg"], w["wu"], 0.05)
    np.testing.assert_array_equal(parts["counts"], ref)


def test_rows_variant_counts_equal_full_segment_hook():
    wl, w = _tiny(seed=8)
    x = np.random.default_rng(15).standard_normal((11, 32))
    rows = [1, 4, 10]
    _, counts = oracle.layer_forward_rows(x, w, 4, rows, kv_len=9, act_eps=0.05)
    full = oracle.layer_forward_segment(x, w, 4, kv_len=9, count_rows=rows, act_eps=0.05, return_parts=True)
    np.testing.assert_array_equal(counts, full["counts"])
