"""Pins of the oracle's prefix key/value caching (the composition of truncation
with KV caching that Table 7 reports)."""
import numpy as np
import pytest

import oracle
import synth


def _w(seed, dtype="f32", d=32, H=4, F=48):
    wl = synth.tiny_workload(dtype=dtype, d=d, n_heads=H, head_dim=d // H, d_ff=F, seed=seed)
    return synth.layer_weights(wl, 0)


@pytest.mark.parametrize("dtype", [None, "bf16"])
def test_cached_response_rows_equal_full_layer_rows(dtype):
    # with the cache filled from the same layer input, caching is exact: the
    # response rows' outputs equal those of the block over [prefix ; response]
    w = _w(1, "bf16" if dtype else "f32")
    rng = np.random.default_rng(2)
    x = synth.round_storage(rng.standard_normal((19, 32)), "bf16")
    ctx = 12
    full = oracle.layer_forward_segment(x, w, 4, dtype=dtype)
    k, v = oracle.kv_prefill(x[:ctx], w, 4, dtype=dtype)
    got = oracle.layer_forward_cached(x[ctx:], k, v, w, 4, dtype=dtype)
    np.testing.assert_allclose(got, full[ctx:], rtol=1e-12 if dtype is None else 2 ** -7, atol=1e-12)


def test_cached_padding_rows_are_never_keys():
    w = _w(3)
    rng = np.random.default_rng(4)
    x = rng.standard_normal((15, 32))
    ctx, valid = 9, 4                       # 9 prefix rows, 4 valid response rows, 2 padding rows
    full = oracle.layer_forward_segment(x, w, 4, kv_len=ctx + valid)
    k, v = oracle.kv_prefill(x[:ctx], w, 4)
    got = oracle.layer_forward_cached(x[ctx:], k, v, w, 4, kv_valid=valid)
    np.testing.assert_allclose(got, full[ctx:], rtol=1e-12, atol=1e-12)


def test_empty_prefix_is_the_plain_block():
    w = _w(5)
    x = np.random.default_rng(6).standard_normal((7, 32))
    z = np.zeros((0, 32))
    np.testing.assert_allclose(oracle.layer_forward_cached(x, z, z, w, 4), oracle.layer_forward_segment(x, w, 4),
                               rtol=1e-12, atol=1e-12)


def test_prefill_matches_the_blocks_key_value_projections():
    w = _w(7)
    x = np.random.default_rng(8).standard_normal((10, 32))
    parts = oracle.layer_forward_segment(x, w, 4, return_parts=True)
    k, v = oracle.kv_prefill(x[:6], w, 4)
    np.testing.assert_allclose(k, parts["k"][:6], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(v, parts["v"][:6], rtol=1e-12, atol=1e-12)


def test_stale_cache_changes_the_result():
    # a cache computed from other prefix states is not the same computation
    w = _w(9)
    rng = np.random.default_rng(10)
    x = rng.standard_normal((14, 32))
    k, v = oracle.kv_prefill(x[:8] + 0.5, w, 4)
    got = oracle.layer_forward_cached(x[8:], k, v, w, 4)
    assert not np.allclose(got, oracle.layer_forward_segment(x, w, 4)[8:])
