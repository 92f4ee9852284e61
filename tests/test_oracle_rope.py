"""Pins of the oracle's optional rotary embedding (the RoFormer rotation in the
half-split layout; the paper names no positional scheme, so this is the
optional reading of the block, off unless rope_theta > 0)."""
import math

import numpy as np
import pytest

import oracle
import synth


def test_rope_equals_complex_rotation():
    # RoFormer's own statement: pair (a, b) is the complex number a + ib multiplied by exp(i * pos * freq)
    rng = np.random.default_rng(0)
    H, dh, L, theta = 3, 8, 11, 500.0
    x = rng.standard_normal((L, H * dh))
    pos = rng.integers(0, 4000, L)
    got = oracle.rope(x, pos, H, theta)
    freq = np.array([theta ** (-(2.0 * i) / dh) for i in range(dh // 2)])
    for h in range(H):
        z = x[:, h * dh:h * dh + dh // 2] + 1j * x[:, h * dh + dh // 2:(h + 1) * dh]
        zr = z * np.exp(1j * pos[:, None] * freq[None, :])
        np.testing.assert_allclose(got[:, h * dh:h * dh + dh // 2], zr.real, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(got[:, h * dh + dh // 2:(h + 1) * dh], zr.imag, rtol=1e-12, atol=1e-12)


def test_rope_quarter_turn_closed_form():
    # theta = 1e4, dh = 4: frequencies 1 and 1e-2.  At pos = 50*pi pair 1 turns by pi/2
    # ((1, 0) -> (0, 1)) and pair 0 by 25 full turns (unchanged).
    x = np.array([[1.0, 1.0, 0.0, 0.0]])
    got = oracle.rope(x, [50 * math.pi], 1, 1e4)
    np.testing.assert_allclose(got, [[1.0, 0.0, 0.0, 1.0]], atol=1e-12)


def test_rope_identity_cases():
    x = np.random.default_rng(1).standard_normal((5, 16))
    np.testing.assert_array_equal(oracle.rope(x, np.zeros(5), 2, 1e4), x)
    np.testing.assert_array_equal(oracle.rope(x, np.arange(5), 2, 0.0), x)


def test_rope_preserves_pair_norms_and_is_relative():
    rng = np.random.default_rng(2)
    H, dh = 2, 16
    q, k = rng.standard_normal((1, H * dh)), rng.standard_normal((1, H * dh))
    rq = oracle.rope(q, [37], H, 1e4)
    half = dh // 2
    for h in range(H):
        a, b = slice(h * dh, h * dh + half), slice(h * dh + half, (h + 1) * dh)
        np.testing.assert_allclose(rq[0, a] ** 2 + rq[0, b] ** 2, q[0, a] ** 2 + q[0, b] ** 2, rtol=1e-12)
    # scores depend on the position difference only
    for m, n, s in ((3, 10, 100), (0, 0, 999), (500, 7, 33)):
        for h in range(H):
            c = slice(h * dh, (h + 1) * dh)
            d1 = oracle.rope(q, [m], H, 1e4)[0, c] @ oracle.rope(k, [n], H, 1e4)[0, c]
            d2 = oracle.rope(q, [m + s], H, 1e4)[0, c] @ oracle.rope(k, [n + s], H, 1e4)[0, c]
            assert abs(d1 - d2) < 1e-10


def _tiny(seed):
    wl = synth.tiny_workload(dtype="f32", d=32, n_heads=4, head_dim=8, d_ff=48, seed=seed)
    return synth.layer_weights(wl, 0)


def test_layer_with_rope_positions_restart_per_segment():
    w = _tiny(3)
    rng = np.random.default_rng(4)
    segs = [rng.standard_normal((n, 32)) for n in (6, 9)]
    cu = np.array([0, 6, 15])
    y = oracle.layer_forward_packed(np.concatenate(segs), cu, w, 4, rope_theta=1e4)
    for i, s in enumerate(segs):
        np.testing.assert_allclose(y[cu[i]:cu[i + 1]], oracle.layer_forward_segment(s, w, 4, rope_theta=1e4),
                                   rtol=0, atol=0)
    assert not np.allclose(y[:6], oracle.layer_forward_segment(segs[0], w, 4))   # the rotation acts


def test_layer_with_rope_truncation_and_rows_invariants():
    w = _tiny(5)
    x = np.random.default_rng(6).standard_normal((12, 32))
    trunc = oracle.layer_forward_segment(x[:8], w, 4, rope_theta=1e4)
    masked = oracle.layer_forward_segment(x, w, 4, kv_len=8, rope_theta=1e4)
    np.testing.assert_allclose(masked[:8], trunc, rtol=1e-12, atol=1e-12)
    rows = [0, 4, 11]
    full = oracle.layer_forward_segment(x, w, 4, kv_len=10, rope_theta=1e4)
    got = oracle.layer_forward_rows(x, w, 4, rows, kv_len=10, rope_theta=1e4)
    np.testing.assert_allclose(got, full[rows], rtol=1e-12, atol=1e-12)


def test_layer_rope_leaves_values_unrotated():
    # with a single key the output is that key's value row, whatever the rotation
    w = _tiny(7)
    x = np.random.default_rng(8).standard_normal((5, 32))
    a = oracle.layer_forward_segment(x, w, 4, kv_len=1, rope_theta=1e4, return_parts=True)
    b = oracle.layer_forward_segment(x, w, 4, kv_len=1, return_parts=True)
    np.testing.assert_allclose(a["o"], b["o"], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(a["o"], np.repeat(b["v"][:1], 5, axis=0), rtol=1e-12, atol=1e-12)
