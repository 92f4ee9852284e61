"""The oracle against brute force on tiny inputs: attention (Eqs. 6-7), the
SwiGLU MLP and its near-zero counts, RMSNorm, written as plain Python loops
over scalars (math module only)."""
import math

import numpy as np

import oracle


def _attention_loops(q, k, v, H):
    L, D = len(q), len(q[0])
    dh = D // H
    out = [[0.0] * D for _ in range(L)]
    for h in range(H):
        for i in range(L):
            e = []
            for j in range(len(k)):
                dot = 0.0
                for c in range(dh):
                    dot += q[i][h * dh + c] * k[j][h * dh + c]
                e.append(dot / math.sqrt(dh))
            m = max(e)
            w = [math.exp(x - m) for x in e]
            z = sum(w)
            for c in range(dh):
                acc = 0.0
                for j in range(len(k)):
                    acc += w[j] / z * v[j][h * dh + c]
                out[i][h * dh + c] = acc
    return out


def _mlp_loops(x, wg, wu, wd, eps):
    F, d = len(wg), len(x)
    a, count = [], 0
    for f in range(F):
        g = sum(x[c] * wg[f][c] for c in range(d))
        u = sum(x[c] * wu[f][c] for c in range(d))
        af = g / (1.0 + math.exp(-g)) * u
        a.append(af)
        count += 1 if abs(af) < eps else 0
    y = [sum(a[f] * wd[c][f] for f in range(F)) for c in range(d)]
    return a, count, y


def test_attention_matches_loops_with_fewer_keys_than_queries():
    rng = np.random.default_rng(0)
    H, dh = 2, 4
    q = rng.standard_normal((5, H * dh))
    k = rng.standard_normal((3, H * dh))
    v = rng.standard_normal((3, H * dh))
    ref = np.array(_attention_loops(q.tolist(), k.tolist(), v.tolist(), H))
    np.testing.assert_allclose(oracle.attention(q, k, v, H), ref, rtol=1e-12, atol=1e-12)


def test_swiglu_mlp_and_counts_match_loops():
    rng = np.random.default_rng(1)
    d, F = 6, 9
    x = rng.standard_normal(d)
    wg, wu, wd = rng.standard_normal((F, d)), rng.standard_normal((F, d)), rng.standard_normal((d, F))
    a_ref, count_ref, y_ref = _mlp_loops(x.tolist(), wg.tolist(), wu.tolist(), wd.tolist(), 0.3)
    a = oracle.swiglu_activation(x[None, :], wg, wu)[0]
    np.testing.assert_allclose(a, a_ref, rtol=1e-12, atol=1e-12)
    assert int(oracle.sparsity_counts(x[None, :], wg, wu, 0.3)[0]) == count_ref
    np.testing.assert_allclose(a @ wd.T, y_ref, rtol=1e-12, atol=1e-12)


def test_rmsnorm_matches_loops():
    rng = np.random.default_rng(2)
    x, g = rng.standard_normal(7), rng.standard_normal(7)
    ms = sum(v * v for v in x) / 7
    ref = [x[c] / math.sqrt(ms + 1e-5) * g[c] for c in range(7)]
    np.testing.assert_allclose(oracle.rmsnorm(x[None, :], g)[0], ref, rtol=1e-12, atol=1e-12)
