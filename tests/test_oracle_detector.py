"""Pins of the oracle's detector (Sec. 3.2 sparsity count, Sec. 3.3 SNR scan)."""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as TF

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _cases(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)["cases"]


@pytest.mark.parametrize("case", _cases("snr_cases.json"), ids=lambda c: c["name"])
def test_snr_golden(case):
    i_star, L_star = oracle.snr_boundary(case["counts"], case["F"], case["tau_jump"], case["gamma"],
                                         case["window"])
    assert (i_star, L_star) == (case["i_star"], case["L_star"])


def test_snr_batch_matches_rows():
    rng = np.random.default_rng(3)
    counts = rng.integers(0, 4, size=(6, 40))
    counts[2, 17:] += 40
    i_s, L_s = oracle.snr_boundaries(counts, 100)
    for b in range(6):
        assert (i_s[b], L_s[b]) == oracle.snr_boundary(counts[b], 100)
    assert (i_s[2], L_s[2]) == (17, 18)


def test_snr_scale_invariance_of_fraction():
    # the test is on fractions c/F: doubling both counts and F cannot move i*
    rng = np.random.default_rng(5)
    for _ in range(50):
        c = rng.integers(0, 64, size=30)
        assert oracle.snr_boundary(c, 64) == oracle.snr_boundary(2 * c, 128)


def test_silu_matches_torch():
    x = np.linspace(-30, 30, 2001)
    ref = TF.silu(torch.from_numpy(x)).numpy()
    np.testing.assert_allclose(oracle.silu(x), ref, rtol=1e-14, atol=1e-300)


def test_swiglu_matches_torch_composition():
    # non-square shapes so a transposed operand cannot pass
    rng = np.random.default_rng(1)
    x, wg, wu = rng.standard_normal((5, 7)), rng.standard_normal((11, 7)), rng.standard_normal((11, 7))
    t = lambda a: torch.from_numpy(a)
    ref = (TF.silu(TF.linear(t(x), t(wg))) * TF.linear(t(x), t(wu))).numpy()
    np.testing.assert_allclose(oracle.swiglu_activation(x, wg, wu), ref, rtol=1e-13, atol=1e-13)


def test_counts_zero_input_is_all_sparse():
    rng = np.random.default_rng(2)
    wg, wu = rng.standard_normal((33, 8)), rng.standard_normal((33, 8))
    assert list(oracle.sparsity_counts(np.zeros((3, 8)), wg, wu, 1e-6)) == [33, 33, 33]


def test_counts_hand_values():
    # d = 1, x = 1, Wu = 1: a_j = silu(g_j).  silu(0)=0, silu(+-1e-3)=+-5.0e-4,
    # silu(0.5)=0.311, silu(-20)=-4.1e-8, silu(3)=2.86; eps=1e-3 -> 4 near zero.
    g = np.array([[0.0], [1e-3], [-1e-3], [0.5], [-20.0], [3.0]])
    assert oracle.sparsity_counts(np.ones((1, 1)), g, np.ones((6, 1)), 1e-3)[0] == 4
    # strict inequality: |a| == eps is not counted
    assert oracle.sparsity_counts(np.ones((1, 1)), np.full((1, 1), 50.0), np.full((1, 1), 0.25), 0.25)[0] == 0


def _planted_check(wl, lens=None):
    lens = lens or synth.lengths(wl)
    x, cu, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    N = lens.window
    out = []
    for b in range(wl.batch):
        rows = x[resp[b]:resp[b] + N]
        c = oracle.sparsity_counts(rows, w["wg"], w["wu"], wl.act_eps)
        i_s, L_s = oracle.snr_boundary(c, wl.d_ff)
        out.append((int(lens.boundary[b]), i_s, L_s, c))
    return out


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_planted_boundary_recovered_tiny(seed, dtype):
    wl = synth.tiny_workload(dtype=dtype, seed=100 + seed, window=96, boundary=("uniform", 8, 90),
                             visual=("fixed", 8), prompt=("fixed", 4))
    for b, i_s, L_s, c in _planted_check(wl):
        assert (i_s, L_s) == (b, b + 1)


@pytest.mark.parametrize("index", [0, 1])
def test_planted_boundary_recovered_workload(index):
    wl = synth.workload(index)
    for b, i_s, L_s, c in _planted_check(wl):
        assert (i_s, L_s) == (b, b + 1)
        s = c / wl.d_ff
        assert 0.0 < s[:b].mean() < 0.06           # valid region: a few percent sparse
        assert s[b:].mean() > 0.3                  # planted padding plateau
        assert s[:b].std() < 0.02
