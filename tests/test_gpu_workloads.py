"""Full-size parity of the ragged workloads (2: batch 16, window 1024; 4: batch 4,
11.8k-row video prefixes, window 2048) in the launch configuration bench.py times.

The oracle cannot redo every row at these sizes, so it checks what it can
compute one by one: every boundary (bit exact, planted), every packed row (bit
exact), the near-zero counts of every token of whole windows (two or three
sequences, every 128-row tile of the window) and around every other boundary,
and the layer output of sampled
query rows of the shortest and longest (and for workload 2 a middle) segment,
with keys/values from all of that segment's kept rows.  Rows past the packed
total must stay untouched.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import check_close, check_counts
from tests.test_gpu_layer import run_path

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    assert S.seer_check_device() == 0


def _sample_rows(L, ctx, Ls, rng, n_random=24):
    rows = {0, L - 1, ctx, ctx - 1, min(L - 1, ctx + Ls - 1), L // 2}
    rows.update(int(v) for v in rng.integers(0, L, size=n_random))
    return sorted(r for r in rows if 0 <= r < L)


@pytest.mark.parametrize("index", [2, 4])
def test_workload_full_size_sampled(index):
    wl = synth.workload(index)
    r = run_path(wl, extra_cap=0)
    lens = r["lens"]
    np.testing.assert_array_equal(r["L"], lens.boundary + 1)
    seg, kv, cu = oracle.segment_layout(lens.ctx, r["L"], wl.window)
    np.testing.assert_array_equal(r["cu"], cu)
    np.testing.assert_array_equal(r["kv"], kv)
    T = int(cu[-1])
    for b in range(wl.batch):                       # packed rows, bit exact
        np.testing.assert_array_equal(r["xp"][cu[b]:cu[b + 1]], r["x"][r["cu_full"][b]:r["cu_full"][b] + seg[b]])
    assert (r["y"][T:] == 9.0).all()                # zero work past the packed total
    x, resp, w = r["x"], r["resp"], r["w"]
    F = wl.d_ff
    order = np.argsort(seg)
    # counts: every token of the whole window (all of its 128-row tiles) of the
    # sequences with the shortest and longest kept segment (plus a middle one for
    # workload 2), and around every other sequence's boundary
    whole = {int(order[0]), int(order[-1])} | ({int(order[len(order) // 2])} if index == 2 else set())
    for b in range(wl.batch):
        if b in whole:
            rows = np.arange(wl.window)
        else:
            bb = int(lens.boundary[b])
            rows = np.arange(max(0, bb - 4), min(wl.window, bb + 5))
        ref = oracle.sparsity_counts(x[resp[b] + rows], w["wg"], w["wu"], wl.act_eps)
        check_counts(r["counts"][b, rows], ref, F, f"workload {index} window {b}")
    rng = np.random.default_rng(index)
    picks = [order[0], order[-1]] + ([order[len(order) // 2]] if index == 2 else [])
    for b in picks:
        L = int(seg[b])
        rows = _sample_rows(L, int(lens.ctx[b]), int(r["L"][b]), rng)
        x_seg = r["xp"][cu[b]:cu[b + 1]]
        ref = oracle.layer_forward_rows(x_seg, w, wl.n_heads, rows, kv_len=int(kv[b]))
        got = r["y"][cu[b] + np.asarray(rows)]
        check_close(got, ref, wl.dtype, f"workload {index} segment {b} ({L} rows)")
