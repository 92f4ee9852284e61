"""Pins of the oracle's routing and compaction layout (Sec. 3.4 Eqs. 3-4, Sec. 3.5)."""
import json
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _cases(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)["cases"]


@pytest.mark.parametrize("case", _cases("routing_cases.json"), ids=lambda c: c["name"])
def test_route_golden(case):
    got = oracle.route(case["L_star"], case["N"], case["tau_pad"], bucket_min=case.get("bucket_min", 8))
    assert len(got) == len(case["groups"])
    for g, e in zip(got, case["groups"]):
        assert g["bucket"] == e["bucket"] and g["members"] == e["members"] and g["path"] == e["path"]
        assert abs(g["rho"] - e["rho"]) < 1e-12


def test_bucket_set_shape():
    assert oracle.bucket_set(1024) == [8, 16, 32, 64, 128, 256, 512, 1024]
    assert oracle.bucket_set(100) == [8, 16, 32, 64, 100]
    assert oracle.bucket_set(8) == [8]
    assert oracle.bucket_set(1024, 64) == [64, 128, 256, 512, 1024]
    assert oracle.bucket_set(50, 64) == [50]
    assert oracle.bucket_set(100, 1) == [1, 2, 4, 8, 16, 32, 64, 100]
    for N in (100, 512, 2048):
        for L in range(1, N + 1, 7):
            b = oracle.bucket_of(L, N)
            smaller = [x for x in oracle.bucket_set(N) if x < b]
            assert L <= b and all(L > x for x in smaller)


def test_pwr_closed_form():
    assert oracle.padding_waste_ratio([64, 64, 64], 64) == 0.0
    assert oracle.padding_waste_ratio([1], 8) == 0.875
    rng = np.random.default_rng(0)
    for _ in range(100):
        B = int(rng.integers(8, 1025))
        L = rng.integers(1, B + 1, size=int(rng.integers(1, 9)))
        r = oracle.padding_waste_ratio(L, B)
        assert 0.0 <= r < 1.0
        assert abs(r - (len(L) * B - L.sum()) / (len(L) * B)) < 1e-12


def test_batch_max_is_single_group_when_lengths_share_a_bucket():
    # Eq. 3: one group holding every sequence is padded to bucket(max L*)
    L = [130, 200, 256, 190]
    g = oracle.route(L, 1024)
    assert len(g) == 1 and g[0]["bucket"] == oracle.bucket_of(max(L), 1024)


def test_segment_layout_static_pads_varlen_packs():
    ctx = np.array([100, 50, 70, 30, 10])
    L = np.array([120, 128, 65, 70, 300])   # 0,1 -> bucket 128 static (rho .047); 2,3 -> 128? no: 65,70 -> 128
    seg, kv, cu = oracle.segment_layout(ctx, L, 1024)
    groups = oracle.route(L, 1024)
    assert groups[0]["bucket"] == 128 and groups[0]["members"] == [0, 1, 2, 3]
    # rho = 1 - 383/512 = 0.252 > 0.2 -> varlen: exact rows
    assert groups[0]["path"] == oracle.PATH_VARLEN
    assert list(seg) == list(ctx + L) and list(kv) == list(ctx + L)
    assert list(cu) == [0] + list(np.cumsum(ctx + L))
    L2 = np.array([120, 128, 110, 125, 300])
    seg2, kv2, _ = oracle.segment_layout(ctx, L2, 1024)
    assert list(seg2[:4]) == list(ctx[:4] + 128) and seg2[4] == ctx[4] + 300
    assert list(kv2) == list(ctx + L2)


def test_pack_rows_keeps_prefix_rows_in_order():
    rng = np.random.default_rng(4)
    full = np.array([7, 3, 9])
    cu = np.concatenate([[0], np.cumsum(full)])
    x = rng.standard_normal((cu[-1], 5))
    seg = np.array([4, 3, 0])
    p = oracle.pack_rows(x, cu, seg)
    assert p.shape == (7, 5)
    np.testing.assert_array_equal(p[:4], x[0:4])
    np.testing.assert_array_equal(p[4:7], x[7:10])
