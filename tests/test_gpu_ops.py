"""GPU parity of each hot-path step, called through the C ABI, against the oracle.

Sizes span several 128-row tiles with ragged tails.  16-bit outputs compare at
|err| <= 1e-2 + 1e-2 |ref| against the exact fp64 result of the same inputs,
fp32 outputs at 1e-4 + 1e-4 |ref|; integer outputs compare exactly.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import check_close, cuda, host, i32, tdtype, to_dev

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    assert S.seer_check_device() == 0


def _rng(seed):
    return np.random.default_rng(seed)


def _store(a, dt):
    """Values representable in storage type dt (f16 via torch's converter)."""
    if dt == "f16":
        return torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.float16).float().numpy()
    return synth.round_storage(a, dt)


# ------------------------------------------------------------------ linear (S6, S8, S11)
@pytest.mark.parametrize("M,N,K", [(300, 512, 256), (128, 256, 64), (1, 256, 128), (777, 768, 512), (129, 256, 4096)])
@pytest.mark.parametrize("op,res,out", [("bf16", None, "bf16"), ("bf16", "bf16", "bf16"), ("f16", "bf16", "f16"),
                                        ("f16", "f16", "bf16")])
def test_linear_16bit(M, N, K, op, res, out):
    rng = _rng(M + N + K)
    a, w = _store(rng.standard_normal((M, K)), op), _store(0.05 * rng.standard_normal((N, K)), op)
    r = _store(rng.standard_normal((M, N)), res) if res else None
    ref = a.astype(np.float64) @ w.astype(np.float64).T + (r if res else 0.0)
    c = torch.full((M, N), float("nan"), dtype=tdtype(out), device=cuda())
    S.seer_linear(to_dev(a, op), to_dev(w, op), op, to_dev(r, res) if res else None, res or out, c, out, M, None, N, K)
    check_close(host(c), ref, "bf16", f"linear {M}x{N}x{K} {op}/{res}/{out}")


def test_linear_device_row_count_leaves_tail_untouched():
    rng = _rng(5)
    M_cap, M, N, K = 512, 333, 256, 128
    a, w = _store(rng.standard_normal((M_cap, K)), "f16"), _store(0.05 * rng.standard_normal((N, K)), "f16")
    c = torch.full((M_cap, N), 7.0, dtype=torch.float16, device=cuda())
    S.seer_linear(to_dev(a, "f16"), to_dev(w, "f16"), "f16", None, "f16", c, "f16", M_cap, i32([M]), N, K)
    out = host(c)
    check_close(out[:M], a[:M].astype(np.float64) @ w.astype(np.float64).T, "bf16", "linear M_dev")
    assert (out[M:] == 7.0).all()   # zero work past the device row count


def test_linear_f32():
    rng = _rng(6)
    M, N, K = 70, 52, 36
    a, w, r = (x.astype(np.float32) for x in (rng.standard_normal((M, K)), rng.standard_normal((N, K)),
                                              rng.standard_normal((M, N))))
    c = torch.empty((M, N), dtype=torch.float32, device=cuda())
    S.seer_linear(to_dev(a, "f32"), to_dev(w, "f32"), "f32", to_dev(r, "f32"), "f32", c, "f32", M, None, N, K)
    check_close(host(c), a.astype(np.float64) @ w.astype(np.float64).T + r, "f32", "linear f32")


# ------------------------------------------------------------------ SwiGLU + count hook (S10, S1)
@pytest.mark.parametrize("op", ["bf16", "f16", "f32"])
def test_swiglu_with_count_hook(op):
    rng = _rng(7)
    M, F, K = 400, 384, 256
    x = _store(rng.standard_normal((M, K)), op)
    wg = _store(0.02 * rng.standard_normal((F, K)), op)
    wu = _store(0.02 * rng.standard_normal((F, K)), op)
    cu = np.array([0, 150, 290, 400])
    resp = np.array([100, 200, 350])
    Nw, eps = 64, 3e-4
    ref_act = oracle.swiglu_activation(x, wg, wu)
    ref_cnt = np.zeros((3, Nw), dtype=np.int64)
    for b in range(3):
        for t in range(Nw):
            r = resp[b] + t
            if r < cu[b + 1]:
                ref_cnt[b, t] = oracle.sparsity_counts(x[r:r + 1], wg, wu, eps)[0]
    act = torch.empty((M, F), dtype=tdtype(op), device=cuda())
    counts = torch.full((3 * Nw,), -1, dtype=torch.int32, device=cuda())
    S.seer_swiglu(to_dev(x, op), to_dev(wg, op), to_dev(wu, op), op, act, op, M, None, F, K, i32(cu), 3,
                  i32(resp), Nw, eps, counts)
    check_close(host(act), ref_act, "f32" if op == "f32" else "bf16", "swiglu act")
    got = counts.cpu().numpy().reshape(3, Nw)
    assert np.abs(got - ref_cnt).max() <= 0.005 * F
    assert ref_cnt.sum() > 0 and np.mean(got == ref_cnt) > 0.9


# ------------------------------------------------------------------ RMSNorm (S5, S9)
# 16-bit rows up to 4096 wide run the register-resident kernel (4, 8 or 16 vectors
# per lane, ragged widths masked); wider rows and fp32 the streaming one
@pytest.mark.parametrize("x_dt,y_dt,d", [("bf16", "f16", 4096), ("f16", "f16", 256), ("bf16", "bf16", 256),
                                         ("f32", "f32", 264), ("bf16", "f16", 1024), ("bf16", "f16", 3072),
                                         ("f16", "f16", 264), ("bf16", "f16", 8192)])
def test_rmsnorm(x_dt, y_dt, d):
    rng = _rng(8)
    M = 333
    x = _store(3 * rng.standard_normal((M, d)), x_dt)
    g = _store(1 + 0.1 * rng.standard_normal(d), y_dt)
    y = torch.empty((M, d), dtype=tdtype(y_dt), device=cuda())
    S.seer_rmsnorm(to_dev(x, x_dt), x_dt, to_dev(g, y_dt), y, y_dt, M, None, d, 1e-5)
    check_close(host(y), oracle.rmsnorm(x, g, 1e-5), "f32" if y_dt == "f32" else "bf16", "rmsnorm")


def test_convert_bf16_to_f16_is_exact_in_range():
    rng = _rng(9)
    v = _store(rng.standard_normal(4096) * np.exp(rng.uniform(-9, 9, 4096)), "bf16")
    src = to_dev(v, "bf16")
    dst = torch.empty(4096, dtype=torch.float16, device=cuda())
    S.seer_convert(src, "bf16", dst, "f16", 4096)
    got = host(dst)
    normal = (np.abs(v) >= 2.0 ** -14) & (np.abs(v) < 65504)
    np.testing.assert_array_equal(got[normal], v[normal])


# ------------------------------------------------------------------ attention (S7)
def _attention_case(dt, H, dh, lens, kv, scale, seed, structured=False):
    rng = _rng(seed)
    D = H * dh
    cu = np.concatenate([[0], np.cumsum(lens)])
    T = int(cu[-1])
    T_cap = T + 37
    qkv = scale * rng.standard_normal((T_cap, 3 * D))
    if structured:
        for b in range(len(lens)):
            j = np.arange(lens[b])
            for h in range(H):
                qkv[cu[b]:cu[b + 1], h * dh] = 18.0
                qkv[cu[b]:cu[b + 1], h * dh + 1:(h + 1) * dh] *= 0.1
                qkv[cu[b]:cu[b + 1], D + h * dh] = j / 16.0
    qkv = _store(qkv, dt)
    ref = np.full((T, D), np.nan)
    for b in range(len(lens)):
        s0, s1 = cu[b], cu[b + 1]
        ref[s0:s1] = oracle.attention(qkv[s0:s1, :D], qkv[s0:s0 + kv[b], D:2 * D], qkv[s0:s0 + kv[b], 2 * D:], H)
    out = torch.full((T_cap, D), 3.0, dtype=tdtype(dt), device=cuda())
    ws_bytes = (H * ((T_cap + 127) // 128 + len(lens)) * 16) + 4096
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_attention(to_dev(qkv, dt), out, dt, i32(cu), i32(kv), len(lens), T_cap, H, dh, ws, ws_bytes)
    got = host(out)
    check_close(got[:T], ref, "f32" if dt == "f32" else "bf16", f"attention lens={lens}")
    assert (got[T:] == 3.0).all()


@pytest.mark.parametrize("dt", ["f16", "bf16"])
@pytest.mark.parametrize("scale", [1.0, 2.0])
def test_attention_16bit_varlen(dt, scale):
    lens = [1, 127, 128, 129, 300, 517, 64]
    kv = [1, 127, 128, 129, 260, 517, 40]     # two segments with padded (masked) key tails
    _attention_case(dt, 2, 128, lens, kv, scale, 11)


@pytest.mark.parametrize("dt", ["f16", "bf16"])
def test_attention_growing_max_forces_rescale(dt):
    # logits grow by ~0.1 per key, so the running max rises by ~18 (log2 units)
    # from one 128-key tile to the next: every tile takes the O-rescale branch
    lens = [517, 300]
    _attention_case(dt, 2, 128, lens, lens, 1.0, 15, structured=True)


def test_attention_many_heads():
    _attention_case("f16", 4, 128, [200, 90], [200, 90], 1.0, 12)


@pytest.mark.parametrize("dt", ["f16", "bf16"])
@pytest.mark.parametrize("H", [8, 3])
def test_attention_many_units_per_cta(dt, H):
    # hundreds of work units, more than there are SMs: each persistent CTA
    # takes units in turn, mixing paired and single query tiles (odd tile
    # counts), masked key tails and one-row segments, for an even and an odd
    # head count
    r = _rng(21)
    lens = [int(x) for x in r.integers(1, 400, 48)]
    lens[3], lens[7], lens[11] = 1, 256, 257
    kv = [max(1, L - int(r.integers(0, min(L, 40)))) for L in lens]
    _attention_case(dt, H, 128, lens, kv, 1.0, 22)


def test_attention_workspace_reused_across_schedules():
    # the unit counter lives in the schedule workspace: a second call with
    # another schedule on the same workspace must start from unit 0 again
    H, dh = 4, 128
    D = H * dh
    T_cap = 3000
    ws_bytes = (H * ((T_cap + 127) // 128 + 64) * 16) + 4096
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    for seed, lens in ((31, [900, 40, 700, 1, 300]), (32, [129] * 20), (33, [2999])):
        rng = _rng(seed)
        cu = np.concatenate([[0], np.cumsum(lens)])
        T = int(cu[-1])
        qkv = _store(rng.standard_normal((T_cap, 3 * D)), "f16")
        out = torch.full((T_cap, D), 3.0, dtype=torch.float16, device=cuda())
        S.seer_attention(to_dev(qkv, "f16"), out, "f16", i32(cu), None, len(lens), T_cap, H, dh, ws, ws_bytes)
        ref = np.concatenate([oracle.attention(qkv[a:b, :D], qkv[a:b, D:2 * D], qkv[a:b, 2 * D:3 * D], H)
                              for a, b in zip(cu[:-1], cu[1:])])
        got = host(out)
        check_close(got[:T], ref, "bf16", f"attention reuse lens={lens}")
        assert (got[T:] == 3.0).all()


def test_attention_f32():
    _attention_case("f32", 4, 64, [1, 70, 33, 130], [1, 70, 20, 130], 1.0, 13)


# ------------------------------------------------------------------ SNR scan (S2)
def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)["cases"]


def test_snr_scan_golden_bit_exact():
    for case in _golden("snr_cases.json"):
        N = len(case["counts"])
        c = i32(case["counts"])
        L = torch.full((1,), -7, dtype=torch.int32, device=cuda())
        I = torch.full((1,), -7, dtype=torch.int32, device=cuda())
        p = S.make_params(0.0, case["tau_jump"], case["gamma"], case["window"])
        S.seer_snr_scan(c, 1, N, case["F"], p, L, I)
        assert (int(I.item()), int(L.item())) == (case["i_star"], case["L_star"]), case["name"]


@pytest.mark.parametrize("B,N", [(256, 1024), (3, 20000)])
def test_snr_scan_large_shapes_match_oracle_exactly(B, N):
    # many sequences (one warp each), and a window longer than the shared-memory
    # staging of the counts (the scan then reads them from global memory)
    rng = _rng(50 + N)
    F = 12288
    counts = rng.integers(0, 100, size=(B, N))
    for b in range(B):
        j = int(rng.integers(1, N - 3))
        counts[b, j:] += int(rng.integers(0, 3000))        # a jump below tau_jump * F (369) is no boundary
    counts[0, :] = 0                                       # no jump at all: L* = N
    p = S.make_params(0.0, 0.03, 0.6, 3)
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    I = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_snr_scan(i32(counts.ravel()), B, N, F, p, L, I)
    i_ref, L_ref = oracle.snr_boundaries(counts, F, 0.03, 0.6, 3)
    np.testing.assert_array_equal(I.cpu().numpy(), i_ref)
    np.testing.assert_array_equal(L.cpu().numpy(), L_ref)
    assert L_ref[0] == N and (L_ref[1:] < N).any()


def test_snr_scan_random_matches_oracle_exactly():
    rng = _rng(14)
    B, N, F = 37, 300, 768
    counts = rng.integers(0, 40, size=(B, N))
    for b in range(B):
        j = int(rng.integers(1, N - 3))
        counts[b, j:] = counts[b, j:] + int(rng.integers(0, 200))
    p = S.make_params(0.0, 0.03, 0.6, 3)
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    I = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_snr_scan(i32(counts.ravel()), B, N, F, p, L, I)
    i_ref, L_ref = oracle.snr_boundaries(counts, F, 0.03, 0.6, 3)
    np.testing.assert_array_equal(I.cpu().numpy(), i_ref)
    np.testing.assert_array_equal(L.cpu().numpy(), L_ref)


@pytest.mark.parametrize("window", [1, 2, 4, 5, 7, 10])
def test_snr_scan_window_variants_match_oracle_exactly(window):
    # look-ahead window variants (Sec. 4.5, Table 12): plateaus of random length around the window
    rng = _rng(40 + window)
    B, N, F = 29, 260, 768
    counts = rng.integers(0, 12, size=(B, N))
    for b in range(B):
        j = int(rng.integers(1, N - window))
        run = int(rng.integers(1, 2 * window + 2))
        counts[b, j:j + run] += int(rng.integers(20, 300))
    p = S.make_params(0.0, 0.03, 0.6, window)
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    I = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_snr_scan(i32(counts.ravel()), B, N, F, p, L, I)
    i_ref, L_ref = oracle.snr_boundaries(counts, F, 0.03, 0.6, window)
    np.testing.assert_array_equal(I.cpu().numpy(), i_ref)
    np.testing.assert_array_equal(L.cpu().numpy(), L_ref)


def test_multi_layer_sparsity_tap():
    # counts of three layers' gate/up weights summed (a count out of 3F), then one scan
    from paper_2607_14557_gb300 import driver as D
    wl = synth.tiny_workload(dtype="bf16", seed=240, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4, window=200,
                             boundary=("uniform", 8, 190), n_layers=3)
    lens = synth.lengths(wl)
    x, cu, resp = synth.hidden_full(wl, lens)
    B, N, F = wl.batch, wl.window, wl.d_ff
    ws = [synth.layer_weights(wl, l) for l in range(3)]
    taps = [D.LayerWeights.from_host(w, "bf16") for w in ws]
    path = D.SeerPath(S.make_dims(wl.d, wl.n_heads, wl.head_dim, F), "bf16", B, N, x.shape[0],
                      S.make_params(wl.act_eps))
    path.detect_multi(to_dev(x, "bf16"), i32(resp), taps)
    torch.cuda.synchronize()
    got = path.counts.cpu().numpy().reshape(B, N)
    for b in range(B):
        ref = sum(oracle.sparsity_counts(x[resp[b]:resp[b] + N], w["wg"], w["wu"], wl.act_eps) for w in ws)
        assert np.abs(got[b] - ref).max() <= 0.005 * 3 * F
    i_ref, L_ref = oracle.snr_boundaries(got, 3 * F)
    np.testing.assert_array_equal(path.L_star.cpu().numpy(), L_ref)
    np.testing.assert_array_equal(path.i_star.cpu().numpy(), i_ref)
    np.testing.assert_array_equal(L_ref, lens.boundary + 1)


# ------------------------------------------------------------------ detector end to end (S1 + S2)
@pytest.mark.parametrize("dtype,seed", [("bf16", 1), ("bf16", 2), ("f32", 3)])
def test_detect_boundary_planted(dtype, seed):
    d = 256
    wl = synth.tiny_workload(dtype=dtype, seed=200 + seed, d=d, n_heads=2 if dtype == "bf16" else 4,
                             head_dim=128 if dtype == "bf16" else 64, d_ff=768, batch=5, window=200,
                             boundary=("uniform", 8, 190))
    lens = synth.lengths(wl)
    x, cu, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    B, N, F = wl.batch, wl.window, wl.d_ff
    counts = torch.empty(B * N, dtype=torch.int32, device=cuda())
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    I = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_detect_boundary(to_dev(x, dtype), dtype, x.shape[0], i32(resp), B, N, to_dev(w["wg"], dtype),
                           to_dev(w["wu"], dtype), S.make_dims(d, wl.n_heads, wl.head_dim, F),
                           S.make_params(wl.act_eps), counts, L, I)
    got = counts.cpu().numpy().reshape(B, N)
    for b in range(B):
        ref = oracle.sparsity_counts(x[resp[b]:resp[b] + N], w["wg"], w["wu"], wl.act_eps)
        assert np.abs(got[b] - ref).max() <= 0.005 * F
    np.testing.assert_array_equal(L.cpu().numpy(), lens.boundary + 1)
    np.testing.assert_array_equal(I.cpu().numpy(), lens.boundary)


# ------------------------------------------------------------------ routing + pack (S3 + S4)
def _pack_case(dtype, ctx, L_star, N, d, tau_pad=0.2, seed=0, extra_cap=50, bucket_min=8):
    rng = _rng(seed)
    B = len(ctx)
    full = np.asarray(ctx) + N
    cu_full = np.concatenate([[0], np.cumsum(full)])
    x = synth.round_storage(rng.standard_normal((int(cu_full[-1]), d)), dtype)
    seg, kv, cu = oracle.segment_layout(ctx, L_star, N, tau_pad, bucket_min=bucket_min)
    ref_rows = oracle.pack_rows(x, cu_full, seg)
    T_cap = int(cu[-1]) + extra_cap
    out = torch.full((T_cap, d), 5.0, dtype=tdtype(dtype), device=cuda())
    cu_out = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    kv_out = torch.empty(B, dtype=torch.int32, device=cuda())
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=cuda())
    hctrl = torch.zeros(S.CTRL_WORDS, dtype=torch.int32).pin_memory()
    p = S.make_params(0.0, tau_pad=tau_pad, bucket_min=bucket_min)
    S.seer_pack_ragged(to_dev(x, dtype), dtype, i32(cu_full), i32(ctx), i32(L_star), B, d, N, T_cap, p, out, cu_out,
                       kv_out, meta, hctrl, 9)
    ctrl = torch.zeros(S.CTRL_WORDS, dtype=torch.int32)
    S.seer_poll_ctrl(hctrl, 9, 5_000_000, ctrl)
    torch.cuda.synchronize()
    got = host(out)
    np.testing.assert_array_equal(got[:cu[-1]], ref_rows)
    assert (got[cu[-1]:] == 5.0).all()           # zero work past the packed total
    np.testing.assert_array_equal(cu_out.cpu().numpy(), cu)
    np.testing.assert_array_equal(kv_out.cpu().numpy(), kv)
    m = meta.cpu().numpy()
    c = ctrl.numpy()
    np.testing.assert_array_equal(m, c)
    groups = oracle.route(L_star, N, tau_pad, bucket_min=bucket_min)
    assert c[0] == 9 and c[1] == cu[-1] and c[2] == seg.max() and c[4] == len(groups)
    assert c[5] == sum(1 << p_ for p_ in {g["path"] for g in groups})
    pad_ref = sum(g["bucket"] * len(g["members"]) - sum(L_star[i] for i in g["members"])
                  for g in groups if g["path"] == oracle.PATH_STATIC)
    assert c[6] == pad_ref
    for gi, g in enumerate(groups):
        assert list(c[8 + 4 * gi: 12 + 4 * gi]) == [g["bucket"], len(g["members"]), g["path"],
                                                   int(np.floor(g["rho"] * 1e6))]
    # graph capacity: the smallest m * 2^e >= total with m in 8..15
    cands = sorted(m_ * 2 ** e for m_ in range(8, 16) for e in range(0, 24))
    assert c[3] == next(v for v in cands if v >= max(cu[-1], 1))


def test_pack_route_mixed_paths_bf16():
    ctx = [100, 50, 70, 30, 10, 64, 64]
    L = [120, 128, 110, 125, 300, 5, 16]
    _pack_case("bf16", ctx, L, 1024, 256, seed=1)


def test_pack_route_varlen_and_eager_f32():
    ctx = [33, 17, 80]
    L = [65, 70, 128]
    _pack_case("f32", ctx, L, 128, 64, seed=2)


def test_pack_route_untruncated_is_identity_layout():
    ctx = [40, 41, 42]
    N = 96
    _pack_case("bf16", ctx, [N, N, N], N, 256, seed=3)


@pytest.mark.parametrize("B,tau_pad,bucket_min", [(64, 0.2, 8), (256, 0.2, 8), (256, -1.0, 1), (256, 0.9, 64)])
def test_pack_route_large_batches(B, tau_pad, bucket_min):
    # the routing ablation's batch sizes: every block recomputes the route of all
    # B sequences in shared memory; groups, layout, control word and rows exact
    rng = _rng(40 + B)
    N = 1024
    ctx = list(map(int, rng.integers(0, 3000, B)))
    L = list(map(int, rng.integers(1, N + 1, B)))
    _pack_case("bf16", ctx, L, N, 64, tau_pad=tau_pad, seed=41 + B, bucket_min=bucket_min)


@pytest.mark.parametrize("bucket_min", [1, 16, 64, 1024])
def test_pack_route_bucket_set_variants(bucket_min):
    # the smallest micro-bucket moves the group boundaries (routing ablation)
    ctx = [100, 50, 70, 30, 10, 64, 64, 20]
    L = [120, 128, 110, 125, 300, 5, 16, 3]
    _pack_case("bf16", ctx, L, 1024, 256, seed=30 + bucket_min, bucket_min=bucket_min)
