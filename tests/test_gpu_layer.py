"""GPU parity of the full path: detect (S1-S2) -> route + pack (S3-S4) ->
truncated layer forward (S5-S11), through the C ABI, against the oracle."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.helpers import check_close, check_counts, cuda, host, i32, layer_weight_tensors, to_dev, weights_struct

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    assert S.seer_check_device() == 0


def run_path(wl, lens=None, tau_pad=0.2, extra_cap=64, data=None, rope_theta=0.0):
    """Detect, pack and run one layer on the GPU; return everything needed to check it."""
    dt = wl.dtype
    lens = lens or synth.lengths(wl)
    x, cu_full, resp = data if data is not None else synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    B, N, F, d = wl.batch, wl.window, wl.d_ff, wl.d
    dims = S.make_dims(d, wl.n_heads, wl.head_dim, F, rope_theta=rope_theta)
    params = S.make_params(wl.act_eps, tau_pad=tau_pad)
    W, WL = layer_weight_tensors(wl, w)
    xd = to_dev(x, dt)
    counts = torch.empty(B * N, dtype=torch.int32, device=cuda())
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_detect_boundary(xd, dt, x.shape[0], i32(resp), B, N, W["w_gate"], W["w_up"], dims, params, counts, L)
    T_cap = int(cu_full[-1]) + extra_cap
    xp = torch.full((T_cap, d), 0.0, dtype=xd.dtype, device=cuda())
    cu = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    kv = torch.empty(B, dtype=torch.int32, device=cuda())
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=cuda())
    S.seer_pack_ragged(xd, dt, i32(cu_full), i32(lens.ctx), L, B, d, N, T_cap, params, xp, cu, kv, meta)
    y = torch.full((T_cap, d), 9.0, dtype=xd.dtype, device=cuda())
    ws_bytes = S.seer_layer_workspace_size(dims, dt, T_cap, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_layer_forward(weights_struct(WL), dims, dt, xp, y, cu, kv, B, T_cap, None, 0, 0.0, None, ws, ws_bytes)
    torch.cuda.synchronize()
    return dict(x=x, cu_full=cu_full, resp=resp, w=w, lens=lens, counts=counts.cpu().numpy().reshape(B, N),
                L=L.cpu().numpy(), cu=cu.cpu().numpy(), kv=kv.cpu().numpy(), xp=host(xp), y=host(y), T_cap=T_cap,
                rope_theta=rope_theta)


def _check_counts(wl, r):
    """Every token of every window: the detector's near-zero counts against the
    oracle's (Sec. 3.2), within 0.5% of F."""
    x, resp, w = r["x"], r["resp"], r["w"]
    worst = 0
    for b in range(wl.batch):
        ref = oracle.sparsity_counts(x[resp[b]:resp[b] + wl.window], w["wg"], w["wu"], wl.act_eps)
        worst = max(worst, check_counts(r["counts"][b], ref, wl.d_ff, f"{wl.name} window {b}"))
    return worst


def _check_path(wl, r):
    lens = r["lens"]
    _check_counts(wl, r)
    np.testing.assert_array_equal(r["L"], lens.boundary + 1)           # planted boundary, bit exact
    seg, kv, cu = oracle.segment_layout(lens.ctx, r["L"], wl.window)
    np.testing.assert_array_equal(r["cu"], cu)
    np.testing.assert_array_equal(r["kv"], kv)
    T = int(cu[-1])
    np.testing.assert_array_equal(r["xp"][:T], oracle.pack_rows(r["x"], r["cu_full"], seg))
    ref = oracle.layer_forward_packed(r["xp"][:T], cu, r["w"], wl.n_heads, kv_len=kv, rope_theta=r["rope_theta"])
    err = check_close(r["y"][:T], ref, wl.dtype, wl.name)
    assert (r["y"][T:] == 9.0).all()                                    # zero work past truncation
    return err


@pytest.mark.parametrize("seed", [0, 1])
def test_tiny_bf16_path(seed):
    wl = synth.tiny_workload(dtype="bf16", seed=300 + seed, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4,
                             window=200, boundary=("uniform", 8, 190), visual=("mult", 96, 1, 3))
    _check_path(wl, run_path(wl))


def test_tiny_bf16_static_route_pads_and_masks():
    # lengths concentrated in one bucket -> static path (padded rows are masked keys)
    wl = synth.tiny_workload(dtype="bf16", seed=310, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4,
                             window=200, boundary=("uniform", 120, 127))
    r = run_path(wl)
    groups = oracle.route(r["L"], wl.window)
    assert any(g["path"] == oracle.PATH_STATIC for g in groups)
    _check_path(wl, r)


def test_workload0_f32_path():
    wl = synth.workload(0)
    _check_path(wl, run_path(wl))


@pytest.mark.parametrize("rope_theta", [0.0, 10000.0])
def test_workload1_bf16_path(rope_theta):
    # 842 packed rows: 7 m-tiles with a partial last tile, fewer GEMM tiles than
    # SMs for the O and down projections (112 tiles); the QKV projection runs
    # through the rotary epilogue when rope_theta > 0.  All 256 counts of the
    # window are compared with the oracle.
    wl = synth.workload(1)
    _check_path(wl, run_path(wl, rope_theta=rope_theta))


def test_batch_permutation_is_bit_exact():
    wl = synth.tiny_workload(dtype="bf16", seed=320, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4,
                             window=160, boundary=("uniform", 8, 150))
    lens = synth.lengths(wl)
    r1 = run_path(wl, lens)
    perm = np.array([2, 0, 3, 1])
    x, cu_full = r1["x"], r1["cu_full"]
    seqs = [x[cu_full[i]:cu_full[i + 1]] for i in range(wl.batch)]
    lens_p = synth.with_lengths(wl, lens, visual=lens.visual[perm], prompt=lens.prompt[perm],
                                boundary=lens.boundary[perm])
    cuf = np.concatenate([[0], np.cumsum(lens_p.full)]).astype(np.int32)
    data = (np.concatenate([seqs[i] for i in perm]), cuf, (cuf[:-1] + lens_p.ctx).astype(np.int32))
    r2 = run_path(wl, lens_p, data=data)
    for j, i in enumerate(perm):
        a = r1["y"][r1["cu"][i]:r1["cu"][i + 1]]
        b = r2["y"][r2["cu"][j]:r2["cu"][j + 1]]
        np.testing.assert_array_equal(a, b)


def test_launch_overlap_gives_identical_results():
    # programmatic dependent launch only changes when blocks are placed: every
    # kernel waits for its predecessors at entry, so on and off agree bit for bit
    wl = synth.tiny_workload(dtype="bf16", seed=325, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4,
                             window=200, boundary=("uniform", 8, 190), visual=("mult", 96, 1, 3))
    lens = synth.lengths(wl)
    assert S.seer_set_launch_overlap(True) is True                      # on by default
    try:
        r_on = run_path(wl, lens)
        assert S.seer_set_launch_overlap(False) is True
        r_off = run_path(wl, lens)
        assert S.seer_set_launch_overlap(True) is False
    finally:
        S.seer_set_launch_overlap(True)
    for k in ("counts", "L", "cu", "kv", "xp", "y"):
        np.testing.assert_array_equal(r_on[k], r_off[k], err_msg=k)
    _check_path(wl, r_on)


def test_layer_count_hook_on_full_window():
    # step-0 style: full (untruncated) window, counts fused into the gate/up epilogue
    wl = synth.tiny_workload(dtype="bf16", seed=330, d=256, n_heads=2, head_dim=128, d_ff=768, batch=3, window=160,
                             boundary=("uniform", 8, 150))
    lens = synth.lengths(wl)
    x, cu_full, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    B, N, F, d = wl.batch, wl.window, wl.d_ff, wl.d
    dims = S.make_dims(d, wl.n_heads, wl.head_dim, F)
    W, WL = layer_weight_tensors(wl, w)
    T = x.shape[0]
    y = torch.empty((T, d), dtype=torch.bfloat16, device=cuda())
    counts = torch.full((B * N,), -1, dtype=torch.int32, device=cuda())
    ws_bytes = S.seer_layer_workspace_size(dims, "bf16", T, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_layer_forward(weights_struct(WL), dims, "bf16", to_dev(x, "bf16"), y, i32(cu_full), None, B, T, i32(resp),
                         N, 0.05, counts, ws, ws_bytes)
    got = counts.cpu().numpy().reshape(B, N)
    yh = host(y)
    for b in range(B):
        seg = x[cu_full[b]:cu_full[b + 1]]
        rows = np.arange(resp[b] - cu_full[b], resp[b] - cu_full[b] + N)
        parts = oracle.layer_forward_segment(seg, w, wl.n_heads, count_rows=rows, act_eps=0.05, return_parts=True)
        check_counts(got[b], parts["counts"], F, f"count hook, window {b}")
        check_close(yh[cu_full[b]:cu_full[b + 1]], parts["y"], "bf16", "full window layer")


def test_naive_pad_comparator_matches_truncated_rows():
    # naive-pad comparator (Eq. 3 batch-max padding): every sequence keeps ctx_b + max L* rows,
    # the padding is masked as keys, so the valid rows equal the truncated path's rows bit for bit
    from paper_2607_14557_gb300 import driver as D
    wl = synth.tiny_workload(dtype="bf16", seed=340, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4, window=160,
                             boundary=("uniform", 8, 150))
    lens = synth.lengths(wl)
    x, cu_full, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    B, N, d = wl.batch, wl.window, wl.d
    dims = S.make_dims(d, wl.n_heads, wl.head_dim, wl.d_ff)
    W = D.LayerWeights.from_host(w, "bf16")
    path = D.SeerPath(dims, "bf16", B, N, x.shape[0], S.make_params(wl.act_eps))
    xd, cuf, ctx = to_dev(x, "bf16"), i32(cu_full), i32(lens.ctx)
    path.step(xd, cuf, i32(resp), ctx, W)
    torch.cuda.synchronize()
    L = path.L_star.cpu().numpy()
    np.testing.assert_array_equal(L, lens.boundary + 1)
    xn, cun, kvn, T = path.naive_pad_inputs(xd, cuf, ctx)
    yn = torch.full((T, d), 9.0, dtype=torch.bfloat16, device=cuda())
    path.layer(W, x=xn, y=yn, cu=cun, kv=kvn, T_cap=T)
    torch.cuda.synchronize()
    seg = lens.ctx + L.max()
    cun_h = cun.cpu().numpy()
    np.testing.assert_array_equal(cun_h, np.concatenate([[0], np.cumsum(seg)]))
    np.testing.assert_array_equal(kvn.cpu().numpy(), lens.ctx + L)
    np.testing.assert_array_equal(host(xn), oracle.pack_rows(x, cu_full, seg))
    cu_t, yt, ynh = path.cu.cpu().numpy(), host(path.y), host(yn)
    for b in range(B):
        n = int(lens.ctx[b] + L[b])
        np.testing.assert_array_equal(ynh[cun_h[b]:cun_h[b] + n], yt[cu_t[b]:cu_t[b] + n])
    assert np.isfinite(ynh).all()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_path_with_rotary_embedding(dtype):
    # optional rotary q/k embedding: fused into the QKV epilogue (16-bit) or a separate kernel (fp32)
    if dtype == "bf16":
        wl = synth.tiny_workload(dtype="bf16", seed=350, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4,
                                 window=200, boundary=("uniform", 8, 190), visual=("mult", 96, 1, 3))
    else:
        wl = synth.workload(0)
    r = run_path(wl, rope_theta=1e4)
    _check_path(wl, r)


def test_rotary_layer_at_long_positions():
    # one 9k-row segment: rotation angles up to ~9000 rad in the fused epilogue (sampled query rows)
    wl = synth.tiny_workload(dtype="bf16", seed=360, d=256, n_heads=2, head_dim=128, d_ff=768, batch=2,
                             window=128, visual=("mult", 4000, 2, 2), prompt=("uniform", 900, 990),
                             boundary=("uniform", 20, 100))
    lens = synth.lengths(wl)
    x, cu_full, _ = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    d, F, B = wl.d, wl.d_ff, wl.batch
    dims = S.make_dims(d, wl.n_heads, wl.head_dim, F, rope_theta=1e4)
    W, WL = layer_weight_tensors(wl, w)
    T = x.shape[0]
    y = torch.empty((T, d), dtype=torch.bfloat16, device=cuda())
    ws_bytes = S.seer_layer_workspace_size(dims, "bf16", T, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_layer_forward(weights_struct(WL), dims, "bf16", to_dev(x, "bf16"), y, i32(cu_full), None, B, T, None, 0,
                         0.0, None, ws, ws_bytes)
    torch.cuda.synchronize()
    yh = host(y)
    rng = np.random.default_rng(3)
    for b in range(B):
        L = int(cu_full[b + 1] - cu_full[b])
        assert L > 8000
        rows = sorted({0, 1, L - 1, L - 2, *map(int, rng.integers(L // 2, L, 14))})
        ref = oracle.layer_forward_rows(x[cu_full[b]:cu_full[b + 1]], w, wl.n_heads, rows, rope_theta=1e4)
        check_close(yh[cu_full[b] + np.asarray(rows)], ref, "bf16", f"rotary layer segment {b}")


def test_run_from_host_pipelined_matches_device_step():
    # the end-to-end call (pinned host input, double-buffered copies overlapping compute)
    # returns exactly what a device-resident step computes
    from paper_2607_14557_gb300 import driver as D
    wl = synth.tiny_workload(dtype="bf16", seed=390, d=256, n_heads=2, head_dim=128, d_ff=768, batch=3, window=160,
                             boundary=("uniform", 8, 150))
    lens = synth.lengths(wl)
    x, cu_full, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    dims = S.make_dims(wl.d, wl.n_heads, wl.head_dim, wl.d_ff)
    W = D.LayerWeights.from_host(w, "bf16")
    path = D.SeerPath(dims, "bf16", wl.batch, wl.window, x.shape[0], S.make_params(wl.act_eps))
    cuf, rs, ctx = i32(cu_full), i32(resp), i32(lens.ctx)
    xd = to_dev(x, "bf16")
    path.step(xd, cuf, rs, ctx, W)
    torch.cuda.synchronize()
    T = int(path.cu[-1].item())
    ref = host(path.y)[:T]
    x_host = xd.cpu().pin_memory()
    y_host = torch.full((x.shape[0], wl.d), 7.0, dtype=torch.bfloat16).pin_memory()
    L_host = torch.zeros(wl.batch, dtype=torch.int32).pin_memory()
    r = path.run_from_host(x_host, cuf, rs, ctx, W, y_host, L_host, 3)
    assert r["total"] == T
    np.testing.assert_array_equal(y_host.float().numpy()[:T], ref)
    assert (y_host.float().numpy()[T:] == 7.0).all()
    np.testing.assert_array_equal(L_host.numpy(), lens.boundary + 1)


def test_tiny_f16_model_path():
    # an f16 model (inputs, weights and outputs f16) through detect -> pack -> layer
    wl = synth.tiny_workload(dtype="bf16", seed=395, d=256, n_heads=2, head_dim=128, d_ff=768, batch=3, window=160,
                             boundary=("uniform", 8, 150))
    lens = synth.lengths(wl)
    xb, cu_full, resp = synth.hidden_full(wl, lens)
    wb = synth.layer_weights(wl, 0)
    f16 = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.float16)
    x = f16(xb).double().numpy()
    w = {k: f16(v).double().numpy() for k, v in wb.items()}
    B, N, F, d = wl.batch, wl.window, wl.d_ff, wl.d
    dims = S.make_dims(d, wl.n_heads, wl.head_dim, F)
    params = S.make_params(wl.act_eps)
    dev = lambda a: f16(a).to(cuda())
    Wt = {"w_qkv": dev(np.concatenate([w["wq"], w["wk"], w["wv"]])), "w_o": dev(w["wo"]), "w_gate": dev(w["wg"]),
          "w_up": dev(w["wu"]), "w_down": dev(w["wd"]), "g_attn": dev(w["g_attn"]), "g_mlp": dev(w["g_mlp"])}
    xd = dev(x)
    counts = torch.empty(B * N, dtype=torch.int32, device=cuda())
    L = torch.empty(B, dtype=torch.int32, device=cuda())
    S.seer_detect_boundary(xd, "f16", x.shape[0], i32(resp), B, N, Wt["w_gate"], Wt["w_up"], dims, params, counts, L)
    T_cap = x.shape[0]
    xp = torch.zeros((T_cap, d), dtype=torch.float16, device=cuda())
    cu = torch.empty(B + 1, dtype=torch.int32, device=cuda())
    kv = torch.empty(B, dtype=torch.int32, device=cuda())
    meta = torch.empty(S.CTRL_WORDS, dtype=torch.int32, device=cuda())
    S.seer_pack_ragged(xd, "f16", i32(cu_full), i32(lens.ctx), L, B, d, N, T_cap, params, xp, cu, kv, meta)
    y = torch.full((T_cap, d), 9.0, dtype=torch.float16, device=cuda())
    ws_bytes = S.seer_layer_workspace_size(dims, "f16", T_cap, B)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    S.seer_layer_forward(weights_struct(Wt), dims, "f16", xp, y, cu, kv, B, T_cap, None, 0, 0.0, None, ws, ws_bytes)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(L.cpu().numpy(), lens.boundary + 1)
    seg, kv_ref, cu_ref = oracle.segment_layout(lens.ctx, L.cpu().numpy(), N)
    np.testing.assert_array_equal(cu.cpu().numpy(), cu_ref)
    T = int(cu_ref[-1])
    np.testing.assert_array_equal(host(xp)[:T], oracle.pack_rows(x, cu_full, seg))
    ref = oracle.layer_forward_packed(host(xp)[:T], cu_ref, w, wl.n_heads, kv_len=kv_ref)
    check_close(host(y)[:T], ref, "bf16", "f16 model layer")
    assert (host(y)[T:] == 9.0).all()


def test_varlen_only_inputs_repack_without_static_padding():
    # the bench prices the static path's padding against this layout: the same batch
    # re-packed with tau_pad < 0, every segment exactly ctx + L* rows (Sec. 3.4-3.5)
    from paper_2607_14557_gb300 import driver as D
    wl = synth.tiny_workload(dtype="bf16", seed=345, d=256, n_heads=2, head_dim=128, d_ff=768, batch=4, window=200,
                             boundary=("uniform", 120, 127))
    lens = synth.lengths(wl)
    x, cu_full, resp = synth.hidden_full(wl, lens)
    w = synth.layer_weights(wl, 0)
    dims = S.make_dims(wl.d, wl.n_heads, wl.head_dim, wl.d_ff)
    W = D.LayerWeights.from_host(w, "bf16")
    path = D.SeerPath(dims, "bf16", wl.batch, wl.window, x.shape[0], S.make_params(wl.act_eps))
    xd, cuf, ctx = to_dev(x, "bf16"), i32(cu_full), i32(lens.ctx)
    path.step(xd, cuf, i32(resp), ctx, W)
    route = path.route()
    L = path.L_star.cpu().numpy()
    assert route["pad_rows"] > 0                    # the routed layout pads a static group
    xv, cuv, kvv, T_cap = path.varlen_only_inputs(xd, cuf, ctx)
    torch.cuda.synchronize()
    seg, kv, cu = oracle.segment_layout(lens.ctx, L, wl.window, -1.0)
    np.testing.assert_array_equal(seg, lens.ctx + L)
    np.testing.assert_array_equal(cuv.cpu().numpy(), cu)
    np.testing.assert_array_equal(kvv.cpu().numpy(), kv)
    T = int(cu[-1])
    np.testing.assert_array_equal(host(xv)[:T], oracle.pack_rows(x, cu_full, seg))
    y = torch.full((T_cap, wl.d), 9.0, dtype=torch.bfloat16, device=cuda())
    path.layer(W, x=xv, y=y, cu=cuv, kv=kvv, T_cap=T_cap)
    torch.cuda.synchronize()
    ref = oracle.layer_forward_packed(host(xv)[:T], cu, w, wl.n_heads, kv_len=kv)
    check_close(host(y)[:T], ref, "bf16", "varlen-only layer")
