"""The allocation-free attention entry point gives the same result as the
workspace-taking one.

seer_attention_noalloc exists for callers that cannot allocate device memory
(their memory belongs to another allocator, or allocation is forbidden on
their hot path): it keeps the attention schedule in a fixed array inside the
library instead of a caller-provided workspace.  This file is collected last
so that a failure here does not hide the other GPU tests in a run that stops
at the first failure.
"""
import numpy as np
import pytest
import torch

from tests.helpers import check_close, cuda, host, i32

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


def _case(seed, lens, kv, H=2, dh=128, dt="f16"):
    rng = np.random.default_rng(seed)
    D = H * dh
    cu = np.concatenate([[0], np.cumsum(lens)])
    T = int(cu[-1])
    qkv = torch.from_numpy(rng.standard_normal((T + 19, 3 * D)).astype(np.float32)).to(torch.float16).to(cuda())
    return qkv, i32(cu), i32(kv), T + 19, D


@pytest.mark.parametrize("dt", ["f16", "bf16"])
def test_noalloc_attention_matches_workspace_entry_point(dt):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    tdt = torch.float16 if dt == "f16" else torch.bfloat16
    cases = [(21, [1, 127, 300, 517], [1, 100, 300, 517]), (22, [640, 33, 129], [640, 33, 64])]
    for seed, lens, kv in cases:      # two calls in a row, different shapes: the shared array is reused
        qkv, cu, kvd, T_cap, D = _case(seed, lens, kv)
        qkv = qkv.to(tdt)
        ws_bytes = 2 * (2 * ((T_cap + 127) // 128 + len(lens)) * 16) + 4096
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
        ref = torch.full((T_cap, D), 5.0, dtype=tdt, device=cuda())
        got = torch.full((T_cap, D), 5.0, dtype=tdt, device=cuda())
        S.seer_attention(qkv, ref, dt, cu, kvd, len(lens), T_cap, 2, 128, ws, ws_bytes)
        S.seer_attention_noalloc(qkv, got, dt, cu, kvd, len(lens), T_cap, 2, 128)
        torch.cuda.synchronize()
        check_close(host(got), host(ref), "bf16", f"noalloc vs workspace attention, lens={lens}")
    assert S.seer_check_device() == 0


def test_noalloc_attention_rejects_batches_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    qkv = torch.zeros((8, 3 * 4096), dtype=torch.float16, device=cuda())
    o = torch.zeros((8, 4096), dtype=torch.float16, device=cuda())
    cu = i32([0, 8])
    with pytest.raises(S.SeerError, match="WORKSPACE"):
        S.seer_attention_noalloc(qkv, o, "f16", cu, None, 1, 300_000, 32, 128)


def test_noalloc_attention_at_the_scratch_limit():
    # 5 heads, 13000 one-row segments and T_capacity 13312: 5 * (ceil(13312/128) +
    # 13000) = 65520 work units of room, exactly what the 1 MiB array holds, of
    # which 65000 are used, so the schedule fills the array almost to its end.  A
    # one-row segment attends to its own key only: its output is its value row.
    # One row more of capacity needs 65525 units and is refused.
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    H, dh, B, T_cap = 5, 128, 13000, 13312
    D = H * dh
    rng = np.random.default_rng(23)
    qkv = torch.from_numpy(rng.standard_normal((T_cap, 3 * D)).astype(np.float32)).to(torch.float16).to(cuda())
    cu = i32(np.arange(B + 1))
    got = torch.full((T_cap, D), 5.0, dtype=torch.float16, device=cuda())
    S.seer_attention_noalloc(qkv, got, "f16", cu, None, B, T_cap, H, dh)
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
    v = host(qkv[:B, 2 * D:])
    check_close(host(got[:B]), v, "bf16", "one-row segments: output = value row")
    assert (host(got[B:]) == 5.0).all()
    ws_bytes = (H * ((T_cap + 127) // 128 + B)) * 16 + 4096
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device=cuda())
    ref = torch.full((T_cap, D), 5.0, dtype=torch.float16, device=cuda())
    S.seer_attention(qkv, ref, "f16", cu, None, B, T_cap, H, dh, ws, ws_bytes)
    torch.cuda.synchronize()
    assert torch.equal(got, ref)
    with pytest.raises(S.SeerError, match="WORKSPACE"):
        S.seer_attention_noalloc(qkv, got, "f16", cu, None, B, T_cap + 1, H, dh)


def test_noalloc_attention_matches_oracle():
    # ragged segments with masked key tails, against the fp64 statement of Eqs. 6-7
    import oracle
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    lens, kv = [300, 1, 129, 640], [280, 1, 129, 500]
    qkv, cu, kvd, T_cap, D = _case(24, lens, kv)
    got = torch.full((T_cap, D), 5.0, dtype=torch.float16, device=cuda())
    S.seer_attention_noalloc(qkv, got, "f16", cu, kvd, len(lens), T_cap, 2, 128)
    torch.cuda.synchronize()
    q = host(qkv)
    c = np.concatenate([[0], np.cumsum(lens)])
    ref = np.concatenate([oracle.attention(q[a:b, :D], q[a:a + k, D:2 * D], q[a:a + k, 2 * D:], 2)
                          for a, b, k in zip(c[:-1], c[1:], kv)])
    check_close(host(got)[:c[-1]], ref, "bf16", "noalloc attention vs oracle")
    assert S.seer_check_device() == 0


def test_noalloc_attention_f32_has_no_schedule_limit():
    # fp32 attention runs without a schedule: a batch whose 16-bit schedule would
    # not fit the array (2 * (ceil(40000/128) + 40000) = 80626 units) still runs
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    H, dh, B = 2, 64, 40000
    D = H * dh
    rng = np.random.default_rng(25)
    qkv = torch.from_numpy(rng.standard_normal((B, 3 * D)).astype(np.float32)).to(cuda())
    got = torch.zeros((B, D), dtype=torch.float32, device=cuda())
    S.seer_attention_noalloc(qkv, got, "f32", i32(np.arange(B + 1)), None, B, B, H, dh)
    torch.cuda.synchronize()
    assert S.seer_check_device() == 0
    check_close(host(got), host(qkv[:, 2 * D:]), "f32", "fp32 one-row segments: output = value row")
    q16 = torch.zeros((B, 3 * H * 128), dtype=torch.float16, device=cuda())
    o16 = torch.zeros((B, H * 128), dtype=torch.float16, device=cuda())
    with pytest.raises(S.SeerError, match="WORKSPACE"):      # refused on the host, before any launch
        S.seer_attention_noalloc(q16, o16, "f16", i32(np.arange(B + 1)), None, B, B, H, 128)
