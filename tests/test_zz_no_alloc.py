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
