"""GPU parity of the standalone rotary-embedding entry point (seer_rope) against
the oracle's rotation, including positions up to 16k (large angles)."""
import numpy as np
import pytest
import torch

import oracle
from tests.helpers import cuda, host, i32, tdtype

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    assert S.seer_check_device() == 0


def _stored(a, dt):
    return torch.from_numpy(np.asarray(a, dtype=np.float32)).to(tdtype(dt)).float().numpy().astype(np.float64)


@pytest.mark.parametrize("dt,dh", [("f32", 128), ("f32", 64), ("f16", 128), ("bf16", 128)])
def test_rope_matches_oracle(dt, dh):
    H = 2
    seg = np.array([5, 16000, 300])
    cu = np.concatenate([[0], np.cumsum(seg)])
    T = int(cu[-1])
    cap = T + 7
    rng = np.random.default_rng(dh)
    qkv = _stored(rng.standard_normal((cap, 3 * H * dh)), dt)
    dev = torch.from_numpy(qkv.astype(np.float32)).to(tdtype(dt)).to(cuda())
    S.seer_rope(dev, dt, i32(cu), len(seg), cap, H, dh, 1e4)
    torch.cuda.synchronize()
    got = host(dev)
    pos = np.concatenate([np.arange(n) for n in seg])
    ref = qkv[:T].copy()
    ref[:, :2 * H * dh] = oracle.rope(qkv[:T, :2 * H * dh], pos, 2 * H, 1e4)
    rel = {"f32": 2e-6, "f16": 2 ** -10, "bf16": 2 ** -7}[dt]
    err = np.abs(got[:T] - ref)
    bound = rel * np.abs(ref) + (1e-5 if dt == "f32" else 1e-3)
    assert (err <= bound).all(), float((err - bound).max())
    np.testing.assert_array_equal(got[:T, 2 * H * dh:], qkv[:T, 2 * H * dh:])     # v untouched
    np.testing.assert_array_equal(got[T:], qkv[T:])                               # rows past the total untouched


def test_rope_rejects_bad_arguments():
    x = torch.zeros((8, 3 * 128), dtype=torch.float32, device=cuda())
    cu = i32([0, 8])
    with pytest.raises(RuntimeError):
        S.seer_rope(x, "f32", cu, 1, 8, 1, 128, 0.0)
    with pytest.raises(RuntimeError):
        S.seer_rope(x, "f32", cu, 1, 8, 1, 256, 1e4)
