"""Failure detection on the GPU without a fault: a pipeline wait that can never
complete gives up after its limit, the timeout code reaches the host through
the device error word, and the context stays usable."""
import time

import numpy as np
import pytest
import torch

from tests.helpers import check_close, cuda, host, to_dev

pytestmark = pytest.mark.gpu

S = pytest.importorskip("paper_2607_14557_gb300.seer")


@pytest.fixture(autouse=True)
def _device_clean():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    assert S.seer_check_device() == 0
    yield
    assert S.seer_check_device() == 0


def test_bounded_wait_times_out_and_reports():
    t0 = time.perf_counter()
    S.seer_selftest_wait_timeout(200_000)          # 0.2 s limit
    code = S.seer_check_device()                    # synchronises, reads and clears the error word
    dt = time.perf_counter() - t0
    assert code == 3                                # kErrTimeout
    assert 0.15 < dt < 10.0
    # the context survives: a GEMM afterwards runs and is correct
    rng = np.random.default_rng(0)
    a = rng.standard_normal((300, 256)).astype(np.float32)
    w = (0.05 * rng.standard_normal((256, 256))).astype(np.float32)
    a16 = torch.from_numpy(a).to(torch.float16).float().numpy()
    w16 = torch.from_numpy(w).to(torch.float16).float().numpy()
    c = torch.empty((300, 256), dtype=torch.float16, device=cuda())
    S.seer_linear(to_dev(a16, "f16"), to_dev(w16, "f16"), "f16", None, "f16", c, "f16", 300, None, 256, 256)
    check_close(host(c), a16.astype(np.float64) @ w16.astype(np.float64).T, "bf16", "GEMM after a timeout")


def test_selftest_rejects_bad_limits():
    with pytest.raises(RuntimeError):
        S.seer_selftest_wait_timeout(0)
