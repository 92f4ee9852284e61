"""The C-ABI library builds, loads without a GPU and exports every declared symbol."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "seer.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(seer_[a-z_0-9]+)\s*\(", src)))


@pytest.fixture(scope="module")
def libseer():
    from paper_2607_14557_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    names = _declared()
    for required in ("seer_detect_boundary", "seer_pack_ragged", "seer_layer_forward", "seer_poll_ctrl",
                     "seer_layer_workspace_size", "seer_last_error", "seer_check_device"):
        assert required in names


def test_every_declared_symbol_is_exported(libseer):
    missing = [n for n in _declared() if not hasattr(libseer, n)]
    assert not missing, missing


def test_host_side_argument_checks_need_no_gpu(libseer):
    from paper_2607_14557_gb300 import seer as S
    L = S.lib()
    dims = S.make_dims(4096, 32, 128, 12288)
    bad = S.make_dims(4096, 32, 100, 12288)
    out = ctypes.c_size_t(0)
    assert L.seer_layer_workspace_size(ctypes.byref(dims), S.SEER_BF16, 1000, 4, ctypes.byref(out)) == 0
    assert out.value > 1000 * 4096 * 2 * 6
    assert L.seer_layer_workspace_size(ctypes.byref(bad), S.SEER_BF16, 1000, 4, ctypes.byref(out)) == 1
    rope = S.make_dims(4096, 32, 128, 12288, rope_theta=10000.0)
    assert L.seer_layer_workspace_size(ctypes.byref(rope), S.SEER_BF16, 1000, 4, ctypes.byref(out)) == 0
    neg = S.make_dims(4096, 32, 128, 12288, rope_theta=-1.0)
    assert L.seer_layer_workspace_size(ctypes.byref(neg), S.SEER_BF16, 1000, 4, ctypes.byref(out)) == 1
    assert b"rope" in L.seer_last_error()
    nan = S.make_dims(4096, 32, 128, 12288, rope_theta=float("nan"))
    assert L.seer_layer_workspace_size(ctypes.byref(nan), S.SEER_BF16, 1000, 4, ctypes.byref(out)) == 1


def test_poll_ctrl_times_out_on_host_flag_never_set(libseer):
    from paper_2607_14557_gb300 import seer as S
    buf = (ctypes.c_int32 * S.CTRL_WORDS)()
    st = S.lib().seer_poll_ctrl(ctypes.addressof(buf), 7, 2000, None)
    assert st == 5   # SEER_ERR_TIMEOUT
    buf[0] = 7
    buf[1] = 1234
    copy = (ctypes.c_int32 * S.CTRL_WORDS)()
    assert S.lib().seer_poll_ctrl(ctypes.addressof(buf), 7, 2000, ctypes.addressof(copy)) == 0
    assert copy[1] == 1234
