"""The C-ABI boundary: the library builds, loads and exports every symbol include/gas.h
declares; host-side helpers and argument checks behave as documented."""

import ctypes
import math

import numpy as np
import pytest
import torch

import paper_2602_18851_gb300 as gas
from oracle import calib


@pytest.fixture(scope="module")
def lib():
    gas.build()
    return gas.load()


def test_exports_every_declared_symbol(lib):
    names = gas.exported_names()
    assert len(names) >= 15
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_header_is_plain_c():
    """No torch or C++ types cross the boundary."""
    src = open(gas.HEADER).read()
    for bad in ("torch", "at::", "std::", "Tensor", "template"):
        assert bad not in src
    assert 'extern "C"' in src


@pytest.mark.parametrize("dh,d,n", [(64, 1600, 1200), (128, 4096, 1024), (128, 5120, 1600),
                                    (128, 8192, 5120), (64, 768, 144)])
def test_host_calibration_helpers_match_oracle(lib, dh, d, n):
    g = gas.gamma_min(dh, n, 1024, 1e-6)
    assert g == pytest.approx(calib.gamma_min(dh, n, 1024, 1e-6), rel=1e-12)
    a = gas.alpha_min(g, d, dh, n, 1024, 1e-6)
    assert a == pytest.approx(calib.alpha_min(g, d, dh, n, 1024, 1e-6), rel=1e-12)


def test_host_helpers_invalid_inputs(lib):
    assert math.isnan(gas.gamma_min(0, 10, 1024, 1e-6))
    assert math.isnan(gas.gamma_min(64, 10, 1024, -1.0))
    assert gas.gamma_min(64, 1, 1, 10.0) == 1.0
    assert math.isnan(gas.alpha_min(0.5, 256, 64, 1, 1024, 1e-6))


def test_status_strings(lib):
    for code, name in [(0, b"GAS_OK"), (1, b"GAS_ERR_INVALID_ARG"), (2, b"GAS_ERR_UNSUPPORTED"),
                       (3, b"GAS_ERR_CUDA"), (4, b"GAS_ERR_ALLOC"), (5, b"GAS_ERR_DEVICE_TIMEOUT")]:
        assert lib.gas_status_string(code) == name


def test_create_rejects_bad_shapes_without_touching_the_device(lib):
    h = ctypes.c_void_p()
    for args, code in [((0, 256, 4, 4, 64), 1), ((2, 256, 4, 3, 64), 2), ((2, 250, 4, 4, 64), 2),
                       ((2, 256, 4, 4, 72), 2), ((2, 256, 4, 4, 32), 2), ((600, 256, 4, 4, 64), 2),
                       ((2, 256, 130, 2, 128), 2)]:
        st = lib.gas_create(*args, ctypes.byref(h))
        assert st == code, (args, st, lib.gas_last_error(None))
        assert h.value is None
    assert lib.gas_create(2, 256, 4, 4, 64, None) == 1


def test_null_handle_calls(lib):
    assert lib.gas_destroy(None) == 0
    assert lib.gas_workspace_bytes(None) == 0
    assert lib.gas_set_method(None, 0) == 1
    assert lib.gas_spectral_norms(None, None, None, 1, None, None, None, None) == 1


@pytest.mark.skipif(torch.cuda.is_available(), reason="CPU-only behaviour")
def test_create_without_gpu_fails_cleanly(lib):
    h = ctypes.c_void_p()
    st = lib.gas_create(2, 256, 4, 4, 64, ctypes.byref(h))
    assert st == 3 and h.value is None
    assert b"device" in lib.gas_last_error(None).lower() or len(lib.gas_last_error(None)) > 0


# ----------------------------------------------------------------------------------
# GPU: argument checks on a live handle
# ----------------------------------------------------------------------------------
@pytest.mark.gpu
def test_gpu_argument_errors(lib):
    L, d, nq, nkv, dh = 2, 256, 4, 2, 64
    hd = gas.Handle(L, d, nq, nkv, dh)
    wq = [torch.zeros(nq * dh, d, device="cuda", dtype=torch.bfloat16) for _ in range(L)]
    wk = [torch.zeros(nkv * dh, d, device="cuda", dtype=torch.bfloat16) for _ in range(L)]
    v = torch.randn(L, nq, d, device="cuda")
    sig = torch.empty(L, nq, device="cuda")
    qa = (ctypes.c_void_p * L)(*[t.data_ptr() for t in wq])
    ka = (ctypes.c_void_p * L)(*[t.data_ptr() for t in wk])
    h = hd._h
    assert lib.gas_spectral_norms(h, qa, ka, 0, v.data_ptr(), None, sig.data_ptr(), None) == 1
    assert lib.gas_spectral_norms(h, None, ka, 3, v.data_ptr(), None, sig.data_ptr(), None) == 1
    assert lib.gas_spectral_norms(h, qa, ka, 3, None, None, sig.data_ptr(), None) == 1
    assert lib.gas_spectral_norms(h, qa, ka, 3, v.data_ptr() + 4, None, sig.data_ptr(), None) == 1
    bad = (ctypes.c_void_p * L)(wq[0].data_ptr() + 2, wq[1].data_ptr())
    assert lib.gas_spectral_norms(h, bad, ka, 3, v.data_ptr(), None, sig.data_ptr(), None) == 1
    nul = (ctypes.c_void_p * L)(wq[0].data_ptr(), None)
    assert lib.gas_spectral_norms(h, nul, ka, 3, v.data_ptr(), None, sig.data_ptr(), None) == 1
    s = torch.empty(L, device="cuda")
    assert lib.gas_scales(h, sig.data_ptr(), 0.5, 1e-6, 448.0, s.data_ptr(), None) == 1
    assert lib.gas_scales(h, sig.data_ptr(), 1.0, 1e-6, 448.0, s.data_ptr(), None) == 1
    assert lib.gas_scales(h, sig.data_ptr(), 0.0, 0.0, 448.0, s.data_ptr(), None) == 1
    assert lib.gas_scales(h, sig.data_ptr(), 0.0, 1e-6, -1.0, s.data_ptr(), None) == 1
    assert lib.gas_set_calibration(h, 0, 0.8, 0.0) == 1
    assert lib.gas_set_calibration(h, 1024, 1.5, 0.0) == 1
    assert lib.gas_set_method(h, 7) == 1
    assert b"method" in lib.gas_last_error(h)
    # a valid call still works after the rejected ones
    assert lib.gas_spectral_norms(h, qa, ka, 3, v.data_ptr(), None, sig.data_ptr(), None) == 0
    torch.cuda.synchronize()
    assert np.all(sig.cpu().numpy() == 0.0)  # zero weights: sigma = 0 exactly
    hd.close()


@pytest.mark.gpu
def test_gpu_workspace_and_resolve(lib):
    with gas.Handle(80, 8192, 64, 8, 128) as h:
        assert h.workspace_bytes > 0
        assert h.workspace_bytes < 2 * 2 ** 30
        g, a = h.resolve_calibration()
        assert g == pytest.approx(calib.gamma_min(128, 5120, 1024, 1e-6), rel=1e-12)
        assert a == pytest.approx(calib.alpha_min(g, 8192, 128, 5120, 1024, 1e-6), rel=1e-12)
        h.set_calibration(alpha_override=0.02)
        assert h.resolve_calibration()[1] == 0.02


def test_graft_entry_build():
    """__graft_entry__.build() compiles the library (sm_103a) and the oracle and imports."""
    import importlib
    import sys
    import os
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    ge = importlib.import_module("__graft_entry__")
    ge.build()
    assert os.path.exists(gas.LIB_PATH)
