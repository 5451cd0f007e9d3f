"""gas_spectral_norms_static: the allocation-free entry point for callers that cannot
allocate device memory (a host framework owns all of HBM, cudaMalloc's device
synchronisation is not allowed on the caller's path, or there is nowhere to keep a
handle).  Its results must match the handle-based gas_spectral_norms on two calls in
a row, and the calls must not change the device's free memory.

Collected last on purpose (file name), and independent of every other test."""

import ctypes

import pytest
import torch

import paper_2602_18851_gb300 as gas
from synth import get_workload
from tests.parity_utils import SIGMA_RTOL, V_ATOL, assert_sigma_close, assert_v_close, gpu_inputs

pytestmark = pytest.mark.gpu


def _handle_reference(wl, wq, wk, v_in, iters):
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method("stream")
        sigma, v_out = h.spectral_norms(wq, wk, iters, v_in)
        torch.cuda.synchronize()
        return sigma.double().cpu().numpy(), v_out.cpu().numpy()


def _static_call(lib, wl, wq, wk, v_in, sigma, v_out, iters):
    qa = (ctypes.c_void_p * wl.layers)(*[t.data_ptr() for t in wq])
    ka = (ctypes.c_void_p * wl.layers)(*[t.data_ptr() for t in wk])
    st = lib.gas_spectral_norms_static(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h, qa, ka, iters,
                                       v_in.data_ptr(), v_out.data_ptr(), sigma.data_ptr(),
                                       torch.cuda.current_stream().cuda_stream)
    return st


def test_static_entry_point_matches_handle_path_twice():
    gas.build()
    lib = gas.load()
    cases = []
    for name in ("tiny-gqa128", "gpt2-small"):
        wl = get_workload(name)
        wq, wk, v_in, _ = gpu_inputs(wl)
        ref_sigma, ref_v = _handle_reference(wl, wq, wk, v_in, wl.iters)
        sigma = torch.full((wl.layers, wl.n_q), float("nan"), device="cuda")
        v_out = torch.full_like(v_in, float("nan"))
        cases.append((wl, wq, wk, v_in, sigma, v_out, ref_sigma, ref_v))
    torch.cuda.synchronize()
    for i, (wl, wq, wk, v_in, sigma, v_out, ref_sigma, ref_v) in enumerate(cases):
        free_before = torch.cuda.mem_get_info()[0]
        st = _static_call(lib, wl, wq, wk, v_in, sigma, v_out, wl.iters)
        assert st == gas.GAS_OK, lib.gas_last_error(None)
        torch.cuda.synchronize()
        if i > 0:  # the first call may load the library's device image; later calls allocate nothing
            assert torch.cuda.mem_get_info()[0] == free_before
        assert_sigma_close(sigma.double().cpu().numpy().ravel(), ref_sigma.ravel(), rtol=SIGMA_RTOL)
        assert_v_close(v_out.cpu().numpy(), ref_v, atol=V_ATOL)


def test_static_entry_point_rejects_oversized_shapes():
    """A shape whose scratch exceeds GAS_STATIC_SCRATCH_BYTES is refused before any
    device work (the 80-layer Llama-2-70B shape needs about 168 MB)."""
    lib = gas.load()
    wl = get_workload("llama2-70b-gqa")
    fake = (ctypes.c_void_p * wl.layers)(*([256] * wl.layers))  # never dereferenced
    st = lib.gas_spectral_norms_static(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h, fake, fake, 30,
                                       256, 256, 256, None)
    assert st == gas.GAS_ERR_UNSUPPORTED
    assert b"scratch" in lib.gas_last_error(None)
