"""gas_spectral_norms_static: the allocation-free entry point for callers that cannot
allocate device memory (a host framework owns all of HBM, cudaMalloc's device
synchronisation is not allowed on the caller's path, or there is nowhere to keep a
handle).  Its results must match the handle-based gas_spectral_norms and the float64
oracle on two calls in a row, the calls must not change the device's free memory, and a
call after cudaDeviceReset (a new context) must still find its scratch array.

Collected last on purpose (file name), and independent of every other test."""

import ctypes
import json
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

import paper_2602_18851_gb300 as gas
from synth import get_workload
from tests.parity_utils import (SIGMA_RTOL, V_ATOL, assert_sigma_close, assert_v_close, gpu_inputs,
                                oracle_for)

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


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


def test_static_entry_point_matches_handle_path_and_oracle_twice():
    gas.build()
    lib = gas.load()
    cases = []
    # the larger shape first: the smaller one's scratch then overlaps what the larger one
    # left behind, none of which the call may read
    for name in ("gpt2-small", "tiny-gqa128", "gpt2-small"):
        wl = get_workload(name)
        wq, wk, v_in, _ = gpu_inputs(wl)
        ref_sigma, ref_v = _handle_reference(wl, wq, wk, v_in, wl.iters)
        o_sig, o_v = oracle_for(wl, wq, wk, v_in)
        sigma = torch.full((wl.layers, wl.n_q), float("nan"), device="cuda")
        v_out = torch.full_like(v_in, float("nan"))
        cases.append((wl, wq, wk, v_in, sigma, v_out, ref_sigma, ref_v, o_sig, o_v))
    torch.cuda.synchronize()
    for i, (wl, wq, wk, v_in, sigma, v_out, ref_sigma, ref_v, o_sig, o_v) in enumerate(cases):
        free_before = torch.cuda.mem_get_info()[0]
        st = _static_call(lib, wl, wq, wk, v_in, sigma, v_out, wl.iters)
        assert st == gas.GAS_OK, lib.gas_last_error(None)
        torch.cuda.synchronize()
        if i > 0:  # the first call may load the library's device image; later calls allocate nothing
            assert torch.cuda.mem_get_info()[0] == free_before
        got_s = sigma.double().cpu().numpy().ravel()
        got_v = v_out.cpu().numpy()
        assert_sigma_close(got_s, ref_sigma.ravel(), rtol=SIGMA_RTOL)
        assert_v_close(got_v, ref_v, atol=V_ATOL)
        w_s = assert_sigma_close(got_s, o_sig, rtol=SIGMA_RTOL)
        w_v = assert_v_close(got_v, o_v, atol=V_ATOL)
        print(f"{wl.name}: sigma rel err vs oracle {w_s:.2e}, v_out {w_v:.2e}")


def test_scratch_query_is_the_rejection_threshold():
    """gas_static_scratch_bytes gives the bytes the entry point checks: a shape needing at
    most GAS_STATIC_SCRATCH_BYTES passes the size check, one byte-step more is refused
    before any device work (so the fake, never-dereferenced pointers are safe)."""
    lib = gas.load()
    limit = 32 * 1024 * 1024
    assert lib.gas_static_scratch_bytes(32, 4096, 32, 128) == 17965056
    assert lib.gas_static_scratch_bytes(0, 4096, 32, 128) == 0
    d, n_q, d_h = 4096, 32, 128
    fits = [L for L in range(1, 513) if lib.gas_static_scratch_bytes(L, d, n_q, d_h) <= limit]
    big = max(fits) + 1
    assert lib.gas_static_scratch_bytes(big, d, n_q, d_h) > limit
    fake = (ctypes.c_void_p * big)(*([256] * big))
    st = lib.gas_spectral_norms_static(big, d, n_q, n_q, d_h, fake, fake, 30, 256, 256, 256, None)
    assert st == gas.GAS_ERR_UNSUPPORTED
    assert str(lib.gas_static_scratch_bytes(big, d, n_q, d_h)).encode() in lib.gas_last_error(None)
    # the 80-layer Llama-2-70B shape needs about 168 MB
    wl = get_workload("llama2-70b-gqa")
    assert lib.gas_static_scratch_bytes(wl.layers, wl.d, wl.n_q, wl.d_h) > 160e6
    fake = (ctypes.c_void_p * wl.layers)(*([256] * wl.layers))
    st = lib.gas_spectral_norms_static(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h, fake, fake, 30,
                                       256, 256, 256, None)
    assert st == gas.GAS_ERR_UNSUPPORTED
    assert b"scratch" in lib.gas_last_error(None)


# Child process: no torch CUDA (torch's allocator would not survive the reset).  It calls
# the entry point, resets the device (a new primary context, the library's device code
# loaded again), calls it again with new buffers, and prints both results.
_CHILD = r"""
import ctypes, json, os, sys
import numpy as np
try:  # the CUDA runtime first, so that the library's dependency resolves to this copy
    rt = ctypes.CDLL("libcudart.so.13", mode=ctypes.RTLD_GLOBAL)
except OSError:
    rt = ctypes.CDLL("/usr/local/cuda/lib64/libcudart.so.13", mode=ctypes.RTLD_GLOBAL)
lib = ctypes.CDLL(os.path.join(sys.argv[1], "paper_2602_18851_gb300", "libgas.so"))
vp = ctypes.c_void_p
lib.gas_spectral_norms_static.argtypes = [ctypes.c_int] * 5 + [vp, vp, ctypes.c_int, vp, vp, vp, vp]
lib.gas_last_error.argtypes = [vp]
lib.gas_last_error.restype = ctypes.c_char_p
rt.cudaMalloc.argtypes = [ctypes.POINTER(vp), ctypes.c_size_t]
rt.cudaMemcpy.argtypes = [vp, vp, ctypes.c_size_t, ctypes.c_int]
rt.cudaFree.argtypes = [vp]
L, d, nq, nkv, dh, iters = (int(x) for x in sys.argv[2:8])
data = np.load(sys.argv[8])
def check(rc, what):
    if rc != 0:
        raise SystemExit(f"{what} failed: {rc}")
def dev_copy(a):
    p = vp()
    check(rt.cudaMalloc(ctypes.byref(p), a.nbytes), "cudaMalloc")
    check(rt.cudaMemcpy(p, a.ctypes.data, a.nbytes, 1), "cudaMemcpy H2D")
    return p
out = []
check(rt.cudaSetDevice(0), "cudaSetDevice")
for rnd in range(2):
    qp = [dev_copy(np.ascontiguousarray(data["wq"][l])) for l in range(L)]
    kp = [dev_copy(np.ascontiguousarray(data["wk"][l])) for l in range(L)]
    v_in = dev_copy(np.ascontiguousarray(data["v_in"]))
    sig = dev_copy(np.full((L, nq), np.nan, np.float32))
    v_out = dev_copy(np.full((L, nq, d), np.nan, np.float32))
    qa = (vp * L)(*[p.value for p in qp])
    ka = (vp * L)(*[p.value for p in kp])
    st = lib.gas_spectral_norms_static(L, d, nq, nkv, dh, qa, ka, iters, v_in, v_out, sig, None)
    if st != 0:
        raise SystemExit(f"call {rnd}: status {st}: {lib.gas_last_error(None)}")
    check(rt.cudaDeviceSynchronize(), "cudaDeviceSynchronize")
    hs = np.empty((L, nq), np.float32)
    hv = np.empty((L, nq, d), np.float32)
    check(rt.cudaMemcpy(hs.ctypes.data, sig, hs.nbytes, 2), "cudaMemcpy D2H")
    check(rt.cudaMemcpy(hv.ctypes.data, v_out, hv.nbytes, 2), "cudaMemcpy D2H")
    out.append({"sigma": hs.tolist(), "v_out": hv.tolist()})
    for p in qp + kp + [v_in, sig, v_out]:
        rt.cudaFree(p)
    if rnd == 0:
        check(rt.cudaDeviceReset(), "cudaDeviceReset")
print("RESULT " + json.dumps(out))
"""


def test_static_entry_point_after_device_reset(tmp_path):
    gas.build()
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl, device="cpu")
    o_sig, o_v = oracle_for(wl, wq, wk, v_in)
    npz = tmp_path / "inputs.npz"
    np.savez(npz, wq=np.stack([w.view(torch.int16).numpy() for w in wq]),
             wk=np.stack([w.view(torch.int16).numpy() for w in wk]), v_in=v_in.numpy())
    args = [str(x) for x in (wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h, wl.iters)]
    r = subprocess.run([sys.executable, "-c", _CHILD, ROOT, *args, str(npz)], capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]
    line = [ln for ln in r.stdout.splitlines() if ln.startswith("RESULT ")][-1]
    res = json.loads(line[len("RESULT "):])
    assert len(res) == 2
    for rnd in res:
        assert_sigma_close(np.array(rnd["sigma"]).ravel(), o_sig, rtol=SIGMA_RTOL)
        assert_v_close(np.array(rnd["v_out"]), o_v, atol=V_ATOL)
