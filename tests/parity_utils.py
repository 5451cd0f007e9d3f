"""Shared plumbing for the GPU parity tests: run the library on seeded inputs, run
the oracle on the same bytes, compare with the tolerances the tests state."""

import numpy as np
import torch

import oracle
from oracle import calib
from synth import make_start_vectors, make_weights
from tests.helpers import tensor_bits

# Tolerances.  sigma and scale: 1e-3 relative (the stated bar).  v_out: unit vectors,
# compared by Euclidean distance <= 1e-3.
SIGMA_RTOL = 1e-3
SCALE_RTOL = 1e-3
V_ATOL = 1e-3


def gpu_inputs(wl, device="cuda"):
    wq, wk, meta = make_weights(wl, device=device)
    v_in = make_start_vectors(wl, device=device)
    return wq, wk, v_in, meta


def run_library(wl, wq, wk, v_in, method="gram", iters=None, write_back=True, fused=True,
                gamma=0.0, delta=1e-6, r_max=448.0, alpha_override=0.0):
    import paper_2602_18851_gb300 as gas
    h = gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h)
    h.set_method(method)
    if alpha_override:
        h.set_calibration(alpha_override=alpha_override)
    iters = wl.iters if iters is None else iters
    if fused:
        sigma, s, v_out = h.refresh(wq, wk, iters, v_in, gamma=gamma, delta_star=delta, r_max=r_max,
                                    write_back=write_back)
    else:
        sigma, v_out = h.spectral_norms(wq, wk, iters, v_in, write_back=write_back)
        s = h.scales(sigma, gamma=gamma, delta_star=delta, r_max=r_max)
    torch.cuda.synchronize()
    status = h.device_status(clear=True)
    out = {"sigma": sigma.double().cpu().numpy(), "s": s.double().cpu().numpy(),
           "v_out": v_out.cpu().numpy() if v_out is not None else None, "status": status,
           "launches": h.last_launch_count}
    h.close()
    return out


def oracle_for(wl, wq, wk, v_in, pairs=None, iters=None, mode="factored", layers=None):
    """Oracle sigma / v_out for the given (layer, head) pairs (default: all heads)."""
    iters = wl.iters if iters is None else iters
    if pairs is None:
        pairs = [(l, h) for l in range(wl.layers) for h in range(wl.n_q)]
    need = sorted({l for l, _ in pairs})
    qb = [None] * wl.layers
    kb = [None] * wl.layers
    for l in need:
        qb[l] = tensor_bits(wq[l])
        kb[l] = tensor_bits(wk[l])
    vin = v_in.detach().cpu().numpy()
    sig, v = oracle.heads(wl.d, wl.n_q, wl.n_kv, wl.d_h, qb, kb, vin, iters, pairs, mode=mode)
    return sig, v


def oracle_scales(wl, sigma_heads, gamma=0.0, delta=1e-6, r_max=448.0, alpha_override=0.0,
                  n_heads_total=None):
    s = np.asarray(sigma_heads, dtype=np.float64)
    n_total = wl.layers * wl.n_q if n_heads_total is None else n_heads_total
    g = gamma if gamma > 0 else calib.gamma_min(wl.d_h, n_total, 1024, delta)
    a = alpha_override if alpha_override > 0 else calib.alpha_min(g, wl.d, wl.d_h, n_total, 1024, delta)
    return calib.scale_from_sigma(s.max(axis=-1), a, wl.d, wl.d_h, 0.8, r_max)


def assert_sigma_close(got, want, rtol=SIGMA_RTOL, what="sigma"):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    assert got.shape == want.shape, (got.shape, want.shape)
    zero = want == 0.0
    assert np.all(got[zero] == 0.0), f"{what}: expected exact zeros"
    rel = np.abs(got[~zero] - want[~zero]) / np.abs(want[~zero])
    worst = float(rel.max()) if rel.size else 0.0
    assert worst <= rtol, f"{what}: max rel err {worst:.3e} > {rtol:.0e}"
    return worst


def assert_v_close(got, want, atol=V_ATOL):
    got = np.asarray(got, dtype=np.float64).reshape(-1, want.shape[-1])
    want = np.asarray(want, dtype=np.float64).reshape(-1, want.shape[-1])
    dist = np.linalg.norm(got - want, axis=-1)
    worst = float(dist.max())
    assert worst <= atol, f"v_out: max distance {worst:.3e} > {atol:.0e}"
    return worst

