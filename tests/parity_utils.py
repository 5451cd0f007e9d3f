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



def top_right_singular(wq_l, wk_l, head, wl):
    """Top right singular vector v_1 of M_h = W^Q_h W^K_g^T = A^T B (d-vector) and the
    singular values.  With B^T = Q R (QR), M = (A^T R^T) Q^T, so v_1 = Q w_1 for the top
    right singular vector w_1 of the d x d_h matrix A^T R^T.  numpy only."""
    from tests.helpers import bits_to_f64, tensor_bits
    g = head // wl.group
    A = bits_to_f64(tensor_bits(wq_l)[head * wl.d_h:(head + 1) * wl.d_h])
    B = bits_to_f64(tensor_bits(wk_l)[g * wl.d_h:(g + 1) * wl.d_h])
    Q, R = np.linalg.qr(B.T)
    _, S, Wt = np.linalg.svd(A.T @ R.T, full_matrices=False)
    return Q @ Wt[0], S


# Backward-error bound for v_out on heads whose start vector is nearly orthogonal to v_1.
V1_BACKWARD_TOL = 1e-6


def assert_v_close_or_v1_backward(got, want, wl, wq, wk, v_in, atol=V_ATOL):
    """v_out within `atol` of the oracle's on every head, or else the exact k-step iterate
    of a start vector that differs from v_in only along the top right singular vector v_1,
    by less than V1_BACKWARD_TOL (relative to ||v_in||).

    Why: the k iterations multiply the start vector's v_1 component c_1 by
    (sigma_1 / sigma_i)^(2k) against every other component.  When |c_1| is near the
    rounding level of the operands (16-bit hi + lo splits, fp32 sums: about 1e-7), the
    rounding moves it by a comparable amount, possibly across zero, and the iterate's
    mixture of v_1 and the rest (its v_1 sign, even) follows that moved c_1.  Start
    vectors that differ along v_1 give iterates normalize(v_k + beta v_1): beta is fitted
    from the v_1 component of the result, and the perturbation it stands for,
    delta = c_1 beta / (v_k . v_1), must stay below the bound.
    Returns (worst distance after the fit, list of (layer, head, c_1, delta))."""
    L, nq, d = wl.layers, wl.n_q, wl.d
    got = np.asarray(got, dtype=np.float64).reshape(L, nq, d)
    want = np.asarray(want, dtype=np.float64).reshape(L, nq, d)
    dist = np.linalg.norm(got - want, axis=-1)
    fitted = []
    vin = v_in.detach().cpu().numpy()
    for l, h in np.argwhere(dist > atol):
        v1, _ = top_right_singular(wq[l], wk[l], int(h), wl)
        v0 = vin[l, h].astype(np.float64)
        c1 = float(v1 @ (v0 / np.linalg.norm(v0)))
        w, g = want[l, h], got[l, h] / np.linalg.norm(got[l, h])
        a, b = float(w @ v1), float(g @ v1)
        r = w - a * v1
        nr = float(np.linalg.norm(r))
        t = b * nr / np.sqrt(max(1.0 - b * b, 1e-300))   # v_1 coefficient that matches g's
        fit = (t * v1 + r) / np.sqrt(t * t + nr * nr)
        dfit = float(np.linalg.norm(got[l, h] - fit))
        delta = c1 * (t - a) / a if abs(a) > 1e-3 else float("inf")
        assert dfit <= atol and abs(delta) < V1_BACKWARD_TOL, (
            f"v_out layer {l} head {h}: distance {dist[l, h]:.3e}; start-vector v_1 component "
            f"{c1:+.3e}, fitted perturbation {delta:+.3e}, distance after the fit {dfit:.3e}")
        fitted.append((int(l), int(h), c1, delta))
        dist[l, h] = dfit
    return float(dist.max()), fitted
