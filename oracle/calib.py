"""Float64 calibration rule of the paper (test infrastructure only).

* Eq. 12 (gamma selection, Section 3.2): h(gamma) = gamma - 1 - ln(gamma) must be at
  least (2/d_h) ln(2 N L / delta*), N = n_layers * n_heads.  gamma_min is the
  smallest gamma > 1 meeting it, found by bisection (h is increasing on (1, inf)).
  When the right-hand side is <= 0 every gamma > 1 qualifies; gamma_min is taken
  as its infimum 1.
* Eq. 13 (alpha selection): alpha_min = sqrt(2 gamma d_h)/d * sqrt(ln(4 N L^2 / delta*)),
  with the logarithm clamped at 0 (a target probability so loose that it is met
  by alpha = 0).
* Eq. 15 (per-layer scale, Section 3.4):
  scale_l = alpha * sigma_l * (d / sqrt(d_h)) / (eta_fp8 * R_max), sigma_l = max_h sigma_{l,h}.
"""

import math

import numpy as np


def h(gamma: float) -> float:
    """h(gamma) = gamma - 1 - ln(gamma) (Proposition 3.4, Eq. 10)."""
    return gamma - 1.0 - math.log(gamma)


def gamma_rhs(d_h: int, n_heads_total: int, seq_len: int, delta_star: float) -> float:
    return (2.0 / d_h) * math.log(2.0 * n_heads_total * seq_len / delta_star)


def gamma_min(d_h: int, n_heads_total: int, seq_len: int, delta_star: float) -> float:
    rhs = gamma_rhs(d_h, n_heads_total, seq_len, delta_star)
    if rhs <= 0.0:
        return 1.0
    lo, hi = 1.0, 2.0
    while h(hi) < rhs:
        hi *= 2.0
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if h(mid) >= rhs:
            hi = mid
        else:
            lo = mid
        if hi - lo <= 1e-13 * hi:
            break
    return hi


def alpha_min(gamma: float, d: int, d_h: int, n_heads_total: int, seq_len: int,
              delta_star: float) -> float:
    lg = math.log(4.0 * n_heads_total * seq_len * seq_len / delta_star)
    return math.sqrt(2.0 * gamma * d_h) / d * math.sqrt(max(lg, 0.0))


def improvement_factor(gamma: float, d: int, d_h: int) -> float:
    """Rank-aware over rank-agnostic tail exponent ratio d/(gamma d_h) (Appendix B.3)."""
    return d / (gamma * d_h)


def scale_from_sigma(sigma_layer, alpha: float, d: int, d_h: int, eta_fp8: float,
                     r_max: float):
    """Eq. 15 for a per-layer sigma (array or scalar)."""
    return alpha * np.asarray(sigma_layer, dtype=np.float64) * (d / math.sqrt(d_h)) / (eta_fp8 * r_max)


def layer_scales(sigma_heads, d: int, d_h: int, *, gamma: float = 0.0,
                 delta_star: float = 1e-6, seq_len: int = 1024, eta_fp8: float = 0.8,
                 r_max: float = 448.0, alpha_override: float = 0.0):
    """Per-layer scales from per-head sigmas [layers, n_q].

    gamma <= 0 selects gamma_min (Eq. 12); alpha_override > 0 replaces alpha_min.
    Returns (scales[layers], gamma, alpha).
    """
    s = np.asarray(sigma_heads, dtype=np.float64)
    layers, n_q = s.shape
    n_total = layers * n_q
    if gamma <= 0.0:
        gamma = gamma_min(d_h, n_total, seq_len, delta_star)
    elif gamma <= 1.0:
        raise ValueError("gamma must exceed 1 (Proposition 3.4)")
    alpha = alpha_override if alpha_override > 0.0 else alpha_min(
        gamma, d, d_h, n_total, seq_len, delta_star)
    sigma_layer = s.max(axis=1)
    return scale_from_sigma(sigma_layer, alpha, d, d_h, eta_fp8, r_max), gamma, alpha
