"""Pins of the per-layer scale (Eq. 15, Section 3.4) and of the slack ratio (Eq. 16,
Section 3.5) against facts the mathematics and the paper fix, not against a retyped
formula.

* Proposition 3.2 bounds every logit S_ij = x_i^T M x_j / sqrt(d_h) of activations on the
  sqrt(d) sphere by sigma(M) d / sqrt(d_h), and the bound is attained by the pair
  x_i = sqrt(d) u_1, x_j = sqrt(d) v_1 (the top singular pair of M).  For that pair the
  slack ratio of Eq. 16 is exactly 1, and the scale of Eq. 15 with alpha = 1 maps the
  logit to exactly eta_fp8 * R_max = 0.8 * 448 = 358.4.  The logits are computed here
  from a dense SVD of the decoded bf16 weights; sigma comes from the oracle's power
  iteration, run to convergence.
* Appendix H prints a GPT-2 XL scale of 5.8 at alpha = 0.08 (d 1600, d_h 64).  The sigma
  that Eq. 15 implies from it must lie inside the per-layer range that Table 6 prints for
  GPT-2 XL (55.8 to 483.9).  A factor d / d_h or d in place of d / sqrt(d_h) falls
  outside that range.
"""

import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import calib, fp8
from tests.helpers import to_bf16_bits

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_tables.json")))


def _decode(bits):
    """bf16 bit patterns -> float64 through torch (independent of the oracle's decoder)."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)
    return t.to(torch.float64).numpy()


def _layer(rng, d, dh, n_q, spikes):
    """One MHA layer (n_q = n_kv) whose heads carry a rank-1 spike of the given sizes,
    so that sigma_1 / sigma_2 of every head is large and power iteration converges."""
    wq = np.empty((n_q * dh, d))
    wk = np.empty((n_q * dh, d))
    for h, s in enumerate(spikes):
        a = rng.standard_normal((dh, d)) * 0.02
        b = rng.standard_normal((dh, d)) * 0.02
        bq = rng.standard_normal(dh); bq /= np.linalg.norm(bq)
        x = rng.standard_normal(d); x /= np.linalg.norm(x)
        y = rng.standard_normal(d); y /= np.linalg.norm(y)
        a += s * np.outer(bq, x)
        b += s * np.outer(bq, y)
        wq[h * dh:(h + 1) * dh] = a
        wk[h * dh:(h + 1) * dh] = b
    return to_bf16_bits(wq), to_bf16_bits(wk)


def _attained_logits(qbits, kbits, head, dh, d, rng, n_rand=64):
    """Largest |S_ij| over sqrt(d)-sphere activations that include the top singular pair of
    head `head`'s M = W^Q_h W^K_h^T, computed from a dense SVD."""
    A = _decode(qbits)[head * dh:(head + 1) * dh]  # (W^Q_h)^T, d_h x d
    B = _decode(kbits)[head * dh:(head + 1) * dh]  # (W^K_h)^T
    M = A.T @ B
    U, s, Vt = np.linalg.svd(M)
    X = rng.standard_normal((n_rand, d))
    X *= math.sqrt(d) / np.linalg.norm(X, axis=1, keepdims=True)
    X = np.vstack([math.sqrt(d) * U[:, 0], math.sqrt(d) * Vt[0], X])
    S = (X @ A.T) @ (X @ B.T).T / math.sqrt(dh)  # q_i . k_j / sqrt(d_h)
    return np.abs(S).max(), s[0]


@pytest.mark.parametrize("d,dh", [(256, 16), (384, 32)])
def test_slack_ratio_and_scale_at_the_attained_bound(d, dh):
    rng = np.random.default_rng(1885100 + d)
    spikes = [3.0, 1.5]  # head 0 carries the layer's maximum sigma
    qb, kb = _layer(rng, d, dh, 2, spikes)
    v0 = rng.standard_normal((1, 2, d)).astype(np.float32)
    sig, _ = oracle.spectral_norms([qb], [kb], v0, 200, 2, 2, dh)
    amax, s1 = _attained_logits(qb, kb, 0, dh, d, rng)
    # the oracle's converged sigma is the top singular value of the dense M
    assert sig[0, 0] == pytest.approx(s1, rel=1e-12)
    assert sig[0, 0] > sig[0, 1]
    # the pair attains Proposition 3.2's bound: max |S| = sigma d / sqrt(d_h)
    assert amax == pytest.approx(s1 * d / math.sqrt(dh), rel=1e-12)
    # Eq. 16: r = max|S| / (sigma_l d / sqrt(d_h)) = 1 (in float32)
    r = fp8.slack_ratio([amax], sig, d, dh)
    assert r[0] == pytest.approx(1.0, rel=2e-6)
    # Eq. 15 with alpha = 1: the attained logit lands exactly on eta * R_max = 358.4
    s, _, a = calib.layer_scales(sig, d, dh, alpha_override=1.0)
    assert a == 1.0
    c = GOLD["scale_constants"]
    assert amax / s[0] == pytest.approx(c["safe_range"], rel=1e-12)
    # and with the eta / R_max of any other format, on eta * R_max
    s2, _, _ = calib.layer_scales(sig, d, dh, alpha_override=1.0, eta_fp8=0.5, r_max=57344.0)
    assert amax / s2[0] == pytest.approx(0.5 * 57344.0, rel=1e-12)
    # the second head's own top pair stays below the layer's bound: r < 1
    amax1, _ = _attained_logits(qb, kb, 1, dh, d, rng)
    assert fp8.slack_ratio([amax1], sig, d, dh)[0] < 0.9


def test_slack_ratio_below_one_on_random_sphere_activations():
    """Proposition 3.2: without the singular pair, activations on the sqrt(d) sphere stay
    strictly inside the bound, so r < 1, and alpha = 1 keeps every scaled logit at or
    below 358.4."""
    rng = np.random.default_rng(1885199)
    d, dh = 256, 16
    qb, kb = _layer(rng, d, dh, 1, [2.0])
    v0 = rng.standard_normal((1, 1, d)).astype(np.float32)
    sig, _ = oracle.spectral_norms([qb], [kb], v0, 200, 1, 1, dh)
    A, B = _decode(qb), _decode(kb)
    X = rng.standard_normal((512, d))
    X *= math.sqrt(d) / np.linalg.norm(X, axis=1, keepdims=True)
    amax = np.abs((X @ A.T) @ (X @ B.T).T / math.sqrt(dh)).max()
    assert 0.0 < fp8.slack_ratio([amax], sig, d, dh)[0] < 1.0
    s, _, _ = calib.layer_scales(sig, d, dh, alpha_override=1.0)
    assert amax / s[0] < 358.4


def test_appendix_h_scale_implies_a_table6_sigma():
    sp = GOLD["spike_test"]
    row = {r["model"]: r for r in GOLD["spectral_stats"]["rows"]}["GPT-2 XL"]
    c = GOLD["scale_constants"]
    per_sigma = float(calib.scale_from_sigma(1.0, sp["alpha"], sp["d"], sp["d_h"], c["eta_fp8"], c["r_max"]))
    sigma = sp["scale_before"] / per_sigma
    assert row["min"] <= sigma <= row["max"], sigma
    # the same through the per-head entry point used by the library's parity tests
    s, _, _ = calib.layer_scales(np.array([[sigma]]), sp["d"], sp["d_h"], alpha_override=sp["alpha"])
    assert s[0] == pytest.approx(sp["scale_before"], rel=1e-12)
    # the factors a slip would produce leave Table 6's range
    for wrong in (sp["d"] / sp["d_h"], sp["d"], math.sqrt(sp["d"])):
        alt = sp["scale_before"] * c["eta_fp8"] * c["r_max"] / (sp["alpha"] * wrong)
        assert not (row["min"] <= alt <= row["max"]), wrong
