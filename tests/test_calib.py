"""Pins for the oracle's calibration rule (Eq. 12, Eq. 13, Eq. 15) against values the
paper prints (Table 2, Table 3, Section 5.1, Appendix H) and against closed forms."""

import json
import math
import os

import numpy as np
import pytest

from oracle import calib

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_tables.json")))
DELTA = GOLD["table3_alpha_min"]["delta_star"]
SEQ = GOLD["table3_alpha_min"]["seq_len"]


def _n_heads(model):
    for r in GOLD["table3_alpha_min"]["rows"]:
        if r["model"] == model:
            return r["N"]
    raise KeyError(model)


@pytest.mark.parametrize("row", GOLD["table2_concentration"]["rows"], ids=lambda r: r["model"])
def test_gamma_matches_table2(row):
    """Table 2 prints gamma to 2 decimals, not consistently rounded: GPT-2 XL's
    2.9853 is printed 2.98, and the 13B / 70B entries sit 0.01-0.02 above the
    minimal gamma (any gamma >= gamma_min satisfies Eq. 12).  Pin:
    |gamma_min - printed| <= 0.02, and printed + 0.01 satisfies Eq. 12."""
    g = calib.gamma_min(row["d_h"], _n_heads(row["model"]), SEQ, DELTA)
    assert abs(g - row["gamma"]) <= 0.02
    rhs = calib.gamma_rhs(row["d_h"], _n_heads(row["model"]), SEQ, DELTA)
    assert calib.h(row["gamma"] + 0.01) >= rhs


@pytest.mark.parametrize("row", GOLD["table2_concentration"]["rows"], ids=lambda r: r["model"])
def test_improvement_factor_table2(row):
    """d/(gamma d_h) rounds to the printed integer factor (Appendix B.3)."""
    assert round(calib.improvement_factor(row["gamma"], row["d"], row["d_h"])) == row["improvement"]
    g = calib.gamma_min(row["d_h"], _n_heads(row["model"]), SEQ, DELTA)
    assert abs(calib.improvement_factor(g, row["d"], row["d_h"]) - row["improvement"]) < 0.5


@pytest.mark.parametrize("row", GOLD["table3_alpha_min"]["rows"], ids=lambda r: r["model"])
def test_alpha_min_matches_table3(row):
    """Table 3 prints alpha_min to 3 decimals.  Pin: half a unit of the printed digit
    plus 1e-4 (GPT-2 XL's printed 0.074 lies 0.0005 above the computed 0.0735)."""
    g = calib.gamma_min(row["d_h"], row["N"], SEQ, DELTA)
    a = calib.alpha_min(g, row["d"], row["d_h"], row["N"], SEQ, DELTA)
    assert abs(a - row["alpha_min"]) <= 0.0006


@pytest.mark.parametrize("row", GOLD["alpha_used"]["rows"], ids=lambda r: r["model"])
def test_alpha_used_exceeds_alpha_min(row):
    """Section 3.2: the alphas used in the experiments exceed alpha_min."""
    t3 = {r["model"]: r for r in GOLD["table3_alpha_min"]["rows"]}[row["model"]]
    g = calib.gamma_min(t3["d_h"], t3["N"], SEQ, DELTA)
    a = calib.alpha_min(g, t3["d"], t3["d_h"], t3["N"], SEQ, DELTA)
    assert row["alpha"] > a


def test_gamma_solution_is_tight():
    """gamma_min satisfies Eq. 12 and anything noticeably below it does not."""
    for dh, n in [(64, 1200), (128, 5120), (128, 1), (64, 10**6)]:
        g = calib.gamma_min(dh, n, SEQ, DELTA)
        rhs = calib.gamma_rhs(dh, n, SEQ, DELTA)
        assert calib.h(g) >= rhs - 1e-12
        assert calib.h(g * (1 - 1e-9)) < rhs


def test_gamma_degenerate_rhs():
    """A target probability looser than 2NL makes the rhs of Eq. 12 <= 0: gamma -> 1."""
    assert calib.gamma_min(64, 1, 1, 10.0) == 1.0
    # alpha with gamma = 1 is still the closed form of Eq. 13.
    a = calib.alpha_min(1.0, 256, 64, 1, 1, 10.0)
    assert a == 0.0  # ln(4 N L^2 / delta*) = ln(0.4) < 0, clamped


def test_h_closed_form():
    """h(gamma) = gamma - 1 - ln gamma: h(1) = 0, h(e) = e - 2, increasing above 1."""
    assert calib.h(1.0) == 0.0
    assert abs(calib.h(math.e) - (math.e - 2.0)) < 1e-15
    xs = np.linspace(1.001, 10, 200)
    hs = [calib.h(x) for x in xs]
    assert all(b > a for a, b in zip(hs, hs[1:]))


def test_tail_terms_meet_target():
    """With gamma_min and alpha_min, N*T1 <= delta*/2 and N*T2 <= delta*/2 (Eqs. 10-11,
    union bound of Section 3.2), with equality up to rounding."""
    for dh, d, n in [(64, 1600, 1200), (128, 8192, 5120)]:
        g = calib.gamma_min(dh, n, SEQ, DELTA)
        a = calib.alpha_min(g, d, dh, n, SEQ, DELTA)
        t1 = SEQ * math.exp(-dh / 2 * (g - 1 - math.log(g)))
        t2 = 2 * SEQ ** 2 * math.exp(-(d ** 2) * a ** 2 / (2 * g * dh))
        assert n * t1 <= DELTA / 2 * (1 + 1e-9)
        assert n * t2 <= DELTA / 2 * (1 + 1e-9)
        assert n * t1 > DELTA / 2 * (1 - 1e-6)
        assert n * t2 > DELTA / 2 * (1 - 1e-6)


def test_scale_formula_closed_form():
    """Eq. 15 with Section 5.1's constants: safe range 0.8 * 448 = 358.4."""
    c = GOLD["scale_constants"]
    assert c["eta_fp8"] * c["r_max"] == pytest.approx(c["safe_range"], abs=1e-12)
    sig = np.array([[1.0, 3.0], [2.0, 0.5]])
    s, g, a = calib.layer_scales(sig, d=4096, d_h=128, alpha_override=0.04)
    expect = 0.04 * np.array([3.0, 2.0]) * (4096 / math.sqrt(128)) / 358.4
    np.testing.assert_allclose(s, expect, rtol=1e-15)
    assert a == 0.04


def test_scale_spike_homogeneity():
    """Appendix H: 4x on both W^Q and W^K multiplies sigma, hence the scale, by 16.
    5.8 * 16 = 92.8 is within 2% of the printed 93.8 (which also includes one step)."""
    sp = GOLD["spike_test"]
    base = np.array([[sp["scale_before"]]])
    s1, _, _ = calib.layer_scales(base, d=1600, d_h=64, alpha_override=0.08)
    s2, _, _ = calib.layer_scales(base * sp["factor"] ** 2, d=1600, d_h=64, alpha_override=0.08)
    assert s2[0] / s1[0] == pytest.approx(16.0, rel=1e-15)
    assert sp["scale_before"] * 16 == pytest.approx(sp["scale_after"], rel=0.02)


def test_gamma_rejects_le_one():
    with pytest.raises(ValueError):
        calib.layer_scales(np.ones((1, 1)), d=64, d_h=64, gamma=0.5)
    with pytest.raises(ValueError):
        calib.layer_scales(np.ones((1, 1)), d=64, d_h=64, gamma=1.0)


def test_nan_sigma_propagates():
    s, _, _ = calib.layer_scales(np.array([[1.0, np.nan]]), d=64, d_h=64)
    assert np.isnan(s[0])


def test_gqa_expansion_memory():
    """Section 4.2: expanding W^K on Mistral-7B costs 32 MB per layer in FP16."""
    m = GOLD["gqa_expansion_memory"]
    nbytes = m["n_q"] * m["d_h"] * m["d"] * m["bytes_per_elem"]
    assert nbytes / 2 ** 20 == m["megabytes"]
