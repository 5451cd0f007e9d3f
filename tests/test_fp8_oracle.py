"""Pins for oracle/fp8.py: the E4M3 format against PyTorch's float8_e4m3fn (an
independent implementation of the same format), hand-worked ties and overflow cases,
Eq. 1's ring semantics, Eq. 16's closed form and Algorithm 4's quantile against
numpy's."""

import math

import numpy as np
import pytest
import torch

from oracle import fp8


def torch_encode(x):
    return torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.float8_e4m3fn).view(torch.uint8).numpy()


def test_table_matches_torch_decode():
    t = torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).float().double().numpy()
    tab = fp8.e4m3_table()
    assert np.array_equal(np.isnan(t), np.isnan(tab))
    assert np.array_equal(t[~np.isnan(t)], tab[~np.isnan(tab)])
    assert tab[0x7E] == 448.0 and tab[0x01] == 2.0 ** -9 and tab[0x08] == 2.0 ** -6
    assert np.isnan(tab[0x7F]) and np.isnan(tab[0xFF])


def test_encode_matches_torch_in_range():
    """Inside +-448 torch's cast rounds to nearest, ties to even, like the oracle; the
    sample includes every midpoint and its float32 neighbours."""
    rng = np.random.default_rng(1885)
    tab = fp8.e4m3_table()
    x = np.concatenate([rng.uniform(-448, 448, 50000),
                        rng.standard_normal(50000) * np.exp(rng.uniform(-14, 5, 50000))]).astype(np.float32)
    x = x[np.abs(x) <= 448]
    mid = ((tab[:126] + tab[1:127]) / 2).astype(np.float32)
    x = np.concatenate([x, mid, -mid, np.nextafter(mid, np.float32(0)), np.nextafter(mid, np.float32(1e3)),
                        tab[:127].astype(np.float32), -tab[:127].astype(np.float32)])
    assert np.array_equal(fp8.e4m3_encode(x), torch_encode(x))


@pytest.mark.parametrize("value,code", [
    (0.0, 0x00), (-0.0, 0x80), (2.0 ** -10, 0x00), (-(2.0 ** -10), 0x80),  # tie 0 | 2^-9 -> even 0
    (3 * 2.0 ** -10, 0x02),              # tie 2^-9 (code 1) | 2^-8 (code 2) -> 2
    (1.0625, 0x38), (1.1875, 0x3A),      # ties around 1.0, 1.125, 1.25
    (15 * 2.0 ** -10, 0x08),             # 7.5 * 2^-9 ties 7 * 2^-9 | 2^-6 -> code 8
    (440.0, 0x7E), (432.0, 0x7E), (431.9, 0x7D), (448.0, 0x7E), (-448.0, 0xFE),
])
def test_encode_hand_cases(value, code):
    assert int(fp8.e4m3_encode(np.float32(value))) == code


def test_overflow_saturates_or_gives_nan():
    over = np.array([np.nextafter(np.float32(448), np.float32(1e3)), 464.0, 1e30, np.inf], dtype=np.float32)
    assert list(fp8.e4m3_encode(over, saturate=True)) == [0x7E] * 4
    assert list(fp8.e4m3_encode(-over, saturate=True)) == [0xFE] * 4
    assert list(fp8.e4m3_encode(over, saturate=False)) == [0x7F] * 4
    assert list(fp8.e4m3_encode(-over, saturate=False)) == [0x7F] * 4
    assert list(fp8.e4m3_encode(np.array([np.nan, -np.nan], np.float32))) == [0x7F, 0x7F]


def test_quantize_stats_on_planted_logits():
    rng = np.random.default_rng(7)
    s = rng.standard_normal(4096).astype(np.float32)
    scale = np.float32(0.01)                         # |S/scale| > 448  <=>  |S| > 4.48
    s[[5, 17, 900]] = [5.0, -7.25, 4.49]
    s[[33]] = 4.48                                   # 4.48 / 0.01 rounds to 448.00003 in float32?
    codes, st = fp8.quantize(s, scale)
    q = (s / scale).astype(np.float32)
    assert st["count"] == 4096
    assert st["amax"] == np.float32(7.25)
    assert st["max_scaled"] == np.float32(np.float32(7.25) / scale)
    assert st["overflow"] == int(np.count_nonzero(np.abs(q) > 448))
    assert st["overflow"] >= 3
    assert codes[5] == 0x7E and codes[17] == 0xFE
    codes_nan, st2 = fp8.quantize(s, scale, saturate=False)
    assert codes_nan[17] == 0x7F and st2["overflow"] == st["overflow"]
    # dividing by the scale is one float32 division: codes equal the encoding of S/scale
    assert np.array_equal(codes, fp8.e4m3_encode(q))


def test_quantize_special_values():
    s = np.array([np.nan, np.inf, -np.inf, -0.0, 0.0, 1e-30], dtype=np.float32)
    codes, st = fp8.quantize(s, np.float32(1.0))
    assert list(codes) == [0x7F, 0x7E, 0xFE, 0x80, 0x00, 0x00]
    assert math.isnan(st["amax"]) and math.isnan(st["max_scaled"])
    assert st["overflow"] == 3
    codes, st = fp8.quantize(np.zeros(0, np.float32), np.float32(2.0))
    assert codes.size == 0 and st == {"amax": 0.0, "max_scaled": 0.0, "overflow": 0, "count": 0}
    _, st = fp8.quantize(np.ones(4, np.float32), np.float32(0.0))  # 1/0 = inf: all overflow
    assert st["overflow"] == 4 and st["max_scaled"] == math.inf


def test_delayed_scaling_ring():
    """Eq. 1: scale = max(history) / (448 eta); the 16-entry history starts at 1.0
    (Appendix G) and forgets a maximum 16 pushes later."""
    ds = fp8.DelayedScaling(layers=2, history_len=16, init=1.0)
    den = np.float32(448 * 0.9)
    assert np.array_equal(ds.scales(0.9), np.full(2, np.float32(1.0) / den))
    ds.push([500.0, 0.5])
    assert ds.scales(0.9)[0] == np.float32(500.0) / den
    assert ds.scales(0.9)[1] == np.float32(1.0) / den   # init entries still in the window
    for _ in range(15):
        ds.push([2.0, 0.5])
    assert ds.scales(0.9)[0] == np.float32(500.0) / den  # 500 is the oldest of 16
    assert ds.scales(0.9)[1] == np.float32(0.5) / den    # every 1.0 has been overwritten
    ds.push([2.0, np.nan])
    assert ds.scales(0.9)[0] == np.float32(2.0) / den
    assert math.isnan(ds.scales(0.9)[1])


def test_delayed_scaling_reenacts_the_spike():
    """Appendix H's mechanism: after steady steps the delayed scale puts the maximum at
    eta * 448; multiplying W^Q and W^K by 4 multiplies every logit by 16, so the first
    spiked step's largest scaled logit is 16 * 0.9 * 448 = 6451.2 (Appendix H reports
    scaled logits above 6500)."""
    ds = fp8.DelayedScaling(layers=1)
    amax = np.float32(3.0)
    for _ in range(20):
        ds.push([amax])
    s_del = ds.scales(0.9)[0]
    _, st = fp8.quantize(np.array([16 * amax], np.float32), s_del)
    assert st["max_scaled"] == pytest.approx(16 * 0.9 * 448, rel=1e-6)
    assert st["overflow"] == 1


def test_slack_ratio_closed_form():
    sig = np.array([[1.0, 3.0, 2.0], [0.5, 0.25, 0.125]], np.float32)
    r = fp8.slack_ratio([6.0, 1.0], sig, d=1024, d_h=64)   # B_max = sigma_l * 1024 / 8
    assert r[0] == pytest.approx(6.0 / (3.0 * 128.0), rel=1e-7)
    assert r[1] == pytest.approx(1.0 / (0.5 * 128.0), rel=1e-7)


@pytest.mark.parametrize("m,q", [(100, 0.9999), (8000, 0.9999), (7, 0.5), (1, 0.9), (50, 0.0), (50, 1.0)])
def test_auto_alpha_quantile_matches_numpy(m, q):
    rng = np.random.default_rng(m)
    r = rng.uniform(7.3e-5, 3.66e-4, m).astype(np.float32)
    want = np.quantile(r.astype(np.float64), q, method="linear")
    assert fp8.auto_alpha(r, q, 1.0) == pytest.approx(want, rel=1e-12)
    assert fp8.auto_alpha(r, q, 1.5) == pytest.approx(1.5 * want, rel=1e-12)


def test_auto_alpha_drops_non_finite():
    r = np.array([1.0, np.nan, 2.0, np.inf, 3.0], np.float32)
    assert fp8.auto_alpha(r, 0.5, 1.0) == 2.0
    assert math.isnan(fp8.auto_alpha(np.array([np.nan], np.float32), 0.5, 1.0))
