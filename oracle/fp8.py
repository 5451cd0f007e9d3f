"""Consumer side of the scale, in plain numpy (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline /
reference leg may use this module; the CUDA library shares no code with it.

* ``e4m3_table`` / ``e4m3_encode`` — the FP8 E4M3 format the scale targets
  (R_max = 448, Section 1): 1 sign bit, 4 exponent bits with bias 7, 3 mantissa bits;
  exponent field 0 holds the subnormals m/8 * 2^-6; the all-ones pattern S.1111.111 is
  NaN, so the largest finite magnitude is 1.75 * 2^8 = 448.  A value is encoded by
  brute force: the nearest of the 127 finite magnitudes, ties to the even code (the
  code's lowest bit is the mantissa's lowest bit).
* ``quantize`` — Algorithm 1, Stage 3: S~ = S / scale, cast to E4M3, with the numbers
  Table 4 reports per layer: the largest scaled logit ("Max Scaled") and whether any
  scaled logit exceeds 448 ("Overflow").
* ``DelayedScaling`` — the delayed-scaling comparator of Eq. 1: a per-layer history of
  activation maxima (16 steps, initialised to 1.0, eta = 0.9 in Appendix G's setup),
  scale_t = max(history) / (448 eta).
* ``slack_ratio`` / ``auto_alpha`` — Section 3.5 and Algorithm 4: r_t = max|S^(t)| /
  B_max^(t) (Eq. 16) with B_max = sigma_l d / sqrt(d_h); alpha_final = Quantile_q(R) *
  kappa.

Readings where the paper is silent (the kernels follow the same ones):
* the division S / scale is one IEEE float32 division, rounded to nearest: the code
  is decided in the kernel's precision;
* rounding to E4M3 is to nearest, ties to even; an overflow (|S~| > 448, or S~ not a
  number) either saturates to +-448 or becomes NaN (code 0x7F), the caller chooses; the
  overflow count includes NaN and infinite S~; every NaN output is code 0x7F;
* the sign of a zero or of a value rounding to zero is kept (-0 is code 0x80);
* amax = max |S| propagates NaN; "Max Scaled" = amax / scale in float32;
* the delayed scale is max(history) / float32(448 eta) in float32, NaN-propagating;
* one slack ratio per (step, layer), sigma_l = max over the layer's heads; slack
  ratios that are not finite are left out of R; the quantile interpolates linearly
  between order statistics (position q (m - 1) among m sorted values).
"""

import math

import numpy as np

R_MAX = 448.0
NAN_CODE = 0x7F
MAX_CODE = 0x7E


def e4m3_table() -> np.ndarray:
    """Values of the 256 codes, in float64 (NaN for 0x7F and 0xFF)."""
    out = np.empty(256, dtype=np.float64)
    for code in range(256):
        sign = -1.0 if code & 0x80 else 1.0
        e = (code >> 3) & 0xF
        m = code & 0x7
        if e == 0xF and m == 0x7:
            out[code] = math.nan
        elif e == 0:
            out[code] = sign * (m / 8.0) * 2.0 ** -6
        else:
            out[code] = sign * (1.0 + m / 8.0) * 2.0 ** (e - 7)
    return out


_MAG = e4m3_table()[:127]  # codes 0x00 .. 0x7E: the finite non-negative magnitudes, increasing


def e4m3_encode(x, saturate: bool = True) -> np.ndarray:
    """Encode float32 values as E4M3 codes (uint8), nearest value, ties to even."""
    x0 = np.asarray(x, dtype=np.float32)
    x = np.atleast_1d(x0).astype(np.float64)
    a = np.abs(x)
    nan = np.isnan(x)
    over = ~nan & (a > R_MAX)
    inr = ~nan & ~over
    mag = np.zeros(x.shape, dtype=np.int64)
    ai = a[inr]
    hi = np.searchsorted(_MAG, ai, side="left")       # first magnitude >= a
    hi = np.minimum(hi, 126)
    lo = np.maximum(hi - 1, 0)
    dlo = ai - _MAG[lo]                                # exact: both are float32 values
    dhi = _MAG[hi] - ai
    pick_hi = (dhi < dlo) | ((dhi == dlo) & (hi % 2 == 0))
    exact = _MAG[hi] == ai
    mag[inr] = np.where(exact | pick_hi, hi, lo)
    mag[over] = MAX_CODE if saturate else NAN_CODE
    code = mag | np.where(np.signbit(x), 0x80, 0)
    code[over & ~np.bool_(saturate)] = NAN_CODE
    code[nan] = NAN_CODE
    return code.astype(np.uint8).reshape(x0.shape)


def scaled_logits(s, scale) -> np.ndarray:
    """S / scale as one float32 division per element."""
    s32 = np.asarray(s, dtype=np.float32)
    with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
        return (s32 / np.float32(scale)).astype(np.float32)


def quantize(s, scale, saturate: bool = True):
    """Algorithm 1, Stage 3 for one layer's logits S (float32 values; bf16 inputs are
    widened exactly).  Returns (codes, stats) with stats = amax, max_scaled, overflow
    (number of scaled logits that are NaN or beyond +-448) and count."""
    s32 = np.asarray(s, dtype=np.float32).ravel()
    q = scaled_logits(s32, scale)
    codes = e4m3_encode(q, saturate)
    if s32.size:
        amax = np.float32(np.max(np.abs(s32)))  # np.max propagates NaN
    else:
        amax = np.float32(0.0)
    with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
        max_scaled = np.float32(amax / np.float32(scale))
        overflow = int(np.count_nonzero(np.isnan(q) | (np.abs(q) > R_MAX)))
    return codes, {"amax": float(amax), "max_scaled": float(max_scaled), "overflow": overflow,
                   "count": int(s32.size)}


def nan_max(values) -> np.float32:
    """Largest value, NaN if any value is NaN."""
    v = np.asarray(values, dtype=np.float32)
    return np.float32(np.max(v))  # np.max propagates NaN


class DelayedScaling:
    """Eq. 1 per layer: a ring of the last `history_len` maxima, initialised to `init`."""

    def __init__(self, layers: int, history_len: int = 16, init: float = 1.0):
        self.hist = np.full((layers, history_len), np.float32(init), dtype=np.float32)
        self.pos = 0

    def scales(self, eta: float = 0.9) -> np.ndarray:
        den = np.float32(R_MAX * eta)
        with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
            return np.array([nan_max(h) / den for h in self.hist], dtype=np.float32)

    def push(self, amax_per_layer) -> None:
        self.hist[:, self.pos] = np.asarray(amax_per_layer, dtype=np.float32)
        self.pos = (self.pos + 1) % self.hist.shape[1]


def slack_ratio(amax_per_layer, sigma_heads, d: int, d_h: int) -> np.ndarray:
    """Eq. 16 per layer: r = amax / B_max, B_max = sigma_l * d / sqrt(d_h), in float32
    (sigma_l = max over the layer's heads)."""
    c = np.float32(d / math.sqrt(d_h))
    sig = np.asarray(sigma_heads, dtype=np.float32)
    sig_l = np.array([nan_max(row) for row in sig.reshape(sig.shape[0], -1)], dtype=np.float32)
    b = (sig_l * c).astype(np.float32)
    with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
        return (np.asarray(amax_per_layer, dtype=np.float32) / b).astype(np.float32)


def quantile_linear(values, q: float) -> float:
    """Quantile by linear interpolation between order statistics, in float64."""
    x = np.sort(np.asarray(values, dtype=np.float64))
    m = x.size
    if m == 0:
        return math.nan
    pos = q * (m - 1)
    lo = int(math.floor(pos))
    hi = min(lo + 1, m - 1)
    frac = pos - lo
    return float(x[lo] + frac * (x[hi] - x[lo]))


def auto_alpha(slack_ratios, q: float = 0.9999, kappa: float = 1.0) -> float:
    """Algorithm 4: alpha_final = Quantile_q(R) * kappa over the finite slack ratios."""
    r = np.asarray(slack_ratios, dtype=np.float64).ravel()
    r = r[np.isfinite(r)]
    return quantile_linear(r, q) * kappa
