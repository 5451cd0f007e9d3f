"""The scale's consumer on the GPU (include/gas_fp8.h) against oracle/fp8.py:
E4M3 codes bit for bit, overflow statistics exactly, delayed-scaling scales and
history (Eq. 1), slack ratios (Eq. 16) and auto-alpha (Algorithm 4), and a synthetic
re-enactment of Appendix H's 4x weight spike through gas_refresh."""

import ctypes
import math

import numpy as np
import pytest
import torch

import paper_2602_18851_gb300 as gas
from oracle import calib, fp8
from synth import get_workload, make_start_vectors, make_weights
from synth.logits import attention_logits, gaussian_logits, special_logits, sphere_tokens


@pytest.fixture(scope="module")
def lib():
    gas.build()
    return gas.load()


# ----------------------------------------------------------------------------------
# host-side checks (no GPU needed)
# ----------------------------------------------------------------------------------
def test_fp8_create_rejects_bad_arguments_without_touching_the_device(lib):
    h = ctypes.c_void_p()
    assert lib.gas_fp8_create(0, 16, 0, ctypes.byref(h)) == gas.GAS_ERR_INVALID_ARG
    assert lib.gas_fp8_create(4, 0, 0, ctypes.byref(h)) == gas.GAS_ERR_INVALID_ARG
    assert lib.gas_fp8_create(4, 16, -1, ctypes.byref(h)) == gas.GAS_ERR_INVALID_ARG
    assert lib.gas_fp8_create(600, 16, 0, ctypes.byref(h)) == gas.GAS_ERR_UNSUPPORTED
    assert lib.gas_fp8_create(80, 16, 300, ctypes.byref(h)) == gas.GAS_ERR_UNSUPPORTED
    assert b"burn_in_steps" in lib.gas_fp8_last_error(None)
    assert lib.gas_fp8_create(4, 16, 0, None) == gas.GAS_ERR_INVALID_ARG
    assert lib.gas_fp8_destroy(None) == gas.GAS_ERR_INVALID_ARG


@pytest.mark.skipif(torch.cuda.is_available(), reason="CPU-only behaviour")
def test_fp8_create_without_gpu_fails_cleanly(lib):
    h = ctypes.c_void_p()
    assert lib.gas_fp8_create(4, 16, 0, ctypes.byref(h)) == gas.GAS_ERR_CUDA
    assert h.value is None


# ----------------------------------------------------------------------------------
# GPU parity
# ----------------------------------------------------------------------------------
MIDS = ((fp8.e4m3_table()[:126] + fp8.e4m3_table()[1:127]) / 2).tolist()


def _logits(n, scale, seed, dtype):
    """n logits: the edge values for this scale first, then Gaussian logits whose
    spread puts a few beyond 448 * scale."""
    sc = abs(scale) if math.isfinite(scale) and scale != 0 else 1.0
    edge = torch.from_numpy(special_logits(scale if math.isfinite(scale) and scale != 0 else 1.0, MIDS))
    body = gaussian_logits(max(n, 0), seed, sd=150.0 * sc, outlier_frac=1e-3, outlier=700.0 * sc,
                           dtype=torch.float32)
    x = torch.cat([edge, body])[:n].to(dtype)
    return x


def _kernel(state, layer, s, scale, saturate):
    sc = torch.tensor([scale], dtype=torch.float32, device="cuda")
    q, stats = state.quantize(layer, s, sc, saturate=saturate)
    torch.cuda.synchronize()
    return q.cpu().numpy(), gas.decode_fp8_stats(stats)[0]


def _same_stats(got, want):
    for k in ("amax", "max_scaled"):
        a, b = got[k], want[k]
        assert (math.isnan(a) and math.isnan(b)) or a == b, (k, a, b)
    assert got["overflow"] == want["overflow"] and got["count"] == want["count"]


@pytest.mark.gpu
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("saturate", [True, False])
@pytest.mark.parametrize("n", [0, 1, 15, 16, 17, 4096 + 7, 1_000_003])
def test_quantize_matches_oracle(lib, dtype, saturate, n):
    with gas.Fp8State(layers=3) as st:
        for i, scale in enumerate([0.0123, 1.0, -0.37]):
            s = _logits(n, scale, 1000 + n + i, dtype)
            codes, stats = _kernel(st, i % 3, s.cuda(), scale, saturate)
            want_codes, want = fp8.quantize(s.float().numpy(), np.float32(scale), saturate)
            assert np.array_equal(codes, want_codes.reshape(codes.shape))
            _same_stats(stats, want)


@pytest.mark.gpu
@pytest.mark.parametrize("scale", [3e-39, 0.0, math.inf, -math.inf, math.nan, 2.0 ** 126, 2.0 ** -126, 1e-30])
def test_quantize_degenerate_scales(lib, scale):
    """Scales outside the reciprocal path's range (subnormal, zero, infinite, NaN, or
    with a subnormal reciprocal) still give the IEEE quotient's code."""
    with gas.Fp8State(layers=1) as st:
        s = _logits(70_001, 1.0, 77, torch.float32)
        codes, stats = _kernel(st, 0, s.cuda(), scale, True)
        want_codes, want = fp8.quantize(s.numpy(), np.float32(scale), True)
        assert np.array_equal(codes, want_codes)
        _same_stats(stats, want)


@pytest.mark.gpu
@pytest.mark.parametrize("scale", [0.0123, 0.7, 3.3e-3, 170.0, 5.5e-6, 1.0 / 3.0])
def test_division_decides_midpoints_like_ieee(lib, scale):
    """Logits whose quotient lands on or next to every E4M3 rounding midpoint: a quotient
    one ulp off would flip a code here."""
    with gas.Fp8State(layers=1) as st:
        x = torch.from_numpy(special_logits(scale, MIDS))
        rng = np.random.default_rng(5)
        y = torch.from_numpy(rng.uniform(-500, 500, 300_000).astype(np.float32) * np.float32(scale))
        s = torch.cat([x, y])
        codes, stats = _kernel(st, 0, s.cuda(), scale, False)
        want_codes, want = fp8.quantize(s.numpy(), np.float32(scale), False)
        assert np.array_equal(codes, want_codes)
        _same_stats(stats, want)


@pytest.mark.gpu
def test_quantize_full_layer_of_the_70b_shape(lib):
    """One Llama-2-70B layer's logits at batch 2 x seq 1024 (Table 8): 2 x 64 x 1024 x
    1024 bf16 values, in the launch configuration the benchmark times.  Statistics over
    every value; codes on a 2M-element sample."""
    n = 2 * 64 * 1024 * 1024
    s = gaussian_logits(n, 4242, sd=0.6, outlier_frac=1e-6, outlier=9.0, device="cuda")
    scale = 0.0125
    with gas.Fp8State(layers=80) as st:
        q, stats_t = st.quantize(17, s, torch.tensor([scale], device="cuda"))
        torch.cuda.synchronize()
        stats = gas.decode_fp8_stats(stats_t)[0]
    s_host = s.float().cpu().numpy()
    qs = fp8.scaled_logits(s_host, np.float32(scale))
    amax = np.float32(np.max(np.abs(s_host)))
    assert stats["count"] == n
    assert stats["amax"] == amax
    assert stats["max_scaled"] == np.float32(amax / np.float32(scale))
    assert stats["overflow"] == int(np.count_nonzero(np.abs(qs) > 448.0)) > 0
    idx = np.random.default_rng(9).integers(0, n, 2_000_000)
    assert np.array_equal(q.cpu().numpy()[idx], fp8.e4m3_encode(qs[idx]))


@pytest.mark.gpu
def test_delayed_scaling_history_and_auto_alpha(lib):
    """Nine steps on 5 layers with a 4-entry history and a 6-step burn-in: Eq. 1 scales,
    per-call statistics, the step maximum over several calls of a layer, a layer left
    out of a step (pushes 0), a NaN logit, the slack ratios of Eq. 16 and Algorithm 4."""
    L, H, T, n_q, d, d_h = 5, 4, 6, 3, 512, 64
    rng = np.random.default_rng(31)
    ds = fp8.DelayedScaling(L, H, 1.0)
    slack = []
    with gas.Fp8State(L, H, T) as st:
        for step in range(9):
            s_del = st.delayed_scales(0.9)
            torch.cuda.synchronize()
            want_s = ds.scales(0.9)
            got_s = s_del.cpu().numpy()
            assert np.array_equal(np.isnan(got_s), np.isnan(want_s))
            assert np.array_equal(got_s[~np.isnan(got_s)], want_s[~np.isnan(want_s)])
            amax = np.zeros(L, np.float32)
            for l in range(L):
                if step == 3 and l == 2:
                    continue  # no call: the layer pushes 0
                for part in range(1 + (l % 2)):  # odd layers: two calls merged into one step maximum
                    x = (rng.standard_normal(5000 + 37 * l) * (0.5 + step + l)).astype(np.float32)
                    if step == 5 and l == 4 and part == 0:
                        x[11] = np.nan
                    codes, stats = _kernel(st, l, torch.from_numpy(x).cuda(), float(got_s[l]), True)
                    want_codes, want = fp8.quantize(x, got_s[l], True)
                    assert np.array_equal(codes, want_codes)
                    _same_stats(stats, want)
                    amax[l] = fp8.nan_max([amax[l], np.float32(want["amax"])])
            sigma = rng.uniform(0.5, 4.0, (L, n_q)).astype(np.float32)
            st.end_step(torch.from_numpy(sigma).cuda(), d=d, d_h=d_h)
            ds.push(amax)
            if step < T:
                slack.append(fp8.slack_ratio(amax, sigma, d, d_h))
        assert st.slack_count() == T * L
        for q, kappa in [(0.9999, 1.0), (0.5, 2.0), (0.0, 1.0), (1.0, 3.0)]:
            a = st.auto_alpha(q, kappa)
            torch.cuda.synchronize()
            want = fp8.auto_alpha(np.concatenate(slack), q, kappa)
            assert float(a.item()) == pytest.approx(want, rel=1e-6)
        st.reset(1.0)
        s_del = st.delayed_scales(0.9)
        torch.cuda.synchronize()
        assert np.all(s_del.cpu().numpy() == np.float32(1.0) / np.float32(448 * 0.9))
        assert st.slack_count() == 0
        assert math.isnan(float(st.auto_alpha().item()))


@pytest.mark.gpu
def test_spike_reenactment_delayed_vs_geometry_aware(lib):
    """Appendix H on the GPT-2-small shape: 13 steps, W^Q and W^K multiplied by 4 from
    step 10 on; per step gas_refresh gives the geometry-aware scales (Eq. 15, alpha_min),
    the delayed comparator gives Eq. 1's, and the same logits (tokens uniform on the
    sqrt(d) sphere) are cast with both.  Every cast is checked against the oracle; the
    delayed run overflows on the spike step (largest scaled logit 16 * 0.9 * 448), the
    geometry-aware run never does and its scale follows sigma by 16x in the same step."""
    wl = get_workload("gpt2-small")
    wq, wk, _ = make_weights(wl, device="cuda")
    v = make_start_vectors(wl, device="cuda")
    x = sphere_tokens(1, 128, wl.d, 555, device="cuda")
    h = gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h)
    geo, dl = gas.Fp8State(wl.layers), gas.Fp8State(wl.layers)
    rows = []
    for step in range(13):
        f = 4.0 if step >= 10 else 1.0
        wqs = [w * f for w in wq]  # exact in bf16 (power of two)
        wks = [w * f for w in wk]
        sigma, s_geo, v = h.refresh(wqs, wks, wl.iters if step == 0 else 2, v)
        s_del = dl.delayed_scales(0.9)
        torch.cuda.synchronize()
        g_host, d_host = s_geo.cpu().numpy(), s_del.cpu().numpy()
        ov_geo = ov_del = 0
        mx_geo = mx_del = 0.0
        for l in range(wl.layers):
            S = attention_logits(wqs[l], wks[l], wl.n_q, wl.n_kv, wl.d_h, x)
            s_np = S.float().cpu().numpy()
            for state, scales, tag in ((geo, s_geo, "geo"), (dl, s_del, "del")):
                q, stats_t = state.quantize(l, S, scales[l:l + 1])
                torch.cuda.synchronize()
                got = gas.decode_fp8_stats(stats_t)[0]
                sc = (g_host if tag == "geo" else d_host)[l]
                want_codes, want = fp8.quantize(s_np, sc, True)
                assert np.array_equal(q.cpu().numpy().ravel(), want_codes)
                _same_stats(got, want)
                if tag == "geo":
                    ov_geo += got["overflow"] > 0
                    mx_geo = max(mx_geo, got["max_scaled"])
                else:
                    ov_del += got["overflow"] > 0
                    mx_del = max(mx_del, got["max_scaled"])
        geo.end_step()
        dl.end_step()
        rows.append((step, ov_del, mx_del, ov_geo, mx_geo, float(g_host.max())))
    for step, ov_del, mx_del, ov_geo, mx_geo, _ in rows:
        assert ov_geo == 0, rows
    assert rows[10][1] == wl.layers and rows[10][2] == pytest.approx(16 * 0.9 * 448, rel=2e-2)
    assert all(r[1] == 0 for r in rows[1:10]), rows        # steady weights: the history keeps up
    assert all(r[1] == 0 for r in rows[11:]), rows         # and catches up one step later
    assert rows[10][5] / rows[9][5] == pytest.approx(16.0, rel=2e-3)
    geo.close()
    dl.close()
    h.close()
