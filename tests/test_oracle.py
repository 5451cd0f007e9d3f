"""Pins for the float64 oracle against things other than itself: dense SVD (LAPACK)
closed forms, planted spectra, the paper's propositions, and explicit GQA expansion.

Chosen so a plausible slip in the oracle (dropped term, transposed operand, wrong
group index, wrong normalisation, off-by-one iteration) fails at least one test.
"""

import math

import numpy as np
import pytest
import torch

import oracle
from synth import get_workload, make_start_vectors, make_weights
from tests.helpers import bits_to_f64, rand_head, sigma_k_closed_form, tensor_bits, to_bf16_bits


def test_form_interaction_is_wq_wkT():
    """M = W^Q_h W^K_g^T (Eq. 4) against a numpy product of the widened bf16 blocks."""
    rng = np.random.default_rng(1)
    A, B = rand_head(rng, 96, 16)
    M = oracle.form_interaction(A, B)
    Wq, Wk = bits_to_f64(A).T, bits_to_f64(B).T          # d x d_h
    np.testing.assert_allclose(M, Wq @ Wk.T, rtol=1e-13, atol=1e-15)
    assert np.linalg.matrix_rank(M) <= 16                  # rank(M) <= d_h


@pytest.mark.parametrize("k", [1, 2, 3, 7, 20])
@pytest.mark.parametrize("mode", ["factored", "explicit"])
def test_sigma_k_matches_svd_closed_form(k, mode):
    """The finite-k estimate equals its SVD closed form (so iteration count, the
    reported sigma of the last iteration and the normalisations are pinned)."""
    rng = np.random.default_rng(100 + k)
    d, dh = 128, 16
    A, B = rand_head(rng, d, dh, spike=(1.5, 2.0))
    v0 = rng.standard_normal(d)
    M = bits_to_f64(A).T @ bits_to_f64(B)
    sig_ref, v_ref, *_ = sigma_k_closed_form(M, v0, k)
    if mode == "factored":
        sig, v = oracle.power_iteration_factored(A, B, v0, k)
    else:
        sig, v = oracle.power_iteration_dense(oracle.form_interaction(A, B), v0, k)
    assert sig == pytest.approx(sig_ref, rel=1e-11)
    np.testing.assert_allclose(v, v_ref, atol=1e-9)


def test_converges_to_sigma1_and_right_singular_vector():
    """k = 500 on a gapped spectrum: sigma -> sigma_1(M) (dense SVD) within 1e-10 and
    v -> +-top RIGHT singular vector (a transposed operand would give the left one)."""
    rng = np.random.default_rng(7)
    d, dh = 200, 32
    A, B = rand_head(rng, d, dh, spike=(2.0, 2.5))
    M = bits_to_f64(A).T @ bits_to_f64(B)
    U, s, Vt = np.linalg.svd(M)
    assert s[1] / s[0] < 0.9
    v0 = rng.standard_normal(d)
    sig, v = oracle.power_iteration_factored(A, B, v0, 500)
    assert sig == pytest.approx(s[0], rel=1e-10)
    assert abs(v @ Vt[0]) == pytest.approx(1.0, abs=1e-10)
    assert abs(v @ U[:, 0]) < 0.99
    # The same weights with the operands swapped are M^T: same sigma, left vector.
    sig_t, v_t = oracle.power_iteration_factored(B, A, v0, 500)
    assert sig_t == pytest.approx(s[0], rel=1e-10)
    assert abs(v_t @ U[:, 0]) == pytest.approx(1.0, abs=1e-10)


def test_explicit_and_factored_agree():
    rng = np.random.default_rng(3)
    d, dh = 160, 32
    A, B = rand_head(rng, d, dh)
    v0 = rng.standard_normal(d)
    s1, v1 = oracle.power_iteration_factored(A, B, v0, 25)
    s2, v2 = oracle.power_iteration_dense(oracle.form_interaction(A, B), v0, 25)
    assert s1 == pytest.approx(s2, rel=1e-12)
    np.testing.assert_allclose(v1, v2, atol=1e-11)


def test_sigma_monotone_in_k_and_below_sigma1():
    """||M v_{k-1}|| is non-decreasing in k and never exceeds sigma_1 (Section 4.1)."""
    rng = np.random.default_rng(11)
    d, dh = 128, 16
    A, B = rand_head(rng, d, dh)
    M = bits_to_f64(A).T @ bits_to_f64(B)
    s1 = np.linalg.svd(M, compute_uv=False)[0]
    v0 = rng.standard_normal(d)
    prev = 0.0
    for k in range(1, 30):
        sig, _ = oracle.power_iteration_factored(A, B, v0, k)
        assert sig >= prev * (1 - 1e-14)
        assert sig <= s1 * (1 + 1e-12)
        prev = sig


def test_corollary_tighter_and_equality_case():
    """Corollary 3.3: ||W^Q W^K^T|| <= ||W^Q|| ||W^K||, equality iff top right singular
    vectors coincide -- e.g. W^K = W^Q (M PSD, sigma = ||W^Q||^2)."""
    rng = np.random.default_rng(5)
    d, dh = 144, 16
    A, B = rand_head(rng, d, dh, spike=(1.0, 1.0))
    v0 = rng.standard_normal(d)
    sig, _ = oracle.power_iteration_factored(A, B, v0, 400)
    nq = np.linalg.norm(bits_to_f64(A), 2)
    nk = np.linalg.norm(bits_to_f64(B), 2)
    assert sig <= nq * nk * (1 + 1e-12)
    assert sig < 0.99 * nq * nk
    sig_eq, _ = oracle.power_iteration_factored(A, A, v0, 400)
    assert sig_eq == pytest.approx(nq * nq, rel=1e-10)


def test_interaction_bound_on_random_activations():
    """Proposition 3.2 / Eq. 7: max_ij |x_i^T M x_j|/sqrt(d_h) <= sigma * max_i ||x_i||^2/sqrt(d_h)
    for x uniform on sqrt(d) S^{d-1} (pre-LN tokens); and the naive bound is looser."""
    rng = np.random.default_rng(9)
    d, dh, L = 128, 16, 256
    A, B = rand_head(rng, d, dh, spike=(2.0, 2.0))
    sig, _ = oracle.power_iteration_factored(A, B, rng.standard_normal(d), 300)
    M = oracle.form_interaction(A, B)
    x = rng.standard_normal((L, d))
    x *= math.sqrt(d) / np.linalg.norm(x, axis=1, keepdims=True)
    S = x @ M @ x.T / math.sqrt(dh)
    bound = sig * np.max(np.sum(x * x, axis=1)) / math.sqrt(dh)
    assert np.max(np.abs(S)) <= bound * (1 + 1e-12)
    # The worst case is attained by the top singular pair scaled to the sphere.
    U, s, Vt = np.linalg.svd(M)
    xi, xj = math.sqrt(d) * U[:, 0], math.sqrt(d) * Vt[0]
    assert abs(xi @ M @ xj) / math.sqrt(dh) == pytest.approx(sig * d / math.sqrt(dh), rel=1e-9)


def test_homogeneity_exact():
    """sigma(cA, B) = |c| sigma(A, B); 4x on both gives 16x (Appendix H spike test)."""
    rng = np.random.default_rng(13)
    d, dh = 96, 16
    A, B = rand_head(rng, d, dh)
    v0 = rng.standard_normal(d)
    s, v = oracle.power_iteration_factored(A, B, v0, 9)
    A4 = to_bf16_bits(4.0 * bits_to_f64(A))
    B4 = to_bf16_bits(4.0 * bits_to_f64(B))
    An = to_bf16_bits(-2.0 * bits_to_f64(A))
    s16, v16 = oracle.power_iteration_factored(A4, B4, v0, 9)
    s2, _ = oracle.power_iteration_factored(An, B, v0, 9)
    assert s16 == pytest.approx(16.0 * s, rel=1e-14)
    assert s2 == pytest.approx(2.0 * s, rel=1e-14)
    np.testing.assert_allclose(v16, v, atol=1e-13)


def test_zero_guards():
    rng = np.random.default_rng(17)
    d, dh = 64, 16
    A, B = rand_head(rng, d, dh)
    s, v = oracle.power_iteration_factored(A, B, np.zeros(d), 5)
    assert s == 0.0 and not np.any(v)
    Z = np.zeros_like(A)
    s, v = oracle.power_iteration_factored(Z, B, rng.standard_normal(d), 5)
    assert s == 0.0 and not np.any(v)
    s, v = oracle.power_iteration_factored(A, Z, rng.standard_normal(d), 5)
    assert s == 0.0 and not np.any(v)


@pytest.mark.parametrize("n_q,n_kv", [(4, 4), (8, 2), (6, 3), (8, 1)])
def test_implicit_gqa_equals_explicit_expansion(n_q, n_kv):
    """Proposition 4.1 / Appendix F: Algorithm 3 with RepeatBlocks/SumGroups equals
    power iteration on M = W^Q W^K_exp^T formed from the expanded keys, and both
    equal the SVD closed form of that M."""
    rng = np.random.default_rng(20 + n_q * 10 + n_kv)
    d, dh, k = 96, 8, 6
    Wq = to_bf16_bits(rng.standard_normal((n_q * dh, d)) * 0.1)
    Wk = to_bf16_bits(rng.standard_normal((n_kv * dh, d)) * 0.1)
    v0 = rng.standard_normal(d)
    s_imp, v_imp = oracle.layer_implicit_gqa(Wq, Wk, n_q, n_kv, dh, v0, k)
    M = oracle.layer_form_expanded(Wq, Wk, n_q, n_kv, dh)
    s_exp, v_exp = oracle.power_iteration_dense(M, v0, k)
    assert s_imp == pytest.approx(s_exp, rel=1e-12)
    np.testing.assert_allclose(v_imp, v_exp, atol=1e-11)
    # independent construction of the expanded keys
    g = n_q // n_kv
    Wq_f, Wk_f = bits_to_f64(Wq), bits_to_f64(Wk)
    Wk_exp = np.concatenate([Wk_f[(h // g) * dh:(h // g + 1) * dh] for h in range(n_q)])
    M_ref = Wq_f.T @ Wk_exp
    np.testing.assert_allclose(M, M_ref, rtol=1e-12, atol=1e-14)
    s_ref, v_ref, *_ = sigma_k_closed_form(M_ref, v0, k)
    assert s_imp == pytest.approx(s_ref, rel=1e-10)


def test_whole_layer_is_sum_of_heads():
    """The whole-layer M of Algorithm 3 is the sum over heads of the per-head M_h."""
    rng = np.random.default_rng(31)
    n_q, n_kv, dh, d = 6, 2, 8, 64
    Wq = to_bf16_bits(rng.standard_normal((n_q * dh, d)))
    Wk = to_bf16_bits(rng.standard_normal((n_kv * dh, d)))
    M = oracle.layer_form_expanded(Wq, Wk, n_q, n_kv, dh)
    acc = np.zeros((d, d))
    for h in range(n_q):
        g = h // (n_q // n_kv)
        acc += oracle.form_interaction(Wq[h * dh:(h + 1) * dh], Wk[g * dh:(g + 1) * dh])
    np.testing.assert_allclose(M, acc, rtol=1e-12, atol=1e-12)


def test_heads_driver_group_map_one_hot():
    """Head h reads KV group h // (n_q/n_kv): with only group g non-zero, exactly the
    heads of group g have sigma > 0."""
    rng = np.random.default_rng(41)
    L, d, n_q, n_kv, dh = 2, 64, 8, 4, 16
    wq = [to_bf16_bits(rng.standard_normal((n_q * dh, d))) for _ in range(L)]
    v_in = rng.standard_normal((L, n_q, d)).astype(np.float32)
    for g in range(n_kv):
        wk = []
        for l in range(L):
            w = np.zeros((n_kv * dh, d), dtype=np.float32)
            w[g * dh:(g + 1) * dh] = rng.standard_normal((dh, d))
            wk.append(to_bf16_bits(w))
        sig, _ = oracle.spectral_norms(wq, wk, v_in, 3, n_q, n_kv, dh)
        nz = sig > 0
        expect = np.zeros((L, n_q), dtype=bool)
        expect[:, g * 2:(g + 1) * 2] = True
        assert np.array_equal(nz, expect)


def test_heads_driver_matches_single_head_calls():
    rng = np.random.default_rng(43)
    L, d, n_q, n_kv, dh = 2, 80, 4, 2, 16
    wq = [to_bf16_bits(rng.standard_normal((n_q * dh, d))) for _ in range(L)]
    wk = [to_bf16_bits(rng.standard_normal((n_kv * dh, d))) for _ in range(L)]
    v_in = rng.standard_normal((L, n_q, d)).astype(np.float32)
    sig, v = oracle.spectral_norms(wq, wk, v_in, 4, n_q, n_kv, dh, threads=2)
    for l in range(L):
        for h in range(n_q):
            g = h // 2
            s1, v1 = oracle.power_iteration_factored(wq[l][h * dh:(h + 1) * dh],
                                                     wk[l][g * dh:(g + 1) * dh],
                                                     v_in[l, h].astype(np.float64), 4)
            assert sig[l, h] == s1
            np.testing.assert_array_equal(v[l, h], v1)


def test_planted_spectrum_closed_form():
    """Planted weights (synth 'planted' recipe, small shape): sigma_k of the oracle is
    within the Weyl bound of the closed form s^Q_1 s^K_1 (rounding residual E):
    |dsigma| <= ||E_Q||_F ||B|| + ||A|| ||E_K||_F + ||E_Q||_F ||E_K||_F, plus the
    convergence term sigma_1 (sigma_2/sigma_1)^(2k-2) tan^2 (loose)."""
    wl = get_workload("llama2-7b-planted").scaled(layers=2, d=512, n_q=4, n_kv=4, d_h=64)
    wq, wk, meta = make_weights(wl, device="cpu")
    v_in = make_start_vectors(wl, device="cpu").numpy()
    sig, _ = oracle.spectral_norms([tensor_bits(w) for w in wq], [tensor_bits(w) for w in wk],
                                   v_in, wl.iters, wl.n_q, wl.n_kv, wl.d_h)
    s_true = meta["sigma_planted"].numpy()
    nq, nk = meta["norm_q"].numpy(), meta["norm_k"].numpy()
    eq, ek = meta["err_q"].numpy(), meta["err_k"].numpy()
    weyl = eq * nk + nq * ek + eq * ek
    conv = s_true * (2.0 ** -1.4) ** (2 * wl.iters - 2) * 1e4
    err = np.abs(sig - s_true)
    assert np.all(err <= weyl + conv), (err, weyl)
    assert np.all(err / s_true < 1e-2)


def test_tiny_workloads_run_and_are_finite():
    for name in ["tiny-mha", "tiny-gqa", "ragged"]:
        wl = get_workload(name)
        wq, wk, _ = make_weights(wl, device="cpu")
        v_in = make_start_vectors(wl, device="cpu").numpy()
        sig, v = oracle.spectral_norms([tensor_bits(w) for w in wq],
                                       [tensor_bits(w) for w in wk],
                                       v_in, wl.iters, wl.n_q, wl.n_kv, wl.d_h)
        assert np.all(np.isfinite(sig)) and np.all(sig > 0)
        np.testing.assert_allclose(np.linalg.norm(v, axis=-1), 1.0, rtol=1e-12)


def test_bf16_widening_exact():
    """The oracle widens bf16 exactly: a bf16 whose value is known reproduces it."""
    x = np.array([1.0, -2.5, 3.140625, 1e-30, 65280.0], dtype=np.float32)
    bits = to_bf16_bits(x)
    t = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(bits_to_f64(bits), t)


def test_weight_decoders_exact_for_every_pattern():
    """All 65536 bit patterns decode like numpy's binary16 and PyTorch's bfloat16."""
    allb = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    try:
        oracle.set_weight_format("f16")
        got = oracle.decode_weights(allb)
        want = allb.view(np.float16).astype(np.float64)
        assert np.array_equal(np.isnan(got), np.isnan(want))
        assert np.array_equal(got[~np.isnan(got)], want[~np.isnan(want)])
    finally:
        oracle.set_weight_format("bf16")
    got = oracle.decode_weights(allb)
    want = torch.from_numpy(allb.astype(np.int16)).view(torch.bfloat16).double().numpy()
    assert np.array_equal(got[~np.isnan(got)], want[~np.isnan(want)])


def test_f16_weights_match_svd_closed_form():
    """Algorithm 2 on binary16 weights equals the SVD closed form of the exactly
    decoded matrices (the bits are not reinterpreted as bf16)."""
    rng = np.random.default_rng(16)
    d, dh, k = 96, 8, 9
    a = (rng.standard_normal((dh, d)) * 0.3).astype(np.float16)
    b = (rng.standard_normal((dh, d)) * 0.3).astype(np.float16)
    v0 = rng.standard_normal(d)
    M = a.astype(np.float64).T @ b.astype(np.float64)
    want, _, _, _, _ = sigma_k_closed_form(M, v0, k)
    try:
        oracle.set_weight_format("f16")
        sig, _ = oracle.power_iteration_factored(a.view(np.uint16), b.view(np.uint16), v0, k)
    finally:
        oracle.set_weight_format("bf16")
    assert sig == pytest.approx(want, rel=1e-10)
