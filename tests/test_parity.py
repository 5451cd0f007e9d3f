"""GPU parity: the CUDA library against the float64 oracle on the same seeded inputs.

sigma and the per-layer scale must match within 1e-3 relative (at the same iteration
count and start vectors), v_out within 1e-3 Euclidean distance, and head / group
indexing exactly (one-hot weights).  Every back end is covered; every workload is
compared on every head (the transient refresh on every head of its cold start and spike
steps, on sampled layers elsewhere).
"""

import numpy as np
import pytest
import torch

from synth import get_workload, make_start_vectors
from tests.parity_utils import (V_ATOL, assert_sigma_close, assert_v_close, assert_v_close_or_v1_backward,
                                gpu_inputs, oracle_for, oracle_scales, run_library)

pytestmark = pytest.mark.gpu

METHODS = ["fused", "gram", "stream"]
SMALL = ["tiny-mha", "tiny-gqa", "tiny-gqa128", "ragged", "ragged128", "tiny-g16", "tiny-g32", "tiny-g64",
         "gpt2-small"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    import paper_2602_18851_gb300 as gas
    gas.build()
    gas.load()


@pytest.mark.parametrize("method", METHODS)
@pytest.mark.parametrize("name", SMALL)
def test_small_workloads_all_heads(name, method):
    wl = get_workload(name)
    torch.manual_seed(0)
    wq, wk, v_in, _ = gpu_inputs(wl)
    got = run_library(wl, wq, wk, v_in, method=method)
    sig, v = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(got["sigma"].ravel(), sig)
    assert_v_close(got["v_out"], v)
    s_ref = oracle_scales(wl, sig.reshape(wl.layers, wl.n_q))
    assert_sigma_close(got["s"], s_ref, what="scale")
    assert got["status"] == 0


@pytest.mark.parametrize("method", METHODS)
def test_gpt2_xl_all_heads(method):
    wl = get_workload("gpt2-xl")
    wq, wk, v_in, _ = gpu_inputs(wl)
    got = run_library(wl, wq, wk, v_in, method=method)
    sig, v = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(got["sigma"].ravel(), sig)
    assert_v_close(got["v_out"], v)
    assert_sigma_close(got["s"], oracle_scales(wl, sig.reshape(wl.layers, wl.n_q)), what="scale")


@pytest.mark.parametrize("method", METHODS)
def test_llama2_7b_planted_all_heads_and_closed_form(method):
    wl = get_workload("llama2-7b-planted")
    wq, wk, v_in, meta = gpu_inputs(wl)
    got = run_library(wl, wq, wk, v_in, method=method)
    sig, v = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(got["sigma"].ravel(), sig)
    assert_v_close(got["v_out"], v)
    # closed form: sigma_1 = s^Q_1 s^K_1 up to the Weyl bound of the bf16 rounding
    s_true = meta["sigma_planted"].numpy()
    weyl = (meta["err_q"] * meta["norm_k"] + meta["norm_q"] * meta["err_k"]
            + meta["err_q"] * meta["err_k"]).numpy()
    err = np.abs(got["sigma"] - s_true)
    assert np.all(err <= weyl + 1e-4 * s_true)


@pytest.mark.parametrize("method", METHODS)
def test_llama2_70b_gqa_all_heads(method):
    """Full 70B shape (80 layers, d 8192, 64/8 heads, d_h 128) at the workload's 30
    iterations on every back end, in the launch configuration the benchmark times.  The
    factored float64 oracle covers all 5120 heads (sigma, v_out and the 80 layer scales);
    the explicit-M oracle (M_h formed, d x d) checks the heads of one sampled layer."""
    wl = get_workload("llama2-70b-gqa")
    wq, wk, v_in, _ = gpu_inputs(wl)
    got = run_library(wl, wq, wk, v_in, method=method)
    sig, v = oracle_for(wl, wq, wk, v_in)
    ws = assert_sigma_close(got["sigma"].ravel(), sig)
    wv, fitted = assert_v_close_or_v1_backward(got["v_out"], v, wl, wq, wk, v_in)
    s_ref = oracle_scales(wl, sig.reshape(wl.layers, wl.n_q))
    wsc = assert_sigma_close(got["s"], s_ref, what="scale")
    assert got["status"] == 0
    print(f"70B {method}: all {wl.heads} heads, worst sigma rel err {ws:.2e}, v_out {wv:.2e}, "
          f"scale {wsc:.2e}; v_out from a start vector moved along v_1 (layer, head, c_1, delta): {fitted}")
    if method == "fused":
        pairs = [(79, h) for h in (0, 7, 8, 63)]
        sig_e, v_e = oracle_for(wl, wq, wk, v_in, pairs=pairs, mode="explicit")
        idx = [l * wl.n_q + h for l, h in pairs]
        np.testing.assert_allclose(sig_e, sig[idx], rtol=1e-12)
        np.testing.assert_allclose(v_e, v.reshape(-1, wl.d)[idx], atol=1e-10)
        assert_sigma_close(np.array([got["sigma"][l, h] for l, h in pairs]), sig_e)
    del wq, wk, v_in
    torch.cuda.empty_cache()


@pytest.mark.parametrize("method", METHODS)
@pytest.mark.parametrize("iters", [1, 2, 5])
def test_iteration_counts(method, iters):
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    got = run_library(wl, wq, wk, v_in, method=method, iters=iters)
    sig, v = oracle_for(wl, wq, wk, v_in, iters=iters)
    assert_sigma_close(got["sigma"].ravel(), sig)
    assert_v_close(got["v_out"], v)


@pytest.mark.parametrize("method", METHODS)
def test_unfused_scales_and_no_writeback(method):
    wl = get_workload("tiny-gqa")
    wq, wk, v_in, _ = gpu_inputs(wl)
    a = run_library(wl, wq, wk, v_in, method=method, fused=False, write_back=False)
    b = run_library(wl, wq, wk, v_in, method=method, fused=True, write_back=True)
    assert a["v_out"] is None
    np.testing.assert_array_equal(a["sigma"], b["sigma"])
    np.testing.assert_allclose(a["s"], b["s"], rtol=1e-6)


@pytest.mark.parametrize("method", METHODS)
def test_calibration_options(method):
    wl = get_workload("tiny-mha")
    wq, wk, v_in, _ = gpu_inputs(wl)
    sig, _ = oracle_for(wl, wq, wk, v_in)
    sig = sig.reshape(wl.layers, wl.n_q)
    for gamma, delta, rmax, ao in [(2.5, 1e-6, 448.0, 0.0), (0.0, 1e-3, 448.0, 0.0),
                                   (0.0, 1e-6, 57344.0, 0.0), (0.0, 1e-6, 448.0, 0.08)]:
        got = run_library(wl, wq, wk, v_in, method=method, gamma=gamma, delta=delta, r_max=rmax,
                          alpha_override=ao)
        ref = oracle_scales(wl, sig, gamma=gamma, delta=delta, r_max=rmax, alpha_override=ao)
        assert_sigma_close(got["s"], ref, what="scale")


@pytest.mark.parametrize("method", METHODS)
def test_one_hot_group_indexing_exact(method):
    """Only KV group g non-zero -> exactly the heads h with h // G == g have sigma > 0;
    only query head h non-zero -> exactly that head has sigma > 0."""
    import paper_2602_18851_gb300 as gas
    L, d, nq, nkv, dh = 2, 512, 8, 2, 128
    gen = torch.Generator(device="cuda").manual_seed(5)
    wq_full = [torch.randn(nq * dh, d, device="cuda", generator=gen).to(torch.bfloat16) for _ in range(L)]
    v_in = torch.randn(L, nq, d, device="cuda", generator=gen)
    with gas.Handle(L, d, nq, nkv, dh) as h:
        h.set_method(method)
        for g in range(nkv):
            wk = []
            for _ in range(L):
                w = torch.zeros(nkv * dh, d, device="cuda")
                w[g * dh:(g + 1) * dh] = torch.randn(dh, d, device="cuda", generator=gen)
                wk.append(w.to(torch.bfloat16))
            sigma, _ = h.spectral_norms(wq_full, wk, 3, v_in)
            nz = (sigma > 0).cpu().numpy()
            expect = np.zeros((L, nq), dtype=bool)
            expect[:, g * (nq // nkv):(g + 1) * (nq // nkv)] = True
            assert np.array_equal(nz, expect)
        wk_full = [torch.randn(nkv * dh, d, device="cuda", generator=gen).to(torch.bfloat16)
                   for _ in range(L)]
        for hq in [0, 3, 7]:
            wq = []
            for _ in range(L):
                w = torch.zeros(nq * dh, d, device="cuda")
                w[hq * dh:(hq + 1) * dh] = torch.randn(dh, d, device="cuda", generator=gen)
                wq.append(w.to(torch.bfloat16))
            sigma, v_out = h.spectral_norms(wq, wk_full, 3, v_in)
            nz = (sigma > 0).cpu().numpy()
            expect = np.zeros((L, nq), dtype=bool)
            expect[:, hq] = True
            assert np.array_equal(nz, expect)
            vo = v_out.cpu().numpy()
            assert np.all(vo[:, [x for x in range(nq) if x != hq]] == 0.0)


@pytest.mark.parametrize("method", METHODS)
def test_zero_start_vectors_and_inplace_warm_start(method):
    import paper_2602_18851_gb300 as gas
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    v_in[1, 3].zero_()
    v_in[0, 0].zero_()
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method(method)
        sig_ref, v_ref = oracle_for(wl, wq, wk, v_in, iters=4)
        v = v_in.clone()
        sigma, vo = h.spectral_norms(wq, wk, 4, v, v_out=v)  # v_out aliases v_in
        assert vo.data_ptr() == v.data_ptr()
        torch.cuda.synchronize()
        s = sigma.cpu().numpy()
        assert s[1, 3] == 0.0 and s[0, 0] == 0.0
        assert np.all(v[1, 3].cpu().numpy() == 0.0)
        assert_sigma_close(s.ravel(), sig_ref)
        assert_v_close(v.cpu().numpy(), v_ref)
        # warm start continues the iteration: 4 + 3 iterations == 7 from the start
        sigma2, _ = h.spectral_norms(wq, wk, 3, v, v_out=v)
        sig7, _ = oracle_for(wl, wq, wk, v_in, iters=7)
        assert_sigma_close(sigma2.cpu().numpy().ravel(), sig7, rtol=2e-3)


@pytest.mark.parametrize("method", METHODS)
@pytest.mark.parametrize("name", ["tiny-gqa128", "ragged"])
def test_start_vector_scale(name, method):
    """Algorithm 2 starts from v / ||v||: sigma and v_out do not depend on the scale of
    the start vectors.  Per-head scales from 2^-20 to 2^20 and non-powers of two, at
    k = 1 (where the first sigma is ||M v|| / ||v||), 2 and the workload's count: the
    library matches the oracle (which normalises first) and, to 1e-4, its own unscaled
    run."""
    wl = get_workload(name)
    wq, wk, v_in, _ = gpu_inputs(wl)
    gen = torch.Generator().manual_seed(7)
    exps = torch.randint(-20, 21, (wl.layers, wl.n_q), generator=gen).double()
    scale = torch.pow(2.0, exps)
    scale[0, 0], scale[-1, -1] = 3.7e-5, 1234.5
    v_scaled = (v_in.double().cpu() * scale[..., None]).float().to(v_in.device)
    for iters in (1, 2, wl.iters):
        base = run_library(wl, wq, wk, v_in, method=method, iters=iters)
        got = run_library(wl, wq, wk, v_scaled, method=method, iters=iters)
        sig, v = oracle_for(wl, wq, wk, v_scaled, iters=iters)
        assert_sigma_close(got["sigma"].ravel(), sig)
        assert_v_close(got["v_out"], v)
        # the 16-bit hi/lo operand of v rounds differently for non-power-of-two scales
        assert_sigma_close(got["sigma"].ravel(), base["sigma"].ravel(), rtol=1e-4, what="sigma vs unscaled")
        assert_v_close(got["v_out"], base["v_out"].reshape(-1, wl.d), atol=1e-4)
        assert got["status"] == 0


# v_out bound of the Gram back ends on the 512-layer case.  They iterate with G = A A^T,
# whose fp32 rounding is relative to ||A||^2: a finite-k iterate that still lies mostly in
# small singular directions (start vectors nearly orthogonal to the top singular vector,
# slow spectra) is perturbed by about eps * kappa^2 instead of the streaming back end's
# eps * kappa.  sigma, the method's output, stays within 1.5e-4 of the oracle there.
V_ATOL_GRAM_ILL = 1e-2


@pytest.mark.parametrize("method", METHODS)
def test_maximum_layer_count(method):
    """512 layers, the most one handle takes (one pointer table per launch): every head
    against the oracle, on a narrow shape (d 64, one 64-column chunk), at k = 6.  Among
    the 4096 heads a few converge slowly from start vectors nearly orthogonal to the top
    singular vector (component ~0.01, sigma_2/sigma_1 ~ 0.9)."""
    wl = get_workload("tiny-gqa").scaled(layers=512, d=64)
    wq, wk, v_in, _ = gpu_inputs(wl)
    got = run_library(wl, wq, wk, v_in, method=method, iters=6)
    sig, v = oracle_for(wl, wq, wk, v_in, iters=6)
    assert_sigma_close(got["sigma"].ravel(), sig)
    assert_v_close(got["v_out"], v, atol=V_ATOL if method == "stream" else V_ATOL_GRAM_ILL)
    assert_sigma_close(got["s"], oracle_scales(wl, sig.reshape(wl.layers, wl.n_q)), what="scale")
    assert got["status"] == 0


@pytest.mark.parametrize("method", METHODS)
def test_nonfinite_weights_flag_status(method):
    import paper_2602_18851_gb300 as gas
    wl = get_workload("tiny-gqa")
    wq, wk, v_in, _ = gpu_inputs(wl)
    wq[1][5, 7] = float("nan")
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method(method)
        sigma, s, _ = h.refresh(wq, wk, 3, v_in)
        torch.cuda.synchronize()
        st = h.device_status(clear=True)
        assert st & gas.GAS_DEV_NONFINITE_SIGMA
        assert torch.isnan(s[1]).item()
        assert torch.isfinite(s[0]).item()
        assert torch.isfinite(sigma[0]).all().item()
        assert h.device_status() == 0


@pytest.mark.parametrize("method", METHODS)
def test_deterministic_and_side_stream(method):
    import paper_2602_18851_gb300 as gas
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method(method)
        a, sa, va = h.refresh(wq, wk, wl.iters, v_in)
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            b, sb, vb = h.refresh(wq, wk, wl.iters, v_in, stream=side)
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        assert torch.equal(a, b) and torch.equal(sa, sb) and torch.equal(va, vb)


def test_methods_agree_with_each_other():
    wl = get_workload("gpt2-small")
    wq, wk, v_in, _ = gpu_inputs(wl)
    a = run_library(wl, wq, wk, v_in, method="gram")
    b = run_library(wl, wq, wk, v_in, method="stream")
    c = run_library(wl, wq, wk, v_in, method="fused")
    assert_sigma_close(a["sigma"].ravel(), b["sigma"].ravel(), rtol=1e-4)
    # the fused kernel runs the same fp32 recurrence as the separate iteration kernel
    assert_sigma_close(c["sigma"].ravel(), a["sigma"].ravel(), rtol=1e-5)


@pytest.mark.parametrize("which", [0, 1])
def test_bounded_wait_runs_out_and_context_stays_usable(which):
    """Failure detection on the device: a wait that nothing completes (an mbarrier phase,
    or a flag no kernel writes) gives up after the 2 s limit, sets the timeout bit of the
    status word and returns; the same handle then refreshes correctly."""
    import time
    import paper_2602_18851_gb300 as gas
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        assert h.device_status(clear=True) == 0
        t0 = time.perf_counter()
        h.selftest_wait_timeout(which)
        code = h.device_status(clear=True)      # synchronises: the kernel has returned
        waited = time.perf_counter() - t0
        assert code == gas.GAS_DEV_WAIT_TIMEOUT
        assert 1.5 < waited < 30.0, waited
        assert h.device_status() == 0           # cleared
        sigma, s, v_out = h.refresh(wq, wk, wl.iters, v_in)
        torch.cuda.synchronize()
        assert h.device_status() == 0
    sig, v = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(sigma.cpu().numpy().ravel(), sig)
    assert_v_close(v_out.cpu().numpy(), v)


def test_transient_refresh_tracks_oracle():
    """Llama-2-70B transient workload on a 4-layer slice: cold start of 30 iterations, then
    99 warm-started refreshes of 2 iterations while the weights take a seeded rank-8 step
    every call (spike of 5e-2 at steps 40-45).  Every step, on a sampled layer: sigma and
    the layer scale against the oracle run lock-step from the GPU's own start vectors
    (strict parity), and sigma against a free-running float64 trajectory that carries its
    own v from the first step (drift)."""
    from synth.gen import TransientWeights
    import paper_2602_18851_gb300 as gas
    import oracle
    from tests.helpers import tensor_bits
    wl = get_workload("llama2-70b-transient").scaled(layers=4)
    assert wl.steps == 100
    tw = TransientWeights(wl, device="cuda")
    v = make_start_vectors(wl, device="cuda")
    layer = 2
    v_free = v[layer:layer + 1].cpu().numpy().copy()
    pairs = [(0, hq) for hq in range(wl.n_q)]
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        for t in range(wl.steps):
            if t > 0:
                tw.step(t)
            iters = wl.cold_iters if t == 0 else wl.iters
            v_gpu_in = v[layer:layer + 1].cpu().numpy().copy()
            sigma, s, v = h.refresh(tw.wq, tw.wk, iters, v, v_out=v)
            qb = [tensor_bits(tw.wq[layer])]
            kb = [tensor_bits(tw.wk[layer])]
            sig_ls, _ = oracle.heads(wl.d, wl.n_q, wl.n_kv, wl.d_h, qb, kb, v_gpu_in, iters, pairs)
            sig_fr, vv = oracle.heads(wl.d, wl.n_q, wl.n_kv, wl.d_h, qb, kb, v_free, iters, pairs)
            v_free = vv.reshape(1, wl.n_q, wl.d).astype(np.float32)
            got = sigma[layer].cpu().numpy()
            assert_sigma_close(got, sig_ls, rtol=1e-3, what=f"sigma, step {t} (lock-step)")
            assert_sigma_close(got, sig_fr, rtol=1e-3, what=f"sigma, step {t} (free-running)")
            s_ref = oracle_scales(wl, sig_ls.reshape(1, wl.n_q), n_heads_total=wl.layers * wl.n_q)
            assert_sigma_close(s[layer:layer + 1].cpu().numpy(), s_ref, what=f"scale, step {t}")


def test_transient_refresh_full_size():
    """The same transient workload at its full size, in the launch configuration the
    benchmark times: all 80 layers of the Llama-2-70B GQA shape, 100 refreshes.  On the
    cold start (step 0) and on the spike steps 40-45 every head of every layer, on the other
    steps layers 0, 39 and 79 (all 64 heads each): sigma and the layer scales against the
    oracle run lock-step from the GPU's own start vectors.  The per-layer perturbations are
    seeded by (step, layer), so layers 0-3 also match the 4-layer slice above."""
    from synth.gen import TransientWeights
    import paper_2602_18851_gb300 as gas
    import oracle
    from tests.helpers import tensor_bits
    wl = get_workload("llama2-70b-transient")
    assert wl.layers == 80 and wl.steps == 100
    tw = TransientWeights(wl, device="cuda")
    v = make_start_vectors(wl, device="cuda")
    full_steps = {0, *range(40, 46)}
    worst = {"all": 0.0, "sample": 0.0}
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        for t in range(wl.steps):
            if t > 0:
                tw.step(t)
            iters = wl.cold_iters if t == 0 else wl.iters
            sample = list(range(wl.layers)) if t in full_steps else [0, 39, 79]
            pairs = [(i, hq) for i in range(len(sample)) for hq in range(wl.n_q)]
            v_gpu_in = v[sample].cpu().numpy()
            sigma, s, v = h.refresh(tw.wq, tw.wk, iters, v, v_out=v)
            qb = [tensor_bits(tw.wq[l]) for l in sample]
            kb = [tensor_bits(tw.wk[l]) for l in sample]
            sig, _ = oracle.heads(wl.d, wl.n_q, wl.n_kv, wl.d_h, qb, kb, v_gpu_in, iters, pairs,
                                  want_v=False)
            got = sigma[sample].cpu().numpy().ravel()
            key = "all" if t in full_steps else "sample"
            worst[key] = max(worst[key], assert_sigma_close(got, sig, rtol=1e-3, what=f"sigma, step {t}"))
            s_ref = oracle_scales(wl, sig.reshape(len(sample), wl.n_q), n_heads_total=wl.layers * wl.n_q)
            assert_sigma_close(s[sample].cpu().numpy(), s_ref, what=f"scale, step {t}")
        assert h.device_status(clear=True) == 0
    print(f"full-size transient: worst sigma rel err {worst['all']:.2e} on all heads of steps 0 and "
          f"40-45, {worst['sample']:.2e} on layers 0/39/79 of the other steps")


def test_bf16_inputs_unchanged():
    """The library never writes the weights or v_in (when v_out is separate)."""
    import paper_2602_18851_gb300 as gas
    wl = get_workload("tiny-gqa")
    wq, wk, v_in, _ = gpu_inputs(wl)
    cq = [w.clone() for w in wq]
    cv = v_in.clone()
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        for m in METHODS:
            h.set_method(m)
            h.refresh(wq, wk, 3, v_in)
    torch.cuda.synchronize()
    assert all(torch.equal(a, b) for a, b in zip(cq, wq))
    assert torch.equal(cv, v_in)

