"""GPU parity of the whole-layer sigma (Section 4.2: one v per layer, M = W^Q W^K_exp^T
over all heads) against the float64 oracle's Algorithm 3."""

import numpy as np
import pytest
import torch

import oracle
from oracle import calib
from synth import get_workload, make_weights
from tests.helpers import tensor_bits
from tests.parity_utils import SIGMA_RTOL, V_ATOL, assert_sigma_close

pytestmark = pytest.mark.gpu


def _layer_inputs(wl, seed=11):
    wq, wk, _ = make_weights(wl, device="cuda")
    gen = torch.Generator(device="cuda").manual_seed(seed)
    v = torch.randn(wl.layers, wl.d, device="cuda", generator=gen)
    return wq, wk, v


def _oracle(wl, wq, wk, v, iters, layers=None):
    layers = range(wl.layers) if layers is None else layers
    sig, vo = [], []
    for l in layers:
        s, vv = oracle.layer_implicit_gqa(tensor_bits(wq[l]), tensor_bits(wk[l]), wl.n_q, wl.n_kv, wl.d_h,
                                          v[l].double().cpu().numpy(), iters)
        sig.append(s)
        vo.append(vv)
    return np.array(sig), np.array(vo)


@pytest.mark.parametrize("name", ["tiny-mha", "tiny-gqa", "tiny-gqa128", "ragged", "tiny-g32", "gpt2-small"])
def test_layer_sigma_matches_algorithm3(name):
    import paper_2602_18851_gb300 as gas
    wl = get_workload(name)
    wq, wk, v = _layer_inputs(wl)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        sigma, s, v_out = h.layer_refresh(wq, wk, wl.iters, v)
        torch.cuda.synchronize()
        assert h.device_status(clear=True) == 0
    ref_s, ref_v = _oracle(wl, wq, wk, v, wl.iters)
    assert_sigma_close(sigma.double().cpu().numpy(), ref_s)
    dist = np.linalg.norm(v_out.double().cpu().numpy() - ref_v, axis=1).max()
    assert dist <= V_ATOL
    g = calib.gamma_min(wl.d_h, wl.layers * wl.n_q, 1024, 1e-6)
    a = calib.alpha_min(g, wl.d, wl.d_h, wl.layers * wl.n_q, 1024, 1e-6)
    s_ref = calib.scale_from_sigma(ref_s, a, wl.d, wl.d_h, 0.8, 448.0)
    assert_sigma_close(s.double().cpu().numpy(), s_ref, rtol=SIGMA_RTOL, what="scale")


def test_layer_sigma_70b_sampled():
    """Llama-2-70B shape, 4 iterations; oracle on two layers."""
    import paper_2602_18851_gb300 as gas
    wl = get_workload("llama2-70b-gqa")
    wq, wk, v = _layer_inputs(wl)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        sigma, _, v_out = h.layer_refresh(wq, wk, 4, v, with_scales=False)
        torch.cuda.synchronize()
    layers = [0, 79]
    ref_s, ref_v = _oracle(wl, wq, wk, v, 4, layers)
    assert_sigma_close(sigma.double().cpu().numpy()[layers], ref_s)
    assert np.linalg.norm(v_out.double().cpu().numpy()[layers] - ref_v, axis=1).max() <= V_ATOL


def test_layer_sigma_bounds_per_head_sigmas():
    """||sum_h M_h|| <= sum_h ||M_h|| and, with one non-zero head, equals it."""
    import paper_2602_18851_gb300 as gas
    wl = get_workload("tiny-gqa128")
    wq, wk, v = _layer_inputs(wl)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        sig_layer, _, _ = h.layer_refresh(wq, wk, 200, v, with_scales=False)
        vh = v[:, None, :].expand(wl.layers, wl.n_q, wl.d).contiguous()
        sig_heads, _ = h.spectral_norms(wq, wk, 200, vh)
        torch.cuda.synchronize()
        assert torch.all(sig_layer <= sig_heads.sum(1) * (1 + 1e-5))
        one = [w.clone() for w in wq]
        for w in one:
            w[wl.d_h:] = 0
        s1, _, _ = h.layer_refresh(one, wk, 200, v, with_scales=False)
        vh1, _ = h.spectral_norms(one, wk, 200, vh)
        torch.cuda.synchronize()
        np.testing.assert_allclose(s1.cpu().numpy(), vh1[:, 0].cpu().numpy(), rtol=1e-4)


def test_layer_zero_start_vector():
    import paper_2602_18851_gb300 as gas
    wl = get_workload("tiny-gqa")
    wq, wk, v = _layer_inputs(wl)
    v[1].zero_()
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        sigma, _, v_out = h.layer_refresh(wq, wk, 5, v, with_scales=False)
        torch.cuda.synchronize()
    assert sigma[1].item() == 0.0
    assert torch.all(v_out[1] == 0).item()
    assert sigma[0].item() > 0
