"""Head widths outside {64, 128} (80, 96, 256) and fp32 weights against the oracle (and,
for fp32 values that bf16 cannot hold, against the dense-SVD closed form of the finite-k
estimate).  d_h 80 and 96 run on every back end (the tensor-core ones place a head in a
128-row tile whose remaining rows are zero); d_h 256 and fp32 weights run on the
streaming back end and the whole-layer path, and the tensor-core back ends refuse them
cleanly."""

import numpy as np
import pytest
import torch

import oracle
import paper_2602_18851_gb300 as gas
from synth import get_workload, make_start_vectors, make_weights
from tests.helpers import sigma_k_closed_form, tensor_bits
from tests.parity_utils import (SIGMA_RTOL, V_ATOL, assert_sigma_close, assert_v_close, gpu_inputs, oracle_for,
                                oracle_scales)

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("method", ["auto", "fused", "gram", "stream"])
@pytest.mark.parametrize("name", ["tiny-dh80", "tiny-dh96", "tiny-dh256"])
def test_other_head_widths_match_oracle(name, method):
    wl = get_workload(name)
    wq, wk, v_in, _ = gpu_inputs(wl)
    tensor_cores = wl.d_h in (80, 96)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method(method)
        if method in ("fused", "gram") and not tensor_cores:
            with pytest.raises(gas.GasError) as e:
                h.refresh(wq, wk, 2, v_in)
            assert e.value.status == gas.GAS_ERR_UNSUPPORTED
            return
        sigma, s, v_out = h.refresh(wq, wk, wl.iters, v_in)
        torch.cuda.synchronize()
        assert h.device_status(clear=True) == 0
        if method == "auto":  # AUTO picks the fused tensor-core back end where it applies
            assert h.last_launch_names()[0].startswith("gram_fused" if tensor_cores else "stream")
    sig_ref, v_ref = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(sigma.double().cpu().numpy().ravel(), sig_ref.ravel(), rtol=SIGMA_RTOL)
    assert_v_close(v_out.cpu().numpy().reshape(-1, wl.d), v_ref.reshape(-1, wl.d), atol=V_ATOL)
    np.testing.assert_allclose(s.double().cpu().numpy(), oracle_scales(wl, sig_ref.reshape(wl.layers, wl.n_q)),
                               rtol=1e-3)


def test_conv1d_layout_needs_whole_head_tiles():
    """Conv1D weights are read as 64-row boxes of whole heads: with d_h 80 the tensor-core
    back ends refuse them, and so does the streaming back end (nn.Linear layout only)."""
    wl = get_workload("tiny-dh80")
    rows = wl.n_q * wl.d_h + wl.n_kv * wl.d_h
    buf = torch.zeros(wl.layers, wl.d, rows, dtype=torch.bfloat16, device="cuda")
    cq = [buf[l].view(-1) for l in range(wl.layers)]
    ck = [buf[l].view(-1)[wl.n_q * wl.d_h:] for l in range(wl.layers)]
    v_in = make_start_vectors(wl, device="cuda")
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_weight_layout(ld_q=rows, ld_k=rows, layout="cols")
        for m in ("auto", "fused", "gram", "stream"):
            h.set_method(m)
            with pytest.raises(gas.GasError) as e:
                h.refresh(cq, ck, 2, v_in)
            assert e.value.status == gas.GAS_ERR_UNSUPPORTED


@pytest.mark.parametrize("name", ["tiny-dh96", "tiny-dh256"])
def test_other_head_widths_whole_layer(name):
    wl = get_workload(name)
    wq, wk, v_in, _ = gpu_inputs(wl)
    v1 = v_in[:, 0, :].contiguous()
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        sigma, _, _ = h.layer_refresh(wq, wk, wl.iters, v1)
        torch.cuda.synchronize()
    for l in range(wl.layers):
        want, _ = oracle.layer_implicit_gqa(tensor_bits(wq[l]), tensor_bits(wk[l]), wl.n_q, wl.n_kv, wl.d_h,
                                            v1[l].double().cpu().numpy(), wl.iters)
        assert float(sigma[l]) == pytest.approx(want, rel=SIGMA_RTOL)


@pytest.mark.parametrize("name", ["tiny-gqa128", "tiny-dh80", "ragged"])
def test_fp32_weights_holding_bf16_values_match_oracle(name):
    """fp32 tensors whose values are exactly the bf16 weights: the fp32 code path must
    give the oracle's result on those bf16 bits."""
    wl = get_workload(name)
    wq, wk, v_in, _ = gpu_inputs(wl)
    fq, fk = [w.float() for w in wq], [w.float() for w in wk]
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_weight_dtype("f32")
        sigma, s, v_out = h.refresh(fq, fk, wl.iters, v_in)
        torch.cuda.synchronize()
        h.set_method("fused")
        with pytest.raises(gas.GasError) as e:
            h.refresh(fq, fk, 2, v_in)
        assert e.value.status == gas.GAS_ERR_UNSUPPORTED
    sig_ref, v_ref = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(sigma.double().cpu().numpy().ravel(), sig_ref.ravel(), rtol=SIGMA_RTOL)
    assert_v_close(v_out.cpu().numpy().reshape(-1, wl.d), v_ref.reshape(-1, wl.d), atol=V_ATOL)


def test_fp32_weights_match_svd_closed_form():
    """Genuine fp32 weights (not representable in bf16): sigma after k iterations equals
    the dense-SVD closed form of the finite-k estimate, per head."""
    rng = np.random.default_rng(32)
    L, d, n_q, n_kv, d_h, k = 2, 256, 4, 2, 64, 6
    wq = [torch.from_numpy(rng.standard_normal((n_q * d_h, d)).astype(np.float32) * 0.05).cuda() for _ in range(L)]
    wk = [torch.from_numpy(rng.standard_normal((n_kv * d_h, d)).astype(np.float32) * 0.05).cuda() for _ in range(L)]
    v_in = torch.from_numpy(rng.standard_normal((L, n_q, d)).astype(np.float32)).cuda()
    with gas.Handle(L, d, n_q, n_kv, d_h) as h:
        h.set_weight_dtype(torch.float32)
        sigma, _, _ = h.refresh(wq, wk, k, v_in)
        torch.cuda.synchronize()
    G = n_q // n_kv
    for l in range(L):
        A_all = wq[l].double().cpu().numpy()
        B_all = wk[l].double().cpu().numpy()
        for hq in range(n_q):
            A = A_all[hq * d_h:(hq + 1) * d_h]
            B = B_all[(hq // G) * d_h:(hq // G + 1) * d_h]
            want, _, _, _, _ = sigma_k_closed_form(A.T @ B, v_in[l, hq].double().cpu().numpy(), k)
            assert float(sigma[l, hq]) == pytest.approx(want, rel=SIGMA_RTOL)


def test_fp32_whole_layer_path():
    wl = get_workload("tiny-dh96")
    wq, wk, v_in, _ = gpu_inputs(wl)
    v1 = v_in[:, 0, :].contiguous()
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_weight_dtype("f32")
        sigma, _, _ = h.layer_refresh([w.float() for w in wq], [w.float() for w in wk], wl.iters, v1)
        torch.cuda.synchronize()
    for l in range(wl.layers):
        want, _ = oracle.layer_implicit_gqa(tensor_bits(wq[l]), tensor_bits(wk[l]), wl.n_q, wl.n_kv, wl.d_h,
                                            v1[l].double().cpu().numpy(), wl.iters)
        assert float(sigma[l]) == pytest.approx(want, rel=SIGMA_RTOL)


def test_fp32_rejects_head_width_256():
    wl = get_workload("tiny-dh256")
    wq, wk, v_in, _ = gpu_inputs(wl)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_weight_dtype("f32")
        with pytest.raises(gas.GasError) as e:
            h.refresh([w.float() for w in wq], [w.float() for w in wk], 2, v_in)
        assert e.value.status == gas.GAS_ERR_UNSUPPORTED
