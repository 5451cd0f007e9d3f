"""Binary16 weights (gas_set_weight_dtype): every back end and the whole-layer path
against the oracle reading the same binary16 bits, and a strided fp16 layout."""

import numpy as np
import pytest
import torch

import oracle
import paper_2602_18851_gb300 as gas
from synth import get_workload, make_start_vectors, make_weights
from tests.parity_utils import (SIGMA_RTOL, V_ATOL, assert_sigma_close, assert_v_close, oracle_for,
                                oracle_scales)
from tests.helpers import tensor_bits

pytestmark = pytest.mark.gpu


@pytest.fixture
def f16_oracle():
    oracle.set_weight_format("f16")
    yield
    oracle.set_weight_format("bf16")


def _inputs(wl):
    wq, wk, _ = make_weights(wl, device="cuda", dtype=torch.float16)
    return wq, wk, make_start_vectors(wl, device="cuda")


@pytest.mark.parametrize("name", ["tiny-gqa128", "tiny-gqa", "ragged128", "gpt2-small", "tiny-g32", "tiny-dh96"])
@pytest.mark.parametrize("method", ["fused", "gram", "stream"])
def test_f16_weights_match_oracle(f16_oracle, name, method):
    wl = get_workload(name)
    wq, wk, v_in = _inputs(wl)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method(method)
        h.set_weight_dtype("f16")
        sigma, s, v_out = h.refresh(wq, wk, wl.iters, v_in)
        torch.cuda.synchronize()
        assert h.device_status(clear=True) == 0
    sig_ref, v_ref = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(sigma.double().cpu().numpy().ravel(), sig_ref.ravel(), rtol=SIGMA_RTOL)
    assert_v_close(v_out.cpu().numpy().reshape(-1, wl.d), v_ref.reshape(-1, wl.d), atol=V_ATOL)
    s_ref = oracle_scales(wl, sig_ref.reshape(wl.layers, wl.n_q))
    np.testing.assert_allclose(s.double().cpu().numpy(), s_ref, rtol=1e-3)


def test_f16_whole_layer_matches_oracle(f16_oracle):
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in = _inputs(wl)
    v1 = v_in[:, 0, :].contiguous()
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_weight_dtype("f16")
        sigma, _, _ = h.layer_refresh(wq, wk, wl.iters, v1)
        torch.cuda.synchronize()
    for l in range(wl.layers):
        want, _ = oracle.layer_implicit_gqa(tensor_bits(wq[l]), tensor_bits(wk[l]), wl.n_q, wl.n_kv, wl.d_h,
                                            v1[l].double().cpu().numpy(), wl.iters)
        assert float(sigma[l]) == pytest.approx(want, rel=SIGMA_RTOL)


def test_f16_padded_rows_match_contiguous():
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in = _inputs(wl)
    outs = []
    for pad in (0, 32):
        with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
            h.set_weight_dtype(torch.float16)
            qs, ks = wq, wk
            if pad:
                qs = [torch.nn.functional.pad(w, (0, pad), value=float("nan")) for w in wq]
                ks = [torch.nn.functional.pad(w, (0, pad), value=float("nan")) for w in wk]
                h.set_weight_layout(ld_q=wl.d + pad, ld_k=wl.d + pad)
            sigma, s, v_out = h.refresh(qs, ks, wl.iters, v_in)
            torch.cuda.synchronize()
            outs.append((sigma.cpu(), s.cpu(), v_out.cpu()))
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_weight_dtype_errors():
    wl = get_workload("tiny-gqa128")
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        lib = gas.load()
        assert lib.gas_set_weight_dtype(h._h, 7) == gas.GAS_ERR_INVALID_ARG
        assert lib.gas_set_weight_dtype(h._h, gas.GAS_DTYPE_BF16) == gas.GAS_OK
        wq, wk, v_in = _inputs(wl)
        with pytest.raises(ValueError):
            h.refresh(wq, wk, 2, v_in)  # binary16 tensors on a bf16 handle
