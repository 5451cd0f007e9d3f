"""Strided weight layouts (gas_set_weight_layout): padded rows and per-head-interleaved
fused projections give exactly the results of the contiguous matrices, on every back
end and on the whole-layer path, and the padding (filled with NaN) is never read."""

import math

import numpy as np
import pytest
import torch

import paper_2602_18851_gb300 as gas
from synth import get_workload
from tests.parity_utils import SIGMA_RTOL, assert_sigma_close, gpu_inputs, oracle_for

pytestmark = pytest.mark.gpu

METHODS = ["fused", "gram", "stream"]


def _run(wl, wq, wk, v_in, method, layout=None, layer=False):
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method(method)
        if layout:
            h.set_weight_layout(**layout)
        if layer:
            sigma, s, v_out = h.layer_refresh(wq, wk, wl.iters, v_in[:, 0, :].contiguous())
        else:
            sigma, s, v_out = h.refresh(wq, wk, wl.iters, v_in)
        torch.cuda.synchronize()
        assert h.device_status(clear=True) == 0
        return sigma.cpu(), s.cpu(), v_out.cpu()


def _padded(ws, pad):
    """Each matrix inside a NaN-filled [rows, d + pad] buffer (row stride d + pad)."""
    out = []
    for w in ws:
        rows, d = w.shape
        big = torch.full((rows, d + pad), float("nan"), dtype=torch.bfloat16, device=w.device)
        big[:, :d] = w
        out.append(big)
    return out


def _interleaved(wq, wk, d_h):
    """MHA fused projection stored per head as [heads][3][d_h][d] (query, key, value
    blocks of a head next to each other); value blocks and nothing else are NaN."""
    qs, ks = [], []
    for q, k in zip(wq, wk):
        heads = q.shape[0] // d_h
        d = q.shape[1]
        buf = torch.full((heads, 3, d_h, d), float("nan"), dtype=torch.bfloat16, device=q.device)
        buf[:, 0] = q.view(heads, d_h, d)
        buf[:, 1] = k.view(heads, d_h, d)
        flat = buf.view(-1)
        qs.append(flat)
        ks.append(flat[d_h * d:])
    return qs, ks


def _same(a, b):
    for x, y in zip(a, b):
        assert torch.equal(x, y), (x.flatten()[:4], y.flatten()[:4])


@pytest.mark.parametrize("name", ["tiny-gqa128", "ragged128", "tiny-gqa", "tiny-dh80"])
@pytest.mark.parametrize("method", METHODS)
def test_padded_rows_match_contiguous(name, method):
    wl = get_workload(name)
    wq, wk, v_in, _ = gpu_inputs(wl)
    ref = _run(wl, wq, wk, v_in, method)
    pq, pk = _padded(wq, 24), _padded(wk, 40)
    got = _run(wl, pq, pk, v_in, method, layout=dict(ld_q=wl.d + 24, ld_k=wl.d + 40))
    _same(got, ref)


@pytest.mark.parametrize("name", ["tiny-mha", "ragged128", "gpt2-small"])
@pytest.mark.parametrize("method", METHODS)
def test_interleaved_fused_projection_matches_contiguous(name, method):
    wl = get_workload(name)
    assert wl.n_q == wl.n_kv
    wq, wk, v_in, _ = gpu_inputs(wl)
    ref = _run(wl, wq, wk, v_in, method)
    iq, ik = _interleaved(wq, wk, wl.d_h)
    hs = 3 * wl.d_h * wl.d
    got = _run(wl, iq, ik, v_in, method, layout=dict(head_stride_q=hs, head_stride_k=hs))
    _same(got, ref)
    # and against the oracle directly
    sig_ref, _ = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(got[0].double().numpy().ravel(), sig_ref.ravel(), rtol=SIGMA_RTOL)


def test_gqa_fused_block_projection_by_pointer_offsets():
    """[Q; K; V] stacked row blocks of one fused [(n_q + 2 n_kv) d_h, d] tensor need no
    layout call: Wq and Wk are row offsets into it."""
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    ref = _run(wl, wq, wk, v_in, "fused")
    fq, fk = [], []
    for q, k in zip(wq, wk):
        fused = torch.cat([q, k, torch.full_like(k, float("nan"))]).contiguous()
        fq.append(fused[: q.shape[0]])
        fk.append(fused[q.shape[0]: q.shape[0] + k.shape[0]])
    got = _run(wl, fq, fk, v_in, "fused")
    _same(got, ref)


def test_whole_layer_path_with_padded_rows():
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    ref = _run(wl, wq, wk, v_in, "fused", layer=True)
    got = _run(wl, _padded(wq, 8), _padded(wk, 16), v_in, "fused",
               layout=dict(ld_q=wl.d + 8, ld_k=wl.d + 16), layer=True)
    _same(got, ref)


def test_layout_argument_errors():
    wl = get_workload("tiny-gqa128")
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        lib = gas.load()
        assert lib.gas_set_weight_layout(h._h, 5, 0, 0, 0, 0) == gas.GAS_ERR_UNSUPPORTED
        assert lib.gas_set_weight_layout(h._h, 0, wl.d - 8, 0, 0, 0) == gas.GAS_ERR_INVALID_ARG
        assert lib.gas_set_weight_layout(h._h, 0, wl.d + 4, 0, 0, 0) == gas.GAS_ERR_INVALID_ARG
        assert lib.gas_set_weight_layout(h._h, 0, 0, 0, wl.d * wl.d_h - 8, 0) == gas.GAS_ERR_INVALID_ARG
        assert b"head strides" in lib.gas_last_error(h._h)
        assert lib.gas_set_weight_layout(h._h, 0, 0, 0, 0, 0) == gas.GAS_OK
        wq, wk, v_in, _ = gpu_inputs(wl)
        h.set_weight_layout(ld_q=wl.d + 64)
        with pytest.raises(ValueError):
            h.refresh(wq, wk, 2, v_in)  # the contiguous tensors do not cover the strided extent


def _conv1d(wq, wk, pad_cols):
    """GPT-2 Conv1D storage: one [d, n_q*d_h + n_kv*d_h + pad] tensor per layer holding
    W^Q (columns 0..), W^K (next columns) and NaN padding; output features contiguous."""
    qs, ks, ld = [], [], None
    for q, k in zip(wq, wk):
        rq, d = q.shape
        rk = k.shape[0]
        ld = rq + rk + pad_cols
        buf = torch.full((d, ld), float("nan"), dtype=q.dtype, device=q.device)
        buf[:, :rq] = q.t()
        buf[:, rq:rq + rk] = k.t()
        flat = buf.view(-1)
        qs.append(flat)
        ks.append(flat[rq:])
    return qs, ks, ld


@pytest.mark.parametrize("name", ["gpt2-small", "tiny-gqa128", "tiny-gqa", "ragged", "tiny-g32"])
@pytest.mark.parametrize("method", ["fused", "gram"])
def test_conv1d_layout_matches_oracle(name, method):
    """Transposed (Conv1D) weights run through MN-major tensor-core operands; sigma, the
    scales and v_out agree with the contiguous run and with the oracle."""
    wl = get_workload(name)
    wq, wk, v_in, _ = gpu_inputs(wl)
    ref = _run(wl, wq, wk, v_in, method)
    cq, ck, ld = _conv1d(wq, wk, pad_cols=8 * ((wl.n_kv * wl.d_h) // 8))
    got = _run(wl, cq, ck, v_in, method, layout=dict(ld_q=ld, ld_k=ld, layout="cols"))
    np.testing.assert_allclose(got[0].numpy(), ref[0].numpy(), rtol=1e-5)
    np.testing.assert_allclose(got[1].numpy(), ref[1].numpy(), rtol=1e-5)
    assert float((got[2] - ref[2]).norm(dim=-1).max()) < 1e-4
    sig_ref, _ = oracle_for(wl, wq, wk, v_in)
    assert_sigma_close(got[0].double().numpy().ravel(), sig_ref.ravel(), rtol=SIGMA_RTOL)


def test_conv1d_layout_rejected_by_streaming_and_whole_layer_paths():
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    cq, ck, ld = _conv1d(wq, wk, 0)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_weight_layout(ld_q=ld, ld_k=ld, layout="cols")
        h.set_method("stream")
        with pytest.raises(gas.GasError) as e:
            h.refresh(cq, ck, 2, v_in)
        assert e.value.status == gas.GAS_ERR_UNSUPPORTED
        with pytest.raises(gas.GasError):
            h.layer_refresh(cq, ck, 2, v_in[:, 0, :].contiguous())
        lib = gas.load()
        assert lib.gas_set_weight_layout(h._h, 1, wl.n_q * wl.d_h - 8, 0, 0, 0) == gas.GAS_ERR_INVALID_ARG
        assert lib.gas_set_weight_layout(h._h, 1, 0, 0, 2 * wl.d_h, 0) == gas.GAS_ERR_INVALID_ARG
