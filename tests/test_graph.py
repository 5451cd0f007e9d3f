"""gas_refresh inside a CUDA graph: once the handle has seen the weight pointers (the
first call uploads their TMA descriptors), a refresh is stream-ordered work with no
host synchronisation, so it can be captured and replayed.  Replays must reproduce the
direct call, and must see weights changed in place between replays (the fused kernel's
key-tile flags take a fresh value on every replay)."""

import pytest
import torch

import paper_2602_18851_gb300 as gas
from synth import get_workload
from tests.parity_utils import SIGMA_RTOL, assert_sigma_close, gpu_inputs, oracle_for

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("method", ["fused", "gram", "stream"])
def test_refresh_replays_in_a_cuda_graph(method):
    wl = get_workload("tiny-gqa128")
    wq, wk, v_in, _ = gpu_inputs(wl)
    sigma = torch.empty(wl.layers, wl.n_q, device="cuda")
    s = torch.empty(wl.layers, device="cuda")
    v_out = torch.empty_like(v_in)
    with gas.Handle(wl.layers, wl.d, wl.n_q, wl.n_kv, wl.d_h) as h:
        h.set_method(method)
        h.refresh(wq, wk, wl.iters, v_in, v_out=v_out, sigma=sigma, s=s)
        torch.cuda.synchronize()
        ref = [t.clone() for t in (sigma, s, v_out)]
        graph = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.graph(graph, stream=side):
            h.refresh(wq, wk, wl.iters, v_in, v_out=v_out, sigma=sigma, s=s)
        for t in (sigma, s, v_out):
            t.zero_()
        for _ in range(3):
            graph.replay()
        torch.cuda.synchronize()
        for a, b in zip((sigma, s, v_out), ref):
            assert torch.equal(a, b)
        # scale the weights in place: the replay must recompute from the new values
        for w in wq + wk:
            w.mul_(2.0)  # exact in bf16
        graph.replay()
        torch.cuda.synchronize()
        assert h.device_status(clear=True) == 0
        torch.testing.assert_close(sigma, 4.0 * ref[0], rtol=1e-6, atol=0)
        sig_ref, _ = oracle_for(wl, wq, wk, v_in)
        assert_sigma_close(sigma.double().cpu().numpy().ravel(), sig_ref.ravel(), rtol=SIGMA_RTOL)
