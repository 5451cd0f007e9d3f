"""The oracle's two forms of Algorithm 2 agree at the head sizes of the real workloads.

``mode="explicit"`` forms M_h = W^Q_h W^K_g^T (d x d, float64) and power-iterates it;
``mode="factored"`` applies M_h as W^Q_h (W^K_g^T v) and W^K_g (W^Q_h^T u) (Section 4.1).
The definition of the method is the explicit one (Appendix E.1); the factored form is
what covers every head of the large workloads, so the two are compared here on heads of
the GPT-2 XL (d 1600, d_h 64), Llama-2-7B (d 4096, d_h 128) and Llama-2-70B GQA
(d 8192, d_h 128, 8 query heads per KV head) shapes at those workloads' iteration counts
and start vectors.  Agreement is to rounding (1e-12 on sigma, 1e-10 on v_out).
"""

import numpy as np
import pytest

import oracle
from synth import get_workload, make_start_vectors, make_weights
from synth.gen import bf16_bits


@pytest.mark.parametrize("name,heads", [
    ("gpt2-xl", [0, 13, 24]),
    ("llama2-7b-planted", [0, 31]),
    ("llama2-70b-gqa", [0, 63]),
])
def test_explicit_equals_factored_at_real_head_size(name, heads):
    wl = get_workload(name).scaled(layers=1)
    wq, wk, _ = make_weights(wl)
    v_in = make_start_vectors(wl).numpy()
    qb, kb = [bf16_bits(wq[0])], [bf16_bits(wk[0])]
    pairs = [(0, h) for h in heads]
    s_f, v_f = oracle.heads(wl.d, wl.n_q, wl.n_kv, wl.d_h, qb, kb, v_in, wl.iters, pairs, mode="factored")
    s_e, v_e = oracle.heads(wl.d, wl.n_q, wl.n_kv, wl.d_h, qb, kb, v_in, wl.iters, pairs, mode="explicit")
    assert np.all(s_f > 0)
    np.testing.assert_allclose(s_e, s_f, rtol=1e-12)
    np.testing.assert_allclose(v_e, v_f, atol=1e-10)
