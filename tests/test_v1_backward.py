"""CPU checks of the v_out comparison used on heads whose start vector is nearly
orthogonal to the top right singular vector v_1 (tests/parity_utils.py,
assert_v_close_or_v1_backward): the oracle's own iterate from a start vector moved along
v_1 by a rounding-sized amount passes, with the perturbation recovered; a moved start
vector far beyond rounding, or a vector that is no such iterate, fails."""

import numpy as np
import pytest
import torch

import oracle
from synth import get_workload
from tests.helpers import tensor_bits
from tests.parity_utils import V1_BACKWARD_TOL, assert_v_close_or_v1_backward, top_right_singular


def _case(c1):
    wl = get_workload("tiny-mha").scaled(layers=1, n_q=1, n_kv=1, d=256, d_h=16, iters=30)
    rng = np.random.default_rng(7)
    # a planted spectrum with sigma_1 / sigma_2 = 1.3 (slow enough that a tiny start
    # component along v_1 still leaves a mixture after 30 iterations)
    U, _ = np.linalg.qr(rng.standard_normal((wl.d, wl.d_h)))
    V, _ = np.linalg.qr(rng.standard_normal((wl.d, wl.d_h)))
    P, _ = np.linalg.qr(rng.standard_normal((wl.d_h, wl.d_h)))
    s = 1.3 ** -np.arange(wl.d_h)
    A = (P * s) @ U.T            # A^T B = U diag(s) P^T P diag(1) V^T = U diag(s) V^T
    B = P @ V.T
    wq = [torch.from_numpy(A.astype(np.float32)).to(torch.bfloat16)]
    wk = [torch.from_numpy(B.astype(np.float32)).to(torch.bfloat16)]
    v1, S = top_right_singular(wq[0], wk[0], 0, wl)
    v0 = rng.standard_normal(wl.d)
    v0 /= np.linalg.norm(v0)
    v0 += (c1 - v1 @ v0) * v1                  # set the start vector's v_1 component
    v_in = torch.from_numpy(v0.astype(np.float32)).reshape(1, 1, wl.d)
    return wl, wq, wk, v_in, v1


def _oracle_v(wl, wq, wk, v0):
    _, v = oracle.power_iteration_factored(tensor_bits(wq[0]), tensor_bits(wk[0]), v0, wl.iters)
    return v


def test_rounding_sized_move_along_v1_is_accepted_and_recovered():
    wl, wq, wk, v_in, v1 = _case(3e-8)
    v0 = v_in.numpy().reshape(-1).astype(np.float64)
    c1 = float(v1 @ (v0 / np.linalg.norm(v0)))
    want = _oracle_v(wl, wq, wk, v0)
    for delta in (-8e-8, -2e-8, 5e-8):
        got = _oracle_v(wl, wq, wk, v0 / np.linalg.norm(v0) + delta * v1)
        assert np.linalg.norm(got - want) > 1e-3   # far apart: the comparison is needed
        worst, fitted = assert_v_close_or_v1_backward(got[None, None], want[None, None], wl, wq, wk, v_in)
        assert worst < 1e-6
        (_, _, c1_seen, d_fit), = fitted
        assert c1_seen == pytest.approx(c1, rel=1e-6)
        assert d_fit == pytest.approx(delta, rel=1e-3, abs=1e-12)


def test_large_move_or_wrong_vector_is_rejected():
    wl, wq, wk, v_in, v1 = _case(3e-8)
    v0 = v_in.numpy().reshape(-1).astype(np.float64)
    want = _oracle_v(wl, wq, wk, v0)
    far = _oracle_v(wl, wq, wk, v0 / np.linalg.norm(v0) + 10 * V1_BACKWARD_TOL * v1)
    with pytest.raises(AssertionError, match="fitted perturbation"):
        assert_v_close_or_v1_backward(far[None, None], want[None, None], wl, wq, wk, v_in)
    rng = np.random.default_rng(3)
    other = rng.standard_normal(wl.d)
    other /= np.linalg.norm(other)
    with pytest.raises(AssertionError):
        assert_v_close_or_v1_backward(other[None, None], want[None, None], wl, wq, wk, v_in)


def test_ordinary_heads_need_no_fit():
    wl, wq, wk, v_in, v1 = _case(0.3)
    v0 = v_in.numpy().reshape(-1).astype(np.float64)
    want = _oracle_v(wl, wq, wk, v0)
    worst, fitted = assert_v_close_or_v1_backward(want[None, None] + 1e-5, want[None, None], wl, wq, wk, v_in)
    assert fitted == [] and worst < 1e-3
