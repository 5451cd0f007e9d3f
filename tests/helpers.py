"""Small helpers shared by the tests (bf16 bit handling, seeded tiny draws)."""

import numpy as np
import torch


def to_bf16_bits(x) -> np.ndarray:
    """Round a float array to bf16 (RNE) and return the uint16 bit patterns."""
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def bits_to_f64(bits) -> np.ndarray:
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def tensor_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def sigma_k_closed_form(M: np.ndarray, v0: np.ndarray, k: int):
    """Exact k-step power-iteration estimate from a dense SVD of M.

    With v0/||v0|| = sum_i c_i v_i (right singular vectors), Algorithm 2 gives
    v_{k-1} ~ sum_i c_i s_i^{2(k-1)} v_i and sigma_k = ||M v_{k-1}||, i.e.
    sigma_k^2 = sum c_i^2 s_i^{4k-2} / sum c_i^2 s_i^{4k-4};  v_k ~ sum c_i s_i^{2k} v_i.
    """
    U, s, Vt = np.linalg.svd(M)
    c = Vt @ (v0 / np.linalg.norm(v0))
    r = s / s[0]
    num = np.sum(c ** 2 * r ** (4 * k - 2))
    den = np.sum(c ** 2 * r ** (4 * k - 4))
    sig = s[0] * np.sqrt(num / den)
    w = c * r ** (2 * k)
    v = Vt.T @ w
    v /= np.linalg.norm(v)
    return sig, v, s, Vt, U


def rand_head(rng, d, dh, scale=0.05, spike=None):
    a = rng.standard_normal((dh, d)) * scale
    b = rng.standard_normal((dh, d)) * scale
    if spike is not None:
        bq = rng.standard_normal(dh); bq /= np.linalg.norm(bq)
        x = rng.standard_normal(d); x /= np.linalg.norm(x)
        y = rng.standard_normal(d); y /= np.linalg.norm(y)
        a += spike[0] * np.outer(bq, x)
        b += spike[1] * np.outer(bq, y)
    return to_bf16_bits(a), to_bf16_bits(b)
