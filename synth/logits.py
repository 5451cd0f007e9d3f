"""Seeded attention logits for the consumer of the scales (E4M3 cast, delayed scaling).

Two recipes, both inputs only (no scale, no quantisation, no statistic is computed
here):

* ``gaussian_logits``  iid N(0, sd^2) logits with a seeded fraction of planted
                       outliers of magnitude `outlier` (random signs), in bf16 or fp32.
* ``attention_logits`` the logits of one layer, S = Q K^T / sqrt(d_h) with
                       Q = X W^Q_h, K = X W^K_{g(h)} (Algorithm 1, Stage 3) for seeded
                       tokens X drawn uniformly on the sphere of radius sqrt(d): the
                       post-LayerNorm model of the inputs in Proposition 3.2.  Computed
                       in fp32 from the bf16 weights, returned as [batch, n_q, T, T].
* ``special_logits``   a fixed list of edge values (signed zeros, infinities, NaN,
                       values whose quotient by `scale` lands on E4M3 rounding midpoints
                       and their float32 neighbours, values just below and above the
                       448 boundary) for the parity tests.
"""

from __future__ import annotations

import math
from typing import Sequence

import numpy as np
import torch

from .gen import _gen


def gaussian_logits(n: int, seed: int, sd: float = 1.0, outlier_frac: float = 0.0, outlier: float = 0.0,
                    dtype=torch.bfloat16, device="cpu") -> torch.Tensor:
    g = _gen(device, seed)
    x = torch.randn(n, generator=g, device=device, dtype=torch.float32) * sd
    if outlier_frac > 0.0 and n > 0:
        k = max(1, int(n * outlier_frac))
        idx = torch.randint(0, n, (k,), generator=g, device=device)
        sign = torch.randint(0, 2, (k,), generator=g, device=device).float() * 2 - 1
        x[idx] = sign * outlier
    return x.to(dtype)


def sphere_tokens(batch: int, tokens: int, d: int, seed: int, device="cpu") -> torch.Tensor:
    """[batch, tokens, d] fp32, each row uniform on the sphere of radius sqrt(d)."""
    g = _gen(device, seed)
    x = torch.randn(batch, tokens, d, generator=g, device=device, dtype=torch.float32)
    return x * (math.sqrt(d) / x.norm(dim=-1, keepdim=True))


def attention_logits(wq: torch.Tensor, wk: torch.Tensor, n_q: int, n_kv: int, d_h: int, x: torch.Tensor,
                     weight_scale: float = 1.0, out_dtype=torch.bfloat16) -> torch.Tensor:
    """S[b, h, i, j] = (x_i A_h^T) . (x_j B_{g(h)}^T) / sqrt(d_h) for one layer, with
    A_h, B_g the rows of the nn.Linear weights (times `weight_scale`)."""
    b, t, d = x.shape
    q = (x.reshape(b * t, d) @ wq.float().t()).reshape(b, t, n_q, d_h).permute(0, 2, 1, 3)
    k = (x.reshape(b * t, d) @ wk.float().t()).reshape(b, t, n_kv, d_h).permute(0, 2, 1, 3)
    k = k.repeat_interleave(n_q // n_kv, dim=1)
    s = (q @ k.transpose(-1, -2)) * (weight_scale * weight_scale / math.sqrt(d_h))
    return s.to(out_dtype).contiguous()


def special_logits(scale: float, mids: Sequence[float]) -> np.ndarray:
    """float32 edge values for a given scale (see module docstring)."""
    sc = np.float32(scale)
    m = np.asarray(mids, dtype=np.float32)
    at = (m * sc).astype(np.float32)
    vals = [np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 1e-38, -1e-38, 1e-45], np.float32),
            at, -at, np.nextafter(at, np.float32(np.inf)), np.nextafter(at, np.float32(-np.inf)),
            (np.float32(448.0) * sc * np.array([1.0, 1 + 2 ** -20, 1 - 2 ** -20, 1.0357142857, 1.036],
                                                np.float32)).astype(np.float32)]
    return np.concatenate(vals).astype(np.float32)
