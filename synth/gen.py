"""Seeded draws of attention weights, start vectors and transient perturbations.

All draws use ``torch.Generator`` on the requested device, so a given seed gives
the same bytes for every consumer that reads the returned tensors (CUDA library
and oracle alike).  Values differ between CPU and CUDA generators and may differ
between torch versions; no stored expectation depends on them.

Recipes (per layer l; A_h = rows [h*d_h,(h+1)*d_h) of Wq[l], B_g = rows of Wk[l]
for KV group g; g(h) = h // (n_q/n_kv)):

* ``spike1``    A, B iid N(0, 0.02^2); per KV group a unit b_g in R^{d_h}, unit c_g
                in R^d, s^K ~ U[0.5,3]: B_g += s^K b_g c_g^T; per head a unit a_h
                in R^d, s^Q ~ U[0.5,3]: A_h += s^Q b_{g(h)} a_h^T.
* ``lognormal`` N(0, 0.02^2) times a per-matrix factor exp(0.5*xi), xi ~ N(0,1),
                drawn independently for every A_h and B_g.
* ``planted``   B_g = V_g diag(s^K) U_{K,g}^T, A_h = V_{g(h)} diag(s^Q) U_{Q,h}^T with
                V_g in O(d_h) and U in R^{d x d_h} orthonormal (float64 QR), and
                s_k = s_1 k^-0.7, s_1 ~ U[1,8] per matrix.  Then
                M_h = A_h^T B_g = U_Q diag(s^Q s^K) U_K^T, so sigma_1 = s^Q_1 s^K_1.
* ``spike4``    N(0, 0.02^2) plus rank-4 spikes: per group orthonormal b_{g,1..4} in
                R^{d_h} and c_{g,1..4} in R^d; per head orthonormal a_{h,1..4};
                B_g += sum_r s b_{g,r} c_{g,r}^T, A_h += sum_r s b_{g(h),r} a_{h,r}^T,
                every s ~ U[1,6].

Weights are rounded to bf16 with round-to-nearest-even (``Tensor.to``).
"""

from __future__ import annotations

from typing import Dict, List, Tuple

import torch

from .configs import (TRANSIENT_EPS, TRANSIENT_RANK, TRANSIENT_SPIKE_EPS,
                      TRANSIENT_SPIKE_STEPS, Workload)


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFF_FFFF_FFFF_FFFF)
    return g


def _unit_rows(n: int, m: int, gen, device, dtype) -> torch.Tensor:
    x = torch.randn(n, m, generator=gen, device=device, dtype=dtype)
    return x / x.norm(dim=1, keepdim=True)


def _orthonormal(batch: int, rows: int, cols: int, gen, device, dtype) -> torch.Tensor:
    """[batch, rows, cols] with orthonormal columns (QR of a Gaussian matrix).

    The Gaussian is drawn on `device`.  Large batches are factored there; small ones,
    and any batch whose device factorisation is unavailable (the device linear-algebra
    library cannot always be loaded, e.g. under a profiler), on the host."""
    x = torch.randn(batch, rows, cols, generator=gen, device=device, dtype=dtype)
    q = r = None
    if x.is_cuda and x.numel() >= (1 << 22):
        try:
            q, r = torch.linalg.qr(x)
        except RuntimeError:
            q = r = None
    if q is None:
        q, r = torch.linalg.qr(x.cpu())
    # Fix the sign ambiguity of QR so the draw is a function of the seed only.
    sgn = torch.sign(torch.diagonal(r, dim1=-2, dim2=-1))
    sgn[sgn == 0] = 1
    return (q * sgn.unsqueeze(-2)).to(device)


def _draw_layer(wl: Workload, layer: int, device, seed: int):
    """Unrounded (fp32 or fp64) weights of one layer and per-layer metadata."""
    gen = _gen(device, seed * 1000003 + layer)
    nq, nkv, dh, d, G = wl.n_q, wl.n_kv, wl.d_h, wl.d, wl.group
    f32 = torch.float32
    meta: Dict[str, torch.Tensor] = {}
    gidx = torch.arange(nq, device=device) // G
    if wl.recipe == "spike1":
        wq = 0.02 * torch.randn(nq * dh, d, generator=gen, device=device, dtype=f32)
        wk = 0.02 * torch.randn(nkv * dh, d, generator=gen, device=device, dtype=f32)
        b = _unit_rows(nkv, dh, gen, device, f32)
        c = _unit_rows(nkv, d, gen, device, f32)
        a = _unit_rows(nq, d, gen, device, f32)
        sk = 0.5 + 2.5 * torch.rand(nkv, generator=gen, device=device, dtype=f32)
        sq = 0.5 + 2.5 * torch.rand(nq, generator=gen, device=device, dtype=f32)
        wk.view(nkv, dh, d).add_(sk[:, None, None] * b[:, :, None] * c[:, None, :])
        wq.view(nq, dh, d).add_(sq[:, None, None] * b[gidx][:, :, None] * a[:, None, :])
    elif wl.recipe == "lognormal":
        wq = 0.02 * torch.randn(nq * dh, d, generator=gen, device=device, dtype=f32)
        wk = 0.02 * torch.randn(nkv * dh, d, generator=gen, device=device, dtype=f32)
        fq = torch.exp(0.5 * torch.randn(nq, generator=gen, device=device, dtype=f32))
        fk = torch.exp(0.5 * torch.randn(nkv, generator=gen, device=device, dtype=f32))
        wq.view(nq, dh, d).mul_(fq[:, None, None])
        wk.view(nkv, dh, d).mul_(fk[:, None, None])
    elif wl.recipe == "planted":
        f64 = torch.float64
        k = torch.arange(1, dh + 1, device=device, dtype=f64)
        s1q = 1.0 + 7.0 * torch.rand(nq, generator=gen, device=device, dtype=f64)
        s1k = 1.0 + 7.0 * torch.rand(nkv, generator=gen, device=device, dtype=f64)
        sq = s1q[:, None] * k[None, :] ** -0.7
        sk = s1k[:, None] * k[None, :] ** -0.7
        v = _orthonormal(nkv, dh, dh, gen, device, f64)          # V_g
        uq = _orthonormal(nq, d, dh, gen, device, f64)           # U_{Q,h}
        uk = _orthonormal(nkv, d, dh, gen, device, f64)          # U_{K,g}
        wk = (v * sk[:, None, :]) @ uk.transpose(1, 2)           # [nkv, dh, d]
        wq = (v[gidx] * sq[:, None, :]) @ uq.transpose(1, 2)     # [nq, dh, d]
        wk = wk.reshape(nkv * dh, d)
        wq = wq.reshape(nq * dh, d)
        meta["sigma_planted"] = (s1q * s1k[gidx])                # closed-form sigma_1(M_h)
        meta["norm_q"] = s1q                                      # ||W^Q_h||_2
        meta["norm_k"] = s1k                                      # ||W^K_g||_2
        meta["gap"] = torch.full((nq,), 2.0 ** -0.7, device=device, dtype=f64) ** 2
    elif wl.recipe == "spike4":
        R = 4
        wq = 0.02 * torch.randn(nq * dh, d, generator=gen, device=device, dtype=f32)
        wk = 0.02 * torch.randn(nkv * dh, d, generator=gen, device=device, dtype=f32)
        b = _orthonormal(nkv, dh, R, gen, device, f32)           # [nkv, dh, R]
        c = _orthonormal(nkv, d, R, gen, device, f32)            # [nkv, d, R]
        a = _orthonormal(nq, d, R, gen, device, f32)             # [nq, d, R]
        sk = 1.0 + 5.0 * torch.rand(nkv, R, generator=gen, device=device, dtype=f32)
        sq = 1.0 + 5.0 * torch.rand(nq, R, generator=gen, device=device, dtype=f32)
        wk.view(nkv, dh, d).add_((b * sk[:, None, :]) @ c.transpose(1, 2))
        wq.view(nq, dh, d).add_((b[gidx] * sq[:, None, :]) @ a.transpose(1, 2))
    else:
        raise ValueError(f"unknown recipe {wl.recipe!r}")
    return wq, wk, meta


def make_weights(wl: Workload, device="cpu", seed: int | None = None, dtype=torch.bfloat16
                 ) -> Tuple[List[torch.Tensor], List[torch.Tensor], Dict[str, torch.Tensor]]:
    """16-bit weights of every layer (bf16 by default, or float16), one tensor per layer
    and matrix, rounded to nearest from the same unrounded draw.

    Returns (wq, wk, meta): wq[l] is ``[n_q*d_h, d]``, wk[l] is ``[n_kv*d_h, d]``.
    For the ``planted`` recipe ``meta`` holds per-head ``sigma_planted``, ``norm_q``,
    ``norm_k`` ([layers, ...] float64) and the Frobenius norms of the bf16 rounding
    residuals ``err_q``/``err_k`` used for the Weyl perturbation bound.
    """
    seed = wl.seed if seed is None else seed
    wq, wk, metas = [], [], []
    for layer in range(wl.layers):
        q, k, meta = _draw_layer(wl, layer, device, seed)
        qb, kb = q.to(dtype), k.to(dtype)
        if wl.recipe == "planted":
            eq = (qb.double() - q.double()).view(wl.n_q, wl.d_h, wl.d).norm(dim=(1, 2))
            ek = (kb.double() - k.double()).view(wl.n_kv, wl.d_h, wl.d).norm(dim=(1, 2))
            meta["err_q"] = eq
            meta["err_k"] = ek
        wq.append(qb.contiguous())
        wk.append(kb.contiguous())
        metas.append(meta)
        del q, k
    out_meta: Dict[str, torch.Tensor] = {}
    if metas and metas[0]:
        for key in metas[0]:
            out_meta[key] = torch.stack([m[key] for m in metas]).cpu()
    return wq, wk, out_meta


def make_start_vectors(wl: Workload, device="cpu", seed: int | None = None) -> torch.Tensor:
    """Seeded N(0, I_d) start vectors, fp32 ``[layers, n_q, d]`` (not normalised)."""
    seed = (wl.seed if seed is None else seed) + 7777
    gen = _gen(device, seed)
    return torch.randn(wl.layers, wl.n_q, wl.d, generator=gen, device=device, dtype=torch.float32)


class TransientWeights:
    """fp32 master weights plus their bf16 copies, perturbed once per simulated step.

    Per step t and per weight matrix W (one A_h or B_g):
    W += eps_t ||W||_F P Q^T / ||P Q^T||_F with Gaussian P (d_h x 8), Q (d x 8) drawn
    from a generator seeded by (seed, t, layer); eps_t = 1e-3, or 5e-2 for t in 40..45.
    The bf16 tensors are updated in place so their device pointers stay fixed.
    """

    def __init__(self, wl: Workload, device="cuda", seed: int | None = None):
        self.wl = wl
        self.device = device
        self.seed = wl.seed if seed is None else seed
        self.master_q, self.master_k, self.wq, self.wk = [], [], [], []
        for layer in range(wl.layers):
            q, k, _ = _draw_layer(wl, layer, device, self.seed)
            q, k = q.float(), k.float()
            self.master_q.append(q)
            self.master_k.append(k)
            self.wq.append(q.to(torch.bfloat16))
            self.wk.append(k.to(torch.bfloat16))

    @staticmethod
    def eps(step: int) -> float:
        return TRANSIENT_SPIKE_EPS if step in TRANSIENT_SPIKE_STEPS else TRANSIENT_EPS

    def step(self, t: int) -> None:
        wl = self.wl
        eps = self.eps(t)
        for layer in range(wl.layers):
            gen = _gen(self.device, (self.seed * 7919 + t) * 100003 + layer)
            for master, bf in ((self.master_q[layer], self.wq[layer]),
                               (self.master_k[layer], self.wk[layer])):
                n = master.shape[0] // wl.d_h
                w = master.view(n, wl.d_h, wl.d)
                p = torch.randn(n, wl.d_h, TRANSIENT_RANK, generator=gen, device=self.device)
                q = torch.randn(n, wl.d, TRANSIENT_RANK, generator=gen, device=self.device)
                pq = p @ q.transpose(1, 2)
                scale = eps * w.norm(dim=(1, 2)) / pq.norm(dim=(1, 2))
                w.add_(pq * scale[:, None, None])
                bf.copy_(master.to(torch.bfloat16))
                del p, q, pq


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 tensor's bytes (host copy)."""
    import numpy as np
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)

