"""Float64 CPU oracle for per-head spectral norms and geometry-aware FP8 scales.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference leg may import this package.  The CUDA
library never calls it and shares no code with it; the only thing the two
sides share is the seeded input generator in ``synth/``.

Pieces (each cites the passage it restates):
* ``gas_oracle.c`` — Algorithm 2 (Appendix E.1) with M = W^Q_h W^K_g^T formed
  explicitly (``mode="explicit"``) or applied in factored form (Section 4.1,
  ``mode="factored"``); Algorithm 3 (Appendix E.2) for a whole layer with
  RepeatBlocks / SumGroups, and the explicit W^K expansion it avoids.
* ``calib.py`` — Eq. 12 (gamma), Eq. 13 (alpha_min), Eq. 15 (per-layer scale).
* ``fp8.py`` — the consumer of the scale: E4M3 cast of S / scale with overflow
  statistics (Algorithm 1, Stage 3; Table 4), delayed scaling (Eq. 1) and auto-alpha
  (Section 3.5, Eq. 16, Algorithm 4).

Readings where the paper is silent: sigma is the last iteration's ||M v_{k-1}||;
a zero start vector or a zero sigma gives sigma = 0 and v_out = 0; head h uses KV
group h // (n_q/n_kv).
"""

import ctypes

import numpy as np

from . import calib  # noqa: F401
from .build import LIB, build

_lib = None


def _load():
    global _lib
    if _lib is None:
        path = build()
        lib = ctypes.CDLL(path)
        u16p = ctypes.POINTER(ctypes.c_uint16)
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int)
        lib.oracle_form_interaction.argtypes = [ctypes.c_int, ctypes.c_int, u16p, u16p, dp]
        lib.oracle_form_interaction.restype = None
        lib.oracle_power_iteration_dense.argtypes = [ctypes.c_int, dp, dp, ctypes.c_int, dp, dp]
        lib.oracle_power_iteration_factored.argtypes = [ctypes.c_int, ctypes.c_int, u16p, u16p,
                                                        dp, ctypes.c_int, dp, dp]
        lib.oracle_heads.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                     ctypes.POINTER(u16p), ctypes.POINTER(u16p),
                                     ctypes.POINTER(ctypes.c_float), ctypes.c_int, ctypes.c_int,
                                     ctypes.c_int, ip, ip, dp, dp, ctypes.c_int]
        lib.oracle_layer_implicit_gqa.argtypes = [ctypes.c_int] * 4 + [u16p, u16p, dp,
                                                                       ctypes.c_int, dp, dp]
        lib.oracle_layer_form_expanded.argtypes = [ctypes.c_int] * 4 + [u16p, u16p, dp]
        lib.oracle_max_threads.restype = ctypes.c_int
        lib.oracle_set_weight_format.argtypes = [ctypes.c_int]
        lib.oracle_set_weight_format.restype = None
        lib.oracle_decode_weights.argtypes = [u16p, ctypes.c_long, dp]
        lib.oracle_decode_weights.restype = None
        _lib = lib
    return _lib


def _u16(a):
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError("bf16 weights must be passed as their uint16 bit patterns")
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_uint16))


def _f64(a):
    a = np.ascontiguousarray(a, dtype=np.float64)
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def form_interaction(A_bits, B_bits):
    """M = W^Q_h W^K_g^T (d x d float64) from the d_h x d bf16 blocks A, B."""
    A, pa = _u16(A_bits)
    B, pb = _u16(B_bits)
    dh, d = A.shape
    M = np.empty((d, d), dtype=np.float64)
    _load().oracle_form_interaction(d, dh, pa, pb, M.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return M


def power_iteration_dense(M, v0, iters):
    """Algorithm 2 on a formed matrix; returns (sigma, v)."""
    M, pm = _f64(M)
    v0, pv = _f64(v0)
    d = M.shape[0]
    sig = ctypes.c_double()
    v = np.empty(d, dtype=np.float64)
    _load().oracle_power_iteration_dense(d, pm, pv, int(iters), ctypes.byref(sig),
                                         v.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return sig.value, v


def power_iteration_factored(A_bits, B_bits, v0, iters):
    """Algorithm 2 for one head in factored form; returns (sigma, v)."""
    A, pa = _u16(A_bits)
    B, pb = _u16(B_bits)
    v0, pv = _f64(v0)
    dh, d = A.shape
    sig = ctypes.c_double()
    v = np.empty(d, dtype=np.float64)
    _load().oracle_power_iteration_factored(d, dh, pa, pb, pv, int(iters), ctypes.byref(sig),
                                            v.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return sig.value, v


def set_weight_format(fmt: str) -> None:
    """Weight bit format every later call decodes: "bf16" (default) or "f16"."""
    _load().oracle_set_weight_format({"bf16": 0, "f16": 1}[fmt])


def decode_weights(bits) -> np.ndarray:
    """The oracle's exact float64 value of each 16-bit weight in the current format."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).ravel()
    out = np.empty(b.size, dtype=np.float64)
    _load().oracle_decode_weights(b.ctypes.data_as(ctypes.POINTER(ctypes.c_uint16)), b.size,
                                  out.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return out


def heads(d, n_q, n_kv, d_h, wq_bits, wk_bits, v_in, iters, pairs, mode="factored",
          want_v=True, threads=0):
    """Per-head sigma (and v_out) for a list of (layer, head) pairs.

    wq_bits[l] / wk_bits[l]: uint16 arrays [n_q*d_h, d] / [n_kv*d_h, d] (None for
    layers that no pair uses).  v_in: float32 [layers, n_q, d].
    Returns (sigma[len(pairs)], v[len(pairs), d] or None).
    """
    lib = _load()
    layers = len(wq_bits)
    u16p = ctypes.POINTER(ctypes.c_uint16)
    keep = []
    qarr = (u16p * layers)()
    karr = (u16p * layers)()
    for l in range(layers):
        if wq_bits[l] is not None:
            a, p = _u16(wq_bits[l])
            keep.append(a)
            qarr[l] = p
        if wk_bits[l] is not None:
            b, p = _u16(wk_bits[l])
            keep.append(b)
            karr[l] = p
    v_in = np.ascontiguousarray(v_in, dtype=np.float32)
    assert v_in.shape[1:] == (n_q, d), v_in.shape
    pairs = list(pairs)
    for (l, hq) in pairs:
        if wq_bits[l] is None or wk_bits[l] is None:
            raise ValueError(f"layer {l} weights missing for pair ({l},{hq})")
    li = np.array([p[0] for p in pairs], dtype=np.int32)
    hi = np.array([p[1] for p in pairs], dtype=np.int32)
    sig = np.empty(len(pairs), dtype=np.float64)
    vout = np.empty((len(pairs), d), dtype=np.float64) if want_v else None
    rc = lib.oracle_heads(d, n_q, n_kv, d_h, qarr, karr,
                          v_in.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), int(iters),
                          1 if mode == "explicit" else 0, len(pairs),
                          li.ctypes.data_as(ctypes.POINTER(ctypes.c_int)),
                          hi.ctypes.data_as(ctypes.POINTER(ctypes.c_int)),
                          sig.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                          vout.ctypes.data_as(ctypes.POINTER(ctypes.c_double)) if want_v else None,
                          int(threads))
    if rc != 0:
        raise RuntimeError(f"oracle_heads failed rc={rc}")
    return sig, vout


def layer_implicit_gqa(Wq_bits, Wk_bits, n_q, n_kv, d_h, v0, iters):
    """Algorithm 3 over a whole layer (M = W^Q W^K_exp^T); returns (sigma, v)."""
    Wq, pq = _u16(Wq_bits)
    Wk, pk = _u16(Wk_bits)
    v0, pv = _f64(v0)
    d = Wq.shape[1]
    sig = ctypes.c_double()
    v = np.empty(d, dtype=np.float64)
    rc = _load().oracle_layer_implicit_gqa(d, n_q, n_kv, d_h, pq, pk, pv, int(iters),
                                           ctypes.byref(sig),
                                           v.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    if rc != 0:
        raise ValueError("n_q must be a multiple of n_kv")
    return sig.value, v


def layer_form_expanded(Wq_bits, Wk_bits, n_q, n_kv, d_h):
    """M = W^Q W^K_exp^T (d x d) with W^K explicitly expanded (what Section 4.2 avoids)."""
    Wq, pq = _u16(Wq_bits)
    Wk, pk = _u16(Wk_bits)
    d = Wq.shape[1]
    M = np.empty((d, d), dtype=np.float64)
    rc = _load().oracle_layer_form_expanded(d, n_q, n_kv, d_h, pq, pk,
                                            M.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    if rc != 0:
        raise ValueError("n_q must be a multiple of n_kv")
    return M


def spectral_norms(wq_bits, wk_bits, v_in, iters, n_q, n_kv, d_h, mode="factored",
                   threads=0):
    """All heads of all layers; returns (sigma[layers, n_q], v_out[layers, n_q, d])."""
    layers = len(wq_bits)
    d = v_in.shape[-1]
    pairs = [(l, hq) for l in range(layers) for hq in range(n_q)]
    sig, v = heads(d, n_q, n_kv, d_h, wq_bits, wk_bits, v_in, iters, pairs, mode=mode,
                   threads=threads)
    return sig.reshape(layers, n_q), v.reshape(layers, n_q, d)


__all__ = ["calib", "form_interaction", "power_iteration_dense", "power_iteration_factored",
           "heads", "layer_implicit_gqa", "layer_form_expanded", "spectral_norms",
           "max_threads", "LIB", "build", "set_weight_format", "decode_weights"]
