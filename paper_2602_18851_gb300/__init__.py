"""Python binding of ``libgas.so`` (include/gas.h): argument marshalling only.

Per-head spectral norms sigma_{l,h} = ||W^Q_h W^K_{g(h)}^T||_2 by implicit power
iteration (paper Section 4, Algorithms 2-3) and per-layer geometry-aware FP8 scales
(Section 3.4, Eq. 15), all computed by the CUDA kernels of the library.  PyTorch only
supplies device memory and the current stream.  There is no fallback: if the library
cannot be loaded every call raises.
"""

from __future__ import annotations

import ctypes
import os
import re
from typing import List, Optional, Sequence

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libgas.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "gas.h")
HEADERS = [HEADER, os.path.join(os.path.dirname(HERE), "include", "gas_fp8.h")]

GAS_OK = 0
GAS_ERR_INVALID_ARG = 1
GAS_ERR_UNSUPPORTED = 2
GAS_ERR_CUDA = 3
GAS_ERR_ALLOC = 4
GAS_ERR_DEVICE_TIMEOUT = 5

GAS_DEV_NONFINITE_SIGMA = 0x1
GAS_DEV_WAIT_TIMEOUT = 0x2

METHOD_AUTO = 0
METHOD_STREAM = 1
METHOD_GRAM = 2
METHOD_FUSED = 3
METHODS = {"auto": METHOD_AUTO, "stream": METHOD_STREAM, "gram": METHOD_GRAM, "fused": METHOD_FUSED}

E4M3_MAX = 448.0


class GasError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{_status_name(status)}: {msg}")
        self.status = status


_lib = None


def _status_name(s: int) -> str:
    return {0: "GAS_OK", 1: "GAS_ERR_INVALID_ARG", 2: "GAS_ERR_UNSUPPORTED", 3: "GAS_ERR_CUDA",
            4: "GAS_ERR_ALLOC", 5: "GAS_ERR_DEVICE_TIMEOUT"}.get(s, f"status {s}")


def build(force: bool = False) -> str:
    from .builder import build as _build
    return _build(force=force)


def exported_names() -> List[str]:
    """Function names declared in include/gas.h and include/gas_fp8.h."""
    names = []
    for path in HEADERS:
        src = open(path).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"\b(gas_[a-z0-9_]+)\s*\(", src)
    return names


def load(path: str = LIB_PATH):
    """Load the library (raises OSError if it is missing: no fallback path exists)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise OSError(f"{path} not found: build it with python -m paper_2602_18851_gb300.builder")
    lib = ctypes.CDLL(path)
    vp, c_int, c_double, c_ll = ctypes.c_void_p, ctypes.c_int, ctypes.c_double, ctypes.c_longlong
    lib.gas_create.argtypes = [c_int] * 5 + [ctypes.POINTER(vp)]
    lib.gas_destroy.argtypes = [vp]
    lib.gas_workspace_bytes.argtypes = [vp]
    lib.gas_workspace_bytes.restype = ctypes.c_size_t
    lib.gas_set_calibration.argtypes = [vp, c_int, c_double, c_double]
    lib.gas_set_method.argtypes = [vp, c_int]
    lib.gas_spectral_norms.argtypes = [vp, vp, vp, c_int, vp, vp, vp, vp]
    lib.gas_scales.argtypes = [vp, vp, c_double, c_double, c_double, vp, vp]
    lib.gas_refresh.argtypes = [vp, vp, vp, c_int, vp, vp, vp, c_double, c_double, c_double, vp, vp]
    lib.gas_gamma_min.argtypes = [c_int, c_ll, c_int, c_double]
    lib.gas_gamma_min.restype = c_double
    lib.gas_alpha_min.argtypes = [c_double, c_int, c_int, c_ll, c_int, c_double]
    lib.gas_alpha_min.restype = c_double
    lib.gas_resolve_calibration.argtypes = [vp, c_double, c_double, ctypes.POINTER(c_double),
                                            ctypes.POINTER(c_double)]
    lib.gas_last_error.argtypes = [vp]
    lib.gas_last_error.restype = ctypes.c_char_p
    lib.gas_status_string.argtypes = [c_int]
    lib.gas_status_string.restype = ctypes.c_char_p
    lib.gas_get_device_status.argtypes = [vp, ctypes.POINTER(c_int), c_int]
    lib.gas_selftest_wait_timeout.argtypes = [vp, c_int, vp]
    lib.gas_last_launch_count.argtypes = [vp]
    lib.gas_set_launch_events.argtypes = [vp, vp, c_int]
    lib.gas_last_launch_name.argtypes = [vp, c_int]
    lib.gas_last_launch_name.restype = ctypes.c_char_p
    lib.gas_spectral_norms_static.argtypes = [c_int] * 5 + [vp, vp, c_int, vp, vp, vp, vp]
    lib.gas_static_scratch_bytes.argtypes = [c_int] * 4
    lib.gas_static_scratch_bytes.restype = ctypes.c_size_t
    lib.gas_layer_refresh.argtypes = [vp, vp, vp, c_int, vp, vp, vp, c_double, c_double, c_double, vp, vp]
    lib.gas_set_weight_layout.argtypes = [vp, c_int, c_ll, c_ll, c_ll, c_ll]
    lib.gas_set_weight_dtype.argtypes = [vp, c_int]
    lib.gas_fp8_create.argtypes = [c_int, c_int, c_int, ctypes.POINTER(vp)]
    lib.gas_fp8_destroy.argtypes = [vp]
    lib.gas_fp8_reset.argtypes = [vp, ctypes.c_float, vp]
    lib.gas_fp8_delayed_scales.argtypes = [vp, c_double, vp, vp]
    lib.gas_fp8_quantize.argtypes = [vp, c_int, vp, c_int, c_ll, vp, vp, c_int, vp, vp]
    lib.gas_fp8_end_step.argtypes = [vp, vp, c_int, c_int, c_int, vp]
    lib.gas_fp8_auto_alpha.argtypes = [vp, c_double, c_double, vp, vp]
    lib.gas_fp8_slack_count.argtypes = [vp, ctypes.POINTER(c_int)]
    lib.gas_fp8_last_error.argtypes = [vp]
    lib.gas_fp8_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(st: int, h=None):
    if st != GAS_OK:
        msg = load().gas_last_error(h)
        raise GasError(st, (msg or b"").decode())


def gamma_min(d_h: int, n_heads_total: int, seq_len: int = 1024, delta_star: float = 1e-6) -> float:
    """Eq. 12: smallest gamma > 1 with gamma - 1 - ln gamma >= (2/d_h) ln(2 N L / delta*)."""
    return load().gas_gamma_min(int(d_h), int(n_heads_total), int(seq_len), float(delta_star))


def alpha_min(gamma: float, d: int, d_h: int, n_heads_total: int, seq_len: int = 1024,
              delta_star: float = 1e-6) -> float:
    """Eq. 13: sqrt(2 gamma d_h)/d * sqrt(ln(4 N L^2 / delta*))."""
    return load().gas_alpha_min(float(gamma), int(d), int(d_h), int(n_heads_total), int(seq_len),
                                float(delta_star))


def _ptr_array(tensors: Sequence[torch.Tensor], rows: int, d: int, name: str, layout=None,
               dtype=torch.bfloat16):
    """Device pointers of per-layer weight tensors.  Default layout: each tensor is the
    contiguous [rows, d] matrix.  With a strided layout (heads, d_h, ld, hs) each tensor
    starts at the matrix's first element and must cover its last one."""
    arr = (ctypes.c_void_p * len(tensors))()
    for i, t in enumerate(tensors):
        if t.dtype != dtype or not t.is_cuda:
            raise ValueError(f"{name}[{i}] must be a CUDA {dtype} tensor")
        if layout is None:
            if not t.is_contiguous() or tuple(t.shape) != (rows, d):
                raise ValueError(f"{name}[{i}] must be contiguous with shape {(rows, d)}, got {tuple(t.shape)}")
        else:
            if layout[0] == "cols":
                _, nrows, ld = layout
                last = (d - 1) * ld + nrows - 1
            else:
                heads, dh, ld, hs = layout
                last = (heads - 1) * hs + (dh - 1) * ld + d - 1
            avail = t.untyped_storage().nbytes() // t.element_size() - t.storage_offset()
            if last >= avail:
                raise ValueError(f"{name}[{i}]: the strided matrix needs {last + 1} elements, "
                                 f"the tensor's storage holds {avail} from its first element")
        arr[i] = t.data_ptr()
    return arr


def _stream_ptr(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


class Handle:
    """One model shape (layers, d, n_q, n_kv, d_h) and its device workspace."""

    def __init__(self, layers: int, d: int, n_q: int, n_kv: int, d_h: int):
        lib = load()
        self.layers, self.d, self.n_q, self.n_kv, self.d_h = layers, d, n_q, n_kv, d_h
        h = ctypes.c_void_p()
        _check(lib.gas_create(layers, d, n_q, n_kv, d_h, ctypes.byref(h)), None)
        self._h = h
        self._lq = self._lk = None  # strided layouts of Wq / Wk (None: contiguous)

    # -- lifetime --------------------------------------------------------------------
    def close(self):
        if getattr(self, "_h", None):
            load().gas_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- configuration -----------------------------------------------------------------
    @property
    def workspace_bytes(self) -> int:
        return int(load().gas_workspace_bytes(self._h))

    def set_calibration(self, seq_len: int = 1024, eta_fp8: float = 0.8, alpha_override: float = 0.0):
        _check(load().gas_set_calibration(self._h, int(seq_len), float(eta_fp8), float(alpha_override)),
               self._h)

    def set_weight_layout(self, ld_q: int = 0, ld_k: int = 0, head_stride_q: int = 0, head_stride_k: int = 0,
                          layout: str = "rows"):
        """Strided weights (include/gas.h, gas_set_weight_layout).  "rows": element (row i
        of head j, column c) at w[j * head_stride + i * ld + c]; "cols" (GPT-2 Conv1D):
        element (row r, column c) at w[c * ld + r].  0 keeps a default."""
        code = {"rows": 0, "cols": 1}[layout]
        _check(load().gas_set_weight_layout(self._h, code, int(ld_q), int(ld_k), int(head_stride_q),
                                            int(head_stride_k)), self._h)
        if layout == "cols":
            self._lq = ("cols", self.n_q * self.d_h, ld_q or self.n_q * self.d_h)
            self._lk = ("cols", self.n_kv * self.d_h, ld_k or self.n_kv * self.d_h)
            return
        lq = ld_q or self.d
        lk = ld_k or self.d
        hq = head_stride_q or lq * self.d_h
        hk = head_stride_k or lk * self.d_h
        default = (lq == self.d and lk == self.d and hq == self.d * self.d_h and hk == self.d * self.d_h)
        self._lq = None if default else (self.n_q, self.d_h, lq, hq)
        self._lk = None if default else (self.n_kv, self.d_h, lk, hk)

    def set_weight_dtype(self, dtype):
        """Weight element type: "bf16" (default) or "f16" (torch dtypes accepted)."""
        code = {"bf16": GAS_DTYPE_BF16, torch.bfloat16: GAS_DTYPE_BF16, "f16": GAS_DTYPE_F16,
                torch.float16: GAS_DTYPE_F16, "f32": GAS_DTYPE_F32, torch.float32: GAS_DTYPE_F32}[dtype]
        _check(load().gas_set_weight_dtype(self._h, code), self._h)
        self._wdtype = {GAS_DTYPE_F16: torch.float16, GAS_DTYPE_F32: torch.float32}.get(code, torch.bfloat16)

    def _weights(self, wq, wk):
        lq, lk = getattr(self, "_lq", None), getattr(self, "_lk", None)
        dt = getattr(self, "_wdtype", torch.bfloat16)
        return (_ptr_array(wq, self.n_q * self.d_h, self.d, "wq", lq, dt),
                _ptr_array(wk, self.n_kv * self.d_h, self.d, "wk", lk, dt))

    def set_method(self, method):
        m = METHODS[method] if isinstance(method, str) else int(method)
        _check(load().gas_set_method(self._h, m), self._h)

    def resolve_calibration(self, gamma: float = 0.0, delta_star: float = 1e-6):
        g, a = ctypes.c_double(), ctypes.c_double()
        _check(load().gas_resolve_calibration(self._h, float(gamma), float(delta_star), ctypes.byref(g),
                                              ctypes.byref(a)), self._h)
        return g.value, a.value

    @property
    def last_launch_count(self) -> int:
        return int(load().gas_last_launch_count(self._h))

    def last_launch_names(self) -> List[str]:
        lib = load()
        return [lib.gas_last_launch_name(self._h, i).decode() for i in range(self.last_launch_count)]

    def set_launch_events(self, events: Optional[Sequence[torch.cuda.Event]]):
        """Bracket each library kernel i of later calls with events[2i] / events[2i+1]."""
        self._events = list(events) if events else []
        if not self._events:
            _check(load().gas_set_launch_events(self._h, None, 0), self._h)
            return
        for e in self._events:
            if e.cuda_event == 0:  # torch creates the CUDA event lazily
                e.record()
        arr = (ctypes.c_void_p * len(self._events))(*[e.cuda_event for e in self._events])
        _check(load().gas_set_launch_events(self._h, arr, len(self._events)), self._h)

    def device_status(self, clear: bool = False) -> int:
        code = ctypes.c_int()
        st = load().gas_get_device_status(self._h, ctypes.byref(code), 1 if clear else 0)
        if st not in (GAS_OK, GAS_ERR_DEVICE_TIMEOUT):
            _check(st, self._h)
        return code.value

    def selftest_wait_timeout(self, which: int, stream=None) -> None:
        """Enqueue a kernel whose bounded wait runs out on purpose (0: an mbarrier phase,
        1: a cross-CTA flag); afterwards device_status() reports GAS_DEV_WAIT_TIMEOUT."""
        _check(load().gas_selftest_wait_timeout(self._h, int(which), _stream_ptr(stream)), self._h)

    # -- compute -------------------------------------------------------------------------
    def _vec_args(self, v_in, v_out, sigma, device):
        shape = (self.layers, self.n_q, self.d)
        if v_in.dtype != torch.float32 or tuple(v_in.shape) != shape or not v_in.is_contiguous():
            raise ValueError(f"v_in must be a contiguous float32 tensor of shape {shape}")
        if sigma is None:
            sigma = torch.empty(self.layers, self.n_q, device=device, dtype=torch.float32)
        return v_out, sigma

    def spectral_norms(self, wq: Sequence[torch.Tensor], wk: Sequence[torch.Tensor], iters: int,
                       v_in: torch.Tensor, v_out: Optional[torch.Tensor] = None,
                       sigma: Optional[torch.Tensor] = None, write_back: bool = True, stream=None):
        """sigma[l,h] after `iters` power iterations from v_in; v_out the unit right
        singular vector estimates (warm start for the next call).  Returns (sigma, v_out)."""
        qa, ka = self._weights(wq, wk)
        if v_out is None and write_back:
            v_out = torch.empty_like(v_in)
        v_out, sigma = self._vec_args(v_in, v_out, sigma, v_in.device)
        st = load().gas_spectral_norms(self._h, qa, ka, int(iters), v_in.data_ptr(),
                                       v_out.data_ptr() if v_out is not None else None,
                                       sigma.data_ptr(), _stream_ptr(stream))
        _check(st, self._h)
        return sigma, v_out

    def scales(self, sigma: torch.Tensor, gamma: float = 0.0, delta_star: float = 1e-6,
               r_max: float = E4M3_MAX, s: Optional[torch.Tensor] = None, stream=None):
        """Per-layer scale (Eq. 15) from per-head sigmas."""
        if s is None:
            s = torch.empty(self.layers, device=sigma.device, dtype=torch.float32)
        st = load().gas_scales(self._h, sigma.data_ptr(), float(gamma), float(delta_star), float(r_max),
                               s.data_ptr(), _stream_ptr(stream))
        _check(st, self._h)
        return s

    def refresh(self, wq, wk, iters: int, v_in: torch.Tensor, v_out: Optional[torch.Tensor] = None,
                sigma: Optional[torch.Tensor] = None, s: Optional[torch.Tensor] = None,
                gamma: float = 0.0, delta_star: float = 1e-6, r_max: float = E4M3_MAX,
                write_back: bool = True, stream=None):
        """Spectral norms and per-layer scales in one call.  Returns (sigma, s, v_out)."""
        qa, ka = self._weights(wq, wk)
        if v_out is None and write_back:
            v_out = torch.empty_like(v_in)
        v_out, sigma = self._vec_args(v_in, v_out, sigma, v_in.device)
        if s is None:
            s = torch.empty(self.layers, device=v_in.device, dtype=torch.float32)
        st = load().gas_refresh(self._h, qa, ka, int(iters), v_in.data_ptr(),
                                v_out.data_ptr() if v_out is not None else None, sigma.data_ptr(),
                                float(gamma), float(delta_star), float(r_max), s.data_ptr(),
                                _stream_ptr(stream))
        _check(st, self._h)
        return sigma, s, v_out


    def layer_refresh(self, wq, wk, iters: int, v_in: torch.Tensor, v_out: Optional[torch.Tensor] = None,
                      sigma: Optional[torch.Tensor] = None, s: Optional[torch.Tensor] = None,
                      gamma: float = 0.0, delta_star: float = 1e-6, r_max: float = E4M3_MAX,
                      write_back: bool = True, with_scales: bool = True, stream=None):
        """Whole-layer sigma_l = ||W^Q W^K_exp^T||_2 (Algorithms 2-3 over all heads), one v
        per layer: v_in [layers, d].  Returns (sigma[layers], s[layers] or None, v_out)."""
        qa, ka = self._weights(wq, wk)
        shape = (self.layers, self.d)
        if v_in.dtype != torch.float32 or tuple(v_in.shape) != shape or not v_in.is_contiguous():
            raise ValueError(f"v_in must be a contiguous float32 tensor of shape {shape}")
        if v_out is None and write_back:
            v_out = torch.empty_like(v_in)
        if sigma is None:
            sigma = torch.empty(self.layers, device=v_in.device, dtype=torch.float32)
        if s is None and with_scales:
            s = torch.empty(self.layers, device=v_in.device, dtype=torch.float32)
        st = load().gas_layer_refresh(self._h, qa, ka, int(iters), v_in.data_ptr(),
                                      v_out.data_ptr() if v_out is not None else None, sigma.data_ptr(),
                                      float(gamma), float(delta_star), float(r_max),
                                      s.data_ptr() if s is not None else None, _stream_ptr(stream))
        _check(st, self._h)
        return sigma, s, v_out


GAS_DTYPE_BF16 = 0
GAS_DTYPE_F32 = 1
GAS_DTYPE_F16 = 2
GAS_FP8_SATURATE = 0x1
GAS_FP8_MAX_SLACK = 16384


def _check_fp8(st: int, h=None):
    if st != GAS_OK:
        msg = load().gas_fp8_last_error(h)
        raise GasError(st, (msg or b"").decode())


def fp8_stats_buffer(count: int = 1, device=None) -> torch.Tensor:
    """Device storage for `count` gas_fp8_stats records (24 bytes each)."""
    return torch.zeros(count, 3, dtype=torch.int64, device=device or "cuda")


def decode_fp8_stats(buf: torch.Tensor) -> List[dict]:
    """Host view of gas_fp8_stats records held in a fp8_stats_buffer tensor."""
    raw = buf.detach().cpu().contiguous()
    f = raw.view(torch.float32).view(-1, 6)
    return [{"amax": float(f[i, 0]), "max_scaled": float(f[i, 1]), "overflow": int(raw[i, 1]),
             "count": int(raw[i, 2])} for i in range(raw.shape[0])]


class Fp8State:
    """The consumer side of the scales (include/gas_fp8.h): E4M3 cast with overflow
    statistics (Algorithm 1, Stage 3), delayed-scaling history (Eq. 1) and the auto-alpha
    slack buffer (Section 3.5, Algorithm 4)."""

    def __init__(self, layers: int, history_len: int = 16, burn_in_steps: int = 0):
        lib = load()
        self.layers = layers
        h = ctypes.c_void_p()
        _check_fp8(lib.gas_fp8_create(int(layers), int(history_len), int(burn_in_steps), ctypes.byref(h)), None)
        self._h = h

    def close(self):
        if getattr(self, "_h", None):
            load().gas_fp8_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def reset(self, history_init: float = 1.0, stream=None):
        _check_fp8(load().gas_fp8_reset(self._h, float(history_init), _stream_ptr(stream)), self._h)

    def delayed_scales(self, eta: float = 0.9, out: Optional[torch.Tensor] = None, stream=None):
        """Eq. 1 for every layer."""
        if out is None:
            out = torch.empty(self.layers, device="cuda", dtype=torch.float32)
        _check_fp8(load().gas_fp8_delayed_scales(self._h, float(eta), out.data_ptr(), _stream_ptr(stream)),
                   self._h)
        return out

    def quantize(self, layer: int, s: torch.Tensor, scale: torch.Tensor, q_out: Optional[torch.Tensor] = None,
                 saturate: bool = True, stats: Optional[torch.Tensor] = None, want_codes: bool = True,
                 stream=None):
        """S / scale -> E4M3 codes (uint8, same shape as S) and one stats record.
        `scale` is a one-element float32 CUDA tensor (e.g. s[l:l+1])."""
        if s.dtype == torch.bfloat16:
            dt = GAS_DTYPE_BF16
        elif s.dtype == torch.float32:
            dt = GAS_DTYPE_F32
        else:
            raise ValueError("logits must be bfloat16 or float32")
        if not s.is_contiguous() or not s.is_cuda:
            raise ValueError("logits must be a contiguous CUDA tensor")
        if scale.dtype != torch.float32 or scale.numel() < 1:
            raise ValueError("scale must be a float32 CUDA tensor with at least one element")
        if q_out is None and want_codes:
            q_out = torch.empty(s.shape, dtype=torch.uint8, device=s.device)
        if stats is None:
            stats = fp8_stats_buffer(1, s.device)
        st = load().gas_fp8_quantize(self._h, int(layer), s.data_ptr() if s.numel() else None, dt, s.numel(),
                                     scale.data_ptr(), q_out.data_ptr() if q_out is not None else None,
                                     GAS_FP8_SATURATE if saturate else 0, stats.data_ptr(), _stream_ptr(stream))
        _check_fp8(st, self._h)
        return q_out, stats

    def end_step(self, sigma: Optional[torch.Tensor] = None, d: int = 0, d_h: int = 0, stream=None):
        """Push the step maxima into the history; with sigma ([layers, n_q]) also record
        the slack ratios of Eq. 16."""
        n_q = int(sigma.shape[-1]) if sigma is not None else 0
        _check_fp8(load().gas_fp8_end_step(self._h, sigma.data_ptr() if sigma is not None else None, n_q,
                                           int(d), int(d_h), _stream_ptr(stream)), self._h)

    def auto_alpha(self, q: float = 0.9999, kappa: float = 1.0, out: Optional[torch.Tensor] = None, stream=None):
        """Algorithm 4 on the recorded slack ratios (one float32 on the device)."""
        if out is None:
            out = torch.empty(1, device="cuda", dtype=torch.float32)
        _check_fp8(load().gas_fp8_auto_alpha(self._h, float(q), float(kappa), out.data_ptr(), _stream_ptr(stream)),
                   self._h)
        return out

    def slack_count(self) -> int:
        c = ctypes.c_int()
        _check_fp8(load().gas_fp8_slack_count(self._h, ctypes.byref(c)), self._h)
        return c.value


__all__ = ["Handle", "Fp8State", "fp8_stats_buffer", "decode_fp8_stats", "GasError", "load", "build", "gamma_min", "alpha_min", "exported_names",
           "METHOD_AUTO", "METHOD_STREAM", "METHOD_GRAM", "METHOD_FUSED", "E4M3_MAX", "LIB_PATH"]
