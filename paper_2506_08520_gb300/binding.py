"""Thin ctypes binding of ``libnystra.so`` (C ABI in ``include/nystra.h``).

Argument marshalling only: every step of the computation runs in the CUDA
kernels behind the C ABI.  torch is used for device memory and streams.
There is no CPU fallback: if the library is missing, every call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libnystra.so")

NYSTRA_F32, NYSTRA_BF16, NYSTRA_F16 = 0, 1, 2
NYSTRA_OK, NYSTRA_EINVAL, NYSTRA_EDTYPE, NYSTRA_ELAUNCH, NYSTRA_ETIMEOUT, NYSTRA_EDEVICE = 0, -1, -2, -3, -4, -5
NYSTRA_LANDMARKS_SEGMENTS, NYSTRA_LANDMARKS_PATCHES = 0, 1
LANDMARKS = {"segments": NYSTRA_LANDMARKS_SEGMENTS, "patches": NYSTRA_LANDMARKS_PATCHES}
# Option flag OR-ed into the landmarks argument: derived factors rounded to
# the 16-bit I/O type (faster, accurate only for soft attention; nystra.h).
NYSTRA_FACTORS_16 = 16
FACTORS = {"pairs": 0, "16": NYSTRA_FACTORS_16}


def _lm(landmarks: str, factors: str = "pairs") -> int:
    return LANDMARKS[landmarks] | FACTORS[factors]
MAX_N, MAX_DH, MAX_M, MAX_ITERS = 1024, 64, 64, 100
QKV_MAX_C = 352
PROJ_MAX_C, PROJ_MAX_N = 384, 65536

_DTYPE_CODE = {torch.float32: NYSTRA_F32, torch.bfloat16: NYSTRA_BF16, torch.float16: NYSTRA_F16}

_lib = None


class NystraError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = f"{where}: {strerror(status)} (status {status})"
        if status == NYSTRA_ELAUNCH:
            msg += f", cudaError {lib().nystra_last_cuda_error()}"
        super().__init__(msg)


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built (no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2506_08520_gb300.build` (no CPU fallback exists)")
        L = ctypes.CDLL(LIB_PATH)
        vp, i = ctypes.c_void_p, ctypes.c_int
        L.nystra_attention.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, vp]
        L.nystra_attention.restype = i
        L.exact_window_attention.argtypes = [vp, vp, vp, vp, i, i, i, i, i, vp]
        L.exact_window_attention.restype = i
        L.nystra_strerror.argtypes = [i]
        L.nystra_strerror.restype = ctypes.c_char_p
        L.nystra_version.restype = i
        L.nystra_last_cuda_error.restype = i
        L.nystra_status.argtypes = [vp]
        L.nystra_status.restype = i
        L.nystra_check.argtypes = [vp]
        L.nystra_check.restype = i
        L.nystra_debug_wait_timeout.argtypes = [ctypes.c_ulonglong, vp]
        L.nystra_debug_wait_timeout.restype = i
        L.nystra_debug_stages.argtypes = [vp, vp, vp, i, i, i, i, i, i, i, i, ctypes.c_longlong, vp, vp]
        L.nystra_attention_ex.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, i, vp]
        L.nystra_attention_ex.restype = i
        L.nystra_pool_bias.argtypes = [vp, i, i, i, i, vp, vp, vp, vp]
        L.nystra_pool_bias.restype = i
        L.nystra_attention_bias.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, vp, vp, vp, i, i, vp]
        L.nystra_attention_bias.restype = i
        L.nystra_attention_qkv.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, vp, vp, vp, i, i, vp]
        L.nystra_attention_qkv.restype = i
        L.nystra_project_qkv.argtypes = [vp, vp, vp, vp, vp, vp, i, i, i, i, i, vp]
        L.nystra_project_qkv.restype = i
        L.nystra_debug_stages.restype = i
        L.nystra_debug_stages_size.argtypes = [i, i, i]
        L.nystra_debug_stages_size.restype = ctypes.c_longlong
        _lib = L
    return _lib


# ---------------------------------------------------------------- raw C ABI
def nystra_attention(q, k, v, out, n_windows, heads, N, d_h, m, iters, dtype, stream) -> int:
    """Raw C-ABI call: pointers as ints, returns the status code."""
    return lib().nystra_attention(q, k, v, out, n_windows, heads, N, d_h, m, iters, dtype, stream)


def nystra_attention_ex(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, dtype, stream) -> int:
    """Raw C-ABI call with a landmark pooling (NYSTRA_LANDMARKS_*)."""
    return lib().nystra_attention_ex(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, dtype, stream)


def nystra_pool_bias(bias, n_bias, N, m, landmarks, bias_L, bias_U, bias_A, stream) -> int:
    return lib().nystra_pool_bias(bias, n_bias, N, m, landmarks, bias_L, bias_U, bias_A, stream)


def nystra_attention_bias(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, bias_L, bias_U, bias_A,
                          bias_windows, dtype, stream) -> int:
    return lib().nystra_attention_bias(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, bias_L, bias_U,
                                       bias_A, bias_windows, dtype, stream)


def nystra_attention_qkv(x, w_qkv, b_qkv, out, n_windows, heads, N, d_h, m, iters, landmarks, bias_L, bias_U,
                         bias_A, bias_windows, dtype, stream) -> int:
    return lib().nystra_attention_qkv(x, w_qkv, b_qkv, out, n_windows, heads, N, d_h, m, iters, landmarks, bias_L,
                                      bias_U, bias_A, bias_windows, dtype, stream)


def nystra_project_qkv(x, w_qkv, b_qkv, q, k, v, n_windows, heads, N, d_h, dtype, stream) -> int:
    return lib().nystra_project_qkv(x, w_qkv, b_qkv, q, k, v, n_windows, heads, N, d_h, dtype, stream)


def exact_window_attention(q, k, v, out, n_windows, heads, N, d_h, dtype, stream) -> int:
    return lib().exact_window_attention(q, k, v, out, n_windows, heads, N, d_h, dtype, stream)


def strerror(status: int) -> str:
    return lib().nystra_strerror(status).decode()


def version() -> int:
    return lib().nystra_version()


def status(stream=None) -> int:
    """Synchronise ``stream`` and return the device-side fault status."""
    return lib().nystra_status(_stream_ptr(stream))


def check(stream=None) -> int:
    """Same as ``status``."""
    return lib().nystra_check(_stream_ptr(stream))


def debug_wait_timeout(limit_ns: int, stream=None) -> int:
    """Test-only: launch a wait that can only time out (see the header)."""
    return lib().nystra_debug_wait_timeout(int(limit_ns), _stream_ptr(stream))


def nystra_debug_stages(q, k, v, n_windows, heads, N, d_h, m, iters, landmarks, dtype, unit, dump, stream) -> int:
    """Raw C-ABI call of the test-only stage dump (see the header)."""
    return lib().nystra_debug_stages(q, k, v, n_windows, heads, N, d_h, m, iters, landmarks, dtype, int(unit), dump,
                                     stream)


def nystra_debug_stages_size(N: int, d_h: int, m: int) -> int:
    return lib().nystra_debug_stages_size(N, d_h, m)


# Regions of the stage dump, in the order and with the shapes the header gives.
def _stage_shapes(N: int, d: int, m: int):
    return [("qbar", (m, d)), ("kbar", (m, d)), ("GLn", (N, m)), ("mU", (m,)), ("W", (m, d + 1)),
            ("GAn", (m, m)), ("Z", (m, m)), ("Y", (m, d + 1)), ("out", (N, d))]


# ------------------------------------------------------------ torch helpers
def _stream_ptr(stream) -> int | None:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _geometry(q: torch.Tensor):
    if q.dim() == 4:
        n_windows, heads, N, d = q.shape
    elif q.dim() == 3:
        (n_windows, N, d), heads = q.shape, 1
    else:
        raise ValueError("expected [n_windows, heads, N, d_h] or [units, N, d_h]")
    return n_windows, heads, N, d


def _check(q, k, v, out):
    for t in (q, k, v, out):
        if not t.is_cuda:
            raise ValueError("tensors must be on a CUDA device (no CPU path)")
        if not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
        if t.shape != q.shape or t.dtype != q.dtype:
            raise ValueError("q, k, v and out must share shape and dtype")
    if q.dtype not in _DTYPE_CODE:
        raise ValueError(f"unsupported dtype {q.dtype}")


def nystra(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, m: int = 16, iters: int = 6,
           out: torch.Tensor | None = None, stream=None, landmarks: str = "segments",
           factors: str = "pairs") -> torch.Tensor:
    """PnP-Nystra attention of device tensors ``[n_windows, heads, N, d_h]``;
    ``landmarks`` is "segments" (default) or "patches" (square patches);
    ``factors`` "pairs" (default: derived factors as 16-bit hi + lo pairs) or
    "16" (rounded to the 16-bit I/O type, NYSTRA_FACTORS_16)."""
    out = torch.empty_like(q) if out is None else out
    _check(q, k, v, out)
    nw, h, N, d = _geometry(q)
    with torch.cuda.device(q.device):
        if landmarks == "segments" and factors == "pairs":
            rc = nystra_attention(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), nw, h, N, d,
                                  m, iters, _DTYPE_CODE[q.dtype], _stream_ptr(stream))
        else:
            rc = nystra_attention_ex(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), nw, h, N, d,
                                     m, iters, _lm(landmarks, factors), _DTYPE_CODE[q.dtype], _stream_ptr(stream))
    if rc != NYSTRA_OK:
        raise NystraError(rc, "nystra_attention")
    return out


def exact(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, out: torch.Tensor | None = None,
          stream=None) -> torch.Tensor:
    """Exact softmax window attention (the computation PnP-Nystra replaces)."""
    out = torch.empty_like(q) if out is None else out
    _check(q, k, v, out)
    nw, h, N, d = _geometry(q)
    with torch.cuda.device(q.device):
        rc = exact_window_attention(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), nw, h, N, d,
                                    _DTYPE_CODE[q.dtype], _stream_ptr(stream))
    if rc != NYSTRA_OK:
        raise NystraError(rc, "exact_window_attention")
    return out


def debug_stages(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, m: int, iters: int, unit: int,
                 stream=None, landmarks: str = "segments") -> dict:
    """Test-only: every intermediate of one unit (fp32 CPU tensors by name)."""
    _check(q, k, v, q)
    nw, h, N, d = _geometry(q)
    size = nystra_debug_stages_size(N, d, m)
    if size < 0:
        raise NystraError(int(size), "nystra_debug_stages_size")
    dump = torch.empty(size, dtype=torch.float32, device=q.device)
    with torch.cuda.device(q.device):
        rc = nystra_debug_stages(q.data_ptr(), k.data_ptr(), v.data_ptr(), nw, h, N, d, m, iters,
                                 LANDMARKS[landmarks], _DTYPE_CODE[q.dtype], unit, dump.data_ptr(),
                                 _stream_ptr(stream))
    if rc != NYSTRA_OK:
        raise NystraError(rc, "nystra_debug_stages")
    torch.cuda.synchronize(q.device)
    host = dump.cpu()
    out, pos = {}, 0
    for name, shape in _stage_shapes(N, d, m):
        n = 1
        for x in shape:
            n *= x
        out[name] = host[pos:pos + n].reshape(shape)
        pos += n
    return out


def pool_bias(bias: torch.Tensor, m: int, landmarks: str = "segments", stream=None):
    """Landmark blocks (B_L, B_U, B_A) of an fp32 device bias ``[..., N, N]``."""
    if not bias.is_cuda or bias.dtype != torch.float32 or not bias.is_contiguous():
        raise ValueError("bias must be a contiguous fp32 CUDA tensor")
    N = bias.shape[-1]
    lead = bias.shape[:-2]
    n = bias.numel() // (N * N)
    bL = torch.empty(lead + (N, m), dtype=torch.float32, device=bias.device)
    bU = torch.empty(lead + (m, N), dtype=torch.float32, device=bias.device)
    bA = torch.empty(lead + (m, m), dtype=torch.float32, device=bias.device)
    with torch.cuda.device(bias.device):
        rc = nystra_pool_bias(bias.data_ptr(), n, N, m, LANDMARKS[landmarks], bL.data_ptr(), bU.data_ptr(),
                              bA.data_ptr(), _stream_ptr(stream))
    if rc != NYSTRA_OK:
        raise NystraError(rc, "nystra_pool_bias")
    return bL, bU, bA


def nystra_biased(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, pooled, m: int = 16, iters: int = 6,
                  out: torch.Tensor | None = None, stream=None, landmarks: str = "segments",
                  factors: str = "pairs") -> torch.Tensor:
    """PnP-Nystra with a score bias already pooled by ``pool_bias``: blocks of
    shape ``[heads, ...]`` (shared by all windows) or ``[n_windows, heads, ...]``."""
    out = torch.empty_like(q) if out is None else out
    _check(q, k, v, out)
    nw, h, N, d = _geometry(q)
    bL, bU, bA = pooled
    bw = bL.numel() // (h * N * m)
    with torch.cuda.device(q.device):
        rc = nystra_attention_bias(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), nw, h, N, d, m, iters,
                                   _lm(landmarks, factors), bL.data_ptr(), bU.data_ptr(), bA.data_ptr(), bw,
                                   _DTYPE_CODE[q.dtype], _stream_ptr(stream))
    if rc != NYSTRA_OK:
        raise NystraError(rc, "nystra_attention_bias")
    return out


def nystra_qkv(x: torch.Tensor, w_qkv: torch.Tensor, heads: int, m: int = 16, iters: int = 6,
               b_qkv: torch.Tensor | None = None, pooled=None, out: torch.Tensor | None = None, stream=None,
               landmarks: str = "segments", factors: str = "pairs") -> torch.Tensor:
    """Fused projection + PnP-Nystra: tokens ``x`` ``[n_windows, N, C]``, weights
    ``w_qkv`` ``[3C, C]`` (a linear layer's weight: Q rows, then K, then V),
    optional fp32 bias ``b_qkv`` ``[3C]`` and pooled score bias (as for
    ``nystra_biased``).  Returns ``[n_windows, heads, N, C / heads]``."""
    if x.dim() != 3 or w_qkv.dim() != 2:
        raise ValueError("expected x [n_windows, N, C] and w_qkv [3C, C]")
    nw, N, C = x.shape
    if heads < 1 or C % heads:
        raise ValueError(f"C={C} does not split into {heads} heads")
    d = C // heads
    if tuple(w_qkv.shape) != (3 * C, C):
        raise ValueError(f"w_qkv must be [{3 * C}, {C}]")
    out = torch.empty((nw, heads, N, d), dtype=x.dtype, device=x.device) if out is None else out
    for t in (x, w_qkv, out):
        if not t.is_cuda or not t.is_contiguous() or t.dtype != x.dtype:
            raise ValueError("x, w_qkv and out must be contiguous CUDA tensors of one dtype (no CPU path)")
    if x.dtype not in _DTYPE_CODE:
        raise ValueError(f"unsupported dtype {x.dtype}")
    if tuple(out.shape) != (nw, heads, N, d):
        raise ValueError(f"out must be [{nw}, {heads}, {N}, {d}]")
    bp = 0
    if b_qkv is not None:
        if not b_qkv.is_cuda or b_qkv.dtype != torch.float32 or not b_qkv.is_contiguous() or b_qkv.numel() != 3 * C:
            raise ValueError(f"b_qkv must be a contiguous fp32 CUDA tensor of {3 * C} values")
        bp = b_qkv.data_ptr()
    bL = bU = bA = 0
    bw = 0
    if pooled is not None:
        bL, bU, bA = (t.data_ptr() for t in pooled)
        bw = pooled[0].numel() // (heads * N * m)
    with torch.cuda.device(x.device):
        rc = nystra_attention_qkv(x.data_ptr(), w_qkv.data_ptr(), bp, out.data_ptr(), nw, heads, N, d, m, iters,
                                  _lm(landmarks, factors), bL, bU, bA, bw, _DTYPE_CODE[x.dtype], _stream_ptr(stream))
    if rc != NYSTRA_OK:
        raise NystraError(rc, "nystra_attention_qkv")
    return out


def project_qkv(x: torch.Tensor, w_qkv: torch.Tensor, heads: int, b_qkv: torch.Tensor | None = None,
                out=None, stream=None):
    """Q, K, V projections of tokens ``x`` ``[n_windows, N, C]`` by ``w_qkv``
    ``[3C, C]`` (+ optional fp32 ``b_qkv`` ``[3C]``), split into heads: returns
    ``(q, k, v)``, each ``[n_windows, heads, N, C / heads]`` in x's dtype,
    ready for ``nystra``/``exact``.  ``out`` may give the three tensors."""
    if x.dim() != 3 or w_qkv.dim() != 2:
        raise ValueError("expected x [n_windows, N, C] and w_qkv [3C, C]")
    nw, N, C = x.shape
    if heads < 1 or C % heads:
        raise ValueError(f"C={C} does not split into {heads} heads")
    d = C // heads
    if tuple(w_qkv.shape) != (3 * C, C):
        raise ValueError(f"w_qkv must be [{3 * C}, {C}]")
    if out is None:
        out = tuple(torch.empty((nw, heads, N, d), dtype=x.dtype, device=x.device) for _ in range(3))
    for t in (x, w_qkv, *out):
        if not t.is_cuda or not t.is_contiguous() or t.dtype != x.dtype:
            raise ValueError("x, w_qkv and the outputs must be contiguous CUDA tensors of one dtype (no CPU path)")
    if x.dtype not in _DTYPE_CODE:
        raise ValueError(f"unsupported dtype {x.dtype}")
    for t in out:
        if tuple(t.shape) != (nw, heads, N, d):
            raise ValueError(f"outputs must be [{nw}, {heads}, {N}, {d}]")
    bp = 0
    if b_qkv is not None:
        if not b_qkv.is_cuda or b_qkv.dtype != torch.float32 or not b_qkv.is_contiguous() or b_qkv.numel() != 3 * C:
            raise ValueError(f"b_qkv must be a contiguous fp32 CUDA tensor of {3 * C} values")
        bp = b_qkv.data_ptr()
    q, k, v = out
    with torch.cuda.device(x.device):
        rc = nystra_project_qkv(x.data_ptr(), w_qkv.data_ptr(), bp, q.data_ptr(), k.data_ptr(), v.data_ptr(), nw,
                                heads, N, d, _DTYPE_CODE[x.dtype], _stream_ptr(stream))
    if rc != NYSTRA_OK:
        raise NystraError(rc, "nystra_project_qkv")
    return q, k, v
