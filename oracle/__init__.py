"""Float64 CPU oracle for PnP-Nystra window attention (arXiv 2506.08520).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package.  The product
path (``paper_2506_08520_gb300``) never imports, links or runs it, and the
two share no code: the oracle is plain C in ``nystra_oracle.c`` (Algorithm 1
with the row-max stabilisation of Sec. 2.2, in float64), wrapped here with
ctypes.

Inputs may be numpy arrays or torch tensors of any float dtype; they are
upcast exactly to float64.  Shapes are ``[..., N, d]`` with all leading axes
flattened into independent units (one unit = one (window, head) pair).

Every function here is pinned by ``tests/test_oracle_pins.py`` against
properties the paper or the mathematics fixes (brute force, exact recovery,
the iteration's residual recursion, invariances, the spectral bound).
"""
import ctypes
import numpy as np

from . import build as _build

_lib = None
_D = ctypes.POINTER(ctypes.c_double)


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(_build.build())
        lib.oracle_threads.restype = ctypes.c_int
        lib.oracle_exact_attention.argtypes = [_D, _D, _D, _D, ctypes.c_long, ctypes.c_int, ctypes.c_int]
        lib.oracle_exact_attention.restype = None
        lib.oracle_exact_attention_bias.argtypes = [_D, _D, _D, _D, ctypes.c_long, ctypes.c_int, ctypes.c_int, _D]
        lib.oracle_exact_attention_bias.restype = None
        lib.oracle_nystra_attention_bias.argtypes = [_D, _D, _D, _D, ctypes.c_long, ctypes.c_int, ctypes.c_int,
                                                     ctypes.c_int, ctypes.c_int, ctypes.c_int, _D]
        lib.oracle_nystra_attention_bias.restype = ctypes.c_int
        lib.oracle_pool_bias.argtypes = [_D, ctypes.c_int, ctypes.c_int, ctypes.c_int, _D, _D, _D]
        lib.oracle_pool_bias.restype = None
        lib.oracle_nystra_attention.argtypes = [_D, _D, _D, _D, ctypes.c_long, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_int, ctypes.c_int]
        lib.oracle_nystra_attention.restype = ctypes.c_int
        lib.oracle_nystra_attention_pool.argtypes = [_D, _D, _D, _D, ctypes.c_long, ctypes.c_int,
                                                     ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int]
        lib.oracle_nystra_attention_pool.restype = ctypes.c_int
        lib.oracle_landmarks.argtypes = [_D, ctypes.c_int, ctypes.c_int, ctypes.c_int, _D]
        lib.oracle_landmarks.restype = None
        lib.oracle_landmarks_patches.argtypes = [_D, ctypes.c_int, ctypes.c_int, ctypes.c_int, _D]
        lib.oracle_landmarks_patches.restype = None
        lib.oracle_pinv_iteration.argtypes = [_D, ctypes.c_int, ctypes.c_int, _D]
        lib.oracle_pinv_iteration.restype = None
        lib.oracle_nystra_stages.argtypes = [_D, _D, _D, _D, ctypes.c_int, ctypes.c_int,
                                             ctypes.c_int, ctypes.c_int, ctypes.c_int] + [_D] * 10
        lib.oracle_nystra_stages.restype = ctypes.c_int
        _lib = lib
    return _lib


def _f64(x) -> np.ndarray:
    if hasattr(x, "detach"):  # torch tensor: exact upcast, then to numpy
        x = x.detach().to("cpu").double().numpy()
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


def _p(a: np.ndarray):
    return a.ctypes.data_as(_D)


def threads() -> int:
    """Host threads the oracle's OpenMP loops use."""
    return int(_load().oracle_threads())


def _bias(bias, q):
    """An additive score bias ``[..., N, N]`` broadcast over the units of q."""
    N = q.shape[-2]
    b = np.broadcast_to(_f64(bias), q.shape[:-2] + (N, N))
    return np.ascontiguousarray(b)


def exact_attention(q, k, v, bias=None) -> np.ndarray:
    """Exact softmax attention, Eq. (1), per unit; float64 ``[..., N, d]``.
    ``bias``: optional additive score bias ``[..., N, N]`` (before the softmax)."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    N, d = q.shape[-2], q.shape[-1]
    out = np.empty_like(q)
    if bias is None:
        _load().oracle_exact_attention(_p(q), _p(k), _p(v), _p(out), q.size // (N * d), N, d)
    else:
        b = _bias(bias, q)
        _load().oracle_exact_attention_bias(_p(q), _p(k), _p(v), _p(out), q.size // (N * d), N, d, _p(b))
    return out


POOLS = {"segments": 0, "patches": 1}


def nystra_attention(q, k, v, m: int, iters: int, pool: str = "segments", bias=None) -> np.ndarray:
    """PnP-Nystra output (Algorithm 1, stabilised form), float64 ``[..., N, d]``.

    ``pool``: "segments" (m contiguous token runs) or "patches" (a square
    window pooled over a square grid of m square patches).  ``bias``: optional
    additive score bias ``[..., N, N]``, seen by the landmark blocks as the mean
    over each landmark's tokens."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    N, d = q.shape[-2], q.shape[-1]
    out = np.empty_like(q)
    b = None if bias is None else _bias(bias, q)
    rc = _load().oracle_nystra_attention_bias(_p(q), _p(k), _p(v), _p(out), q.size // (N * d),
                                              N, d, int(m), int(iters), POOLS[pool],
                                              None if b is None else _p(b))
    if rc != 0:
        raise ValueError(f"oracle: invalid m={m} for N={N} with {pool} pooling, iters={iters}")
    return out


def landmarks(x, m: int, pool: str = "segments") -> np.ndarray:
    """Landmarks of one unit ``[N, d]`` -> ``[m, d]`` (Alg. 1 step 1): segment
    means, or with ``pool="patches"`` square-patch means of a square window."""
    x = _f64(x)
    N, d = x.shape
    out = np.empty((m, d))
    if pool == "patches":
        w, p = int(round(N ** 0.5)), int(round(m ** 0.5))
        if w * w != N or p * p != m or w % p:
            raise ValueError(f"oracle: {m} square patches do not tile a window of {N} tokens")
        _load().oracle_landmarks_patches(_p(x), N, d, int(m), _p(out))
    else:
        _load().oracle_landmarks(_p(x), N, d, int(m), _p(out))
    return out


def pool_bias(B, m: int, pool: str = "segments"):
    """One unit's score bias ``[N, N]`` through the landmarks: (B_L ``[N, m]``,
    B_U ``[m, N]``, B_A ``[m, m]``), each entry the mean over the landmarks' tokens."""
    B = _f64(B)
    N = B.shape[0]
    BL, BU, BA = np.empty((N, m)), np.empty((m, N)), np.empty((m, m))
    _load().oracle_pool_bias(_p(B), N, int(m), POOLS[pool], _p(BL), _p(BU), _p(BA))
    return BL, BU, BA


def pinv_iteration(A, iters: int) -> np.ndarray:
    """Iterative pseudo-inverse of a square matrix (Alg. 1 step 4)."""
    A = _f64(A)
    m = A.shape[0]
    Z = np.empty_like(A)
    _load().oracle_pinv_iteration(_p(A), m, int(iters), _p(Z))
    return Z


def nystra_stages(q, k, v, m: int, iters: int, pool: str = "segments") -> dict:
    """All intermediates of one unit (``q, k, v``: ``[N, d]``)."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    N, d = q.shape
    st = {
        "qbar": np.empty((m, d)), "kbar": np.empty((m, d)), "mL": np.empty(N), "mU": np.empty(m),
        "GLn": np.empty((N, m)), "GUn": np.empty((m, N)), "GAn": np.empty((m, m)),
        "Z": np.empty((m, m)), "num": np.empty((N, d)), "den": np.empty(N),
    }
    out = np.empty((N, d))
    order = ["qbar", "kbar", "mL", "mU", "GLn", "GUn", "GAn", "Z", "num", "den"]
    rc = _load().oracle_nystra_stages(_p(q), _p(k), _p(v), _p(out), N, d, int(m), int(iters), POOLS[pool],
                                      *[_p(st[n]) for n in order])
    if rc != 0:
        raise ValueError(f"oracle: invalid m={m} for N={N} with {pool} pooling")
    st["out"] = out
    return st


def project_qkv(x, w_qkv, b_qkv, heads: int):
    """The projections of Eq. (1), Q = X W_Q, K = X W_K, V = X W_V, for every
    window, split into heads.  ``x``: ``[n_windows, N, C]`` tokens, C = heads*d.
    ``w_qkv``: ``[3C, C]``, the transposes of W_Q, W_K, W_V stacked (row o holds
    output feature o: the layout of a linear layer's weight), so Q[:, f] is
    x @ w_qkv[f] and K, V take rows C + f and 2C + f.  ``b_qkv``: optional
    ``[3C]`` bias of the restoration models' projection layers (Eq. (1) has
    none).  Head h owns features h*d .. h*d + d - 1 of each.  Returns float64
    q, k, v ``[n_windows, heads, N, d]``."""
    x, w = _f64(x), _f64(w_qkv)
    nw, N, C = x.shape
    if C % heads or w.shape != (3 * C, C):
        raise ValueError(f"oracle: w_qkv {w.shape} does not project C={C} for {heads} heads")
    y = x @ w.T  # [nw, N, 3C]
    if b_qkv is not None:
        y = y + _f64(b_qkv)
    y = y.reshape(nw, N, 3, heads, C // heads).transpose(2, 0, 3, 1, 4)
    return tuple(np.ascontiguousarray(y[i]) for i in range(3))


def nystra_attention_qkv(x, w_qkv, b_qkv, heads: int, m: int, iters: int, pool: str = "segments",
                         bias=None) -> np.ndarray:
    """PnP-Nystra of the projected tokens: project_qkv, then nystra_attention.
    float64 ``[n_windows, heads, N, d]``."""
    q, k, v = project_qkv(x, w_qkv, b_qkv, heads)
    return nystra_attention(q, k, v, m, iters, pool, bias)
