"""The multi-core CPU path (``libnystra_host.so``, C ABI in
``include/nystra_host.h``): PnP-Nystra and exact window attention in fp32 on
the host cores, for CPU deployments (the paper reports CPU speedups too).

A separate library with separate entry points: the GPU binding never calls
it, and it is not a fallback for the GPU path.  Argument marshalling only.

    python -m paper_2506_08520_gb300.host [workload] [--threads T] [--units U]

times both on a sample of a workload's units and prints one JSON line.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import time

import torch

from . import binding, workloads

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libnystra_host.so")
_lib = None


def lib() -> ctypes.CDLL:
    """The loaded CPU library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with `python -m paper_2506_08520_gb300.build`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i = ctypes.c_void_p, ctypes.c_int
        L.nystra_attention_host.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, i]
        L.nystra_attention_host.restype = i
        L.exact_window_attention_host.argtypes = [vp, vp, vp, vp, i, i, i, i, i]
        L.exact_window_attention_host.restype = i
        L.nystra_pool_bias_host.argtypes = [vp, i, i, i, i, vp, vp, vp, i]
        L.nystra_pool_bias_host.restype = i
        L.nystra_attention_bias_host.argtypes = [vp, vp, vp, vp, i, i, i, i, i, i, i, vp, vp, vp, i, i]
        L.nystra_attention_bias_host.restype = i
        L.nystra_host_threads.restype = i
        L.nystra_host_exp.argtypes = [vp, vp, i]
        L.nystra_host_exp.restype = None
        _lib = L
    return _lib


def threads() -> int:
    return lib().nystra_host_threads()


def exp(x: torch.Tensor) -> torch.Tensor:
    """The CPU path's exponential on a contiguous float32 CPU tensor (test-only)."""
    if x.device.type != "cpu" or x.dtype != torch.float32 or not x.is_contiguous():
        raise ValueError("exp takes a contiguous float32 CPU tensor")
    y = torch.empty_like(x)
    lib().nystra_host_exp(x.data_ptr(), y.data_ptr(), x.numel())
    return y


def _check(q, k, v, out):
    for t in (q, k, v, out):
        if t.device.type != "cpu" or t.dtype != torch.float32 or not t.is_contiguous():
            raise ValueError("the CPU path takes contiguous float32 CPU tensors")
    if q.shape != k.shape or q.shape != v.shape or q.shape != out.shape or q.dim() != 4:
        raise ValueError("q, k, v, out must share one [n_windows, heads, N, d_h] shape")


def nystra(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, m: int = 16, iters: int = 6,
           landmarks: str = "segments", out: torch.Tensor | None = None, n_threads: int = 0) -> torch.Tensor:
    """PnP-Nystra attention of float32 CPU tensors ``[n_windows, heads, N, d_h]``."""
    out = torch.empty_like(q) if out is None else out
    _check(q, k, v, out)
    nw, h, N, d = q.shape
    rc = lib().nystra_attention_host(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), nw, h, N, d, m,
                                     iters, binding.LANDMARKS[landmarks], n_threads)
    if rc != binding.NYSTRA_OK:
        raise RuntimeError(f"nystra_attention_host: status {rc}")
    return out


def pool_bias(bias: torch.Tensor, m: int, landmarks: str = "segments", n_threads: int = 0):
    """The landmark blocks ``(bias_L [n, N, m], bias_U [n, m, N], bias_A [n, m, m])``
    of float32 CPU score biases ``bias`` ``[n, N, N]`` (per head, or per window
    and head), for ``nystra_biased``."""
    if bias.device.type != "cpu" or bias.dtype != torch.float32 or not bias.is_contiguous() or bias.dim() != 3:
        raise ValueError("bias must be a contiguous float32 CPU tensor [n, N, N]")
    n, N, _ = bias.shape
    L = torch.empty(n, N, m)
    U = torch.empty(n, m, N)
    A = torch.empty(n, m, m)
    rc = lib().nystra_pool_bias_host(bias.data_ptr(), n, N, m, binding.LANDMARKS[landmarks], L.data_ptr(),
                                     U.data_ptr(), A.data_ptr(), n_threads)
    if rc != binding.NYSTRA_OK:
        raise RuntimeError(f"nystra_pool_bias_host: status {rc}")
    return L, U, A


def nystra_biased(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, pooled, m: int = 16, iters: int = 6,
                  landmarks: str = "segments", out: torch.Tensor | None = None, n_threads: int = 0) -> torch.Tensor:
    """PnP-Nystra with a pooled score bias (``pool_bias``): slices per head
    (``heads`` slices, shared by every window) or per window and head."""
    out = torch.empty_like(q) if out is None else out
    _check(q, k, v, out)
    nw, h, N, d = q.shape
    L, U, A = pooled
    bw = L.shape[0] // h
    rc = lib().nystra_attention_bias_host(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), nw, h, N, d, m,
                                          iters, binding.LANDMARKS[landmarks], L.data_ptr(), U.data_ptr(),
                                          A.data_ptr(), bw, n_threads)
    if rc != binding.NYSTRA_OK:
        raise RuntimeError(f"nystra_attention_bias_host: status {rc}")
    return out


def exact(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, out: torch.Tensor | None = None,
          n_threads: int = 0) -> torch.Tensor:
    """Exact softmax window attention (Eq. 1) of float32 CPU tensors."""
    out = torch.empty_like(q) if out is None else out
    _check(q, k, v, out)
    nw, h, N, d = q.shape
    rc = lib().exact_window_attention_host(q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(), nw, h, N, d,
                                           n_threads)
    if rc != binding.NYSTRA_OK:
        raise RuntimeError(f"exact_window_attention_host: status {rc}")
    return out


def _rate(fn, units_tokens: int, min_s: float = 1.0) -> float:
    fn()
    n, t0 = 0, time.perf_counter()
    while True:
        fn()
        n += 1
        dt = time.perf_counter() - t0
        if dt >= min_s:
            return units_tokens * n / dt


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("workload", nargs="?", default="sr720p-w32-m16-bf16")
    ap.add_argument("--threads", type=int, default=0)
    ap.add_argument("--units", type=int, default=512, help="units sampled from the workload (its first windows)")
    args = ap.parse_args(argv)
    wl = workloads.WORKLOADS[args.workload]
    q, k, v = (x.float() for x in workloads.make_qkv(wl))
    nw = max(1, min(wl.n_windows, -(-args.units // wl.heads)))
    q, k, v = (x[:nw].contiguous() for x in (q, k, v))
    units_tokens = nw * wl.heads * wl.N
    o = torch.empty_like(q)
    r_ny = _rate(lambda: nystra(q, k, v, wl.m, wl.iters, wl.landmarks, out=o, n_threads=args.threads), units_tokens)
    r_ex = _rate(lambda: exact(q, k, v, out=o, n_threads=args.threads), units_tokens)
    print(json.dumps({"workload": wl.name, "units": nw * wl.heads, "N": wl.N, "d_h": wl.d, "m": wl.m,
                      "iters": wl.iters, "threads": args.threads if args.threads > 0 else threads(),
                      "nystra_tokens_heads_per_s": r_ny, "exact_tokens_heads_per_s": r_ex,
                      "speedup": r_ny / r_ex, "dtype": "f32", "device": "host cores"}))
    return 0


if __name__ == "__main__":
    raise SystemExit(main())
