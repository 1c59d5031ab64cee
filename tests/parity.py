"""Helpers shared by the GPU parity tests: run the CUDA path, run the oracle on
the same (upcast) inputs, and compare per unit."""
import numpy as np
import torch

import oracle
from paper_2506_08520_gb300 import binding

# Max over units of ||O_gpu - O_ref||_F / ||O_ref||_F.
TOL = {"f32": 1e-4, "bf16": 2e-2, "f16": 2e-2}
DT = {torch.float32: "f32", torch.bfloat16: "bf16", torch.float16: "f16"}


def per_unit_rel(out: np.ndarray, ref: np.ndarray) -> np.ndarray:
    N, d = ref.shape[-2:]
    o = out.reshape(-1, N * d)
    r = ref.reshape(-1, N * d)
    return np.linalg.norm(o - r, axis=1) / np.linalg.norm(r, axis=1)


def gpu_nystra(q, k, v, m, iters, landmarks="segments"):
    qd, kd, vd = (x.cuda() for x in (q, k, v))
    out = binding.nystra(qd, kd, vd, m=m, iters=iters, landmarks=landmarks)
    torch.cuda.synchronize()
    return out


def gpu_exact(q, k, v):
    qd, kd, vd = (x.cuda() for x in (q, k, v))
    out = binding.exact(qd, kd, vd)
    torch.cuda.synchronize()
    return out


def units_view(x: torch.Tensor) -> torch.Tensor:
    return x.reshape(-1, x.shape[-2], x.shape[-1])


def sample_units(n_units: int, k: int = 384, seed: int = 0) -> np.ndarray:
    """All units if few, else the first and last, an even stride and random picks."""
    if n_units <= k:
        return np.arange(n_units)
    rng = np.random.default_rng(seed)
    idx = np.concatenate([[0, n_units - 1], np.linspace(0, n_units - 1, k // 2).astype(int),
                          rng.choice(n_units, k // 2 - 2, replace=False)])
    return np.unique(idx)


def check_nystra(q, k, v, m, iters, sample=None, landmarks="segments"):
    """Run GPU on everything, the oracle on the sampled units; return (max err, worst unit)."""
    out = units_view(gpu_nystra(q, k, v, m, iters, landmarks).cpu())
    qu, ku, vu = units_view(q), units_view(k), units_view(v)
    idx = np.arange(qu.shape[0]) if sample is None else sample
    ref = oracle.nystra_attention(qu[idx], ku[idx], vu[idx], m, iters, landmarks)
    got = out[idx].double().numpy()
    assert np.isfinite(got).all(), "non-finite GPU output"
    err = per_unit_rel(got, ref)
    w = int(np.argmax(err))
    return float(err[w]), int(idx[w])


def check_exact(q, k, v, sample=None):
    out = units_view(gpu_exact(q, k, v).cpu())
    qu, ku, vu = units_view(q), units_view(k), units_view(v)
    idx = np.arange(qu.shape[0]) if sample is None else sample
    ref = oracle.exact_attention(qu[idx], ku[idx], vu[idx])
    err = per_unit_rel(out[idx].double().numpy(), ref)
    w = int(np.argmax(err))
    return float(err[w]), int(idx[w])
