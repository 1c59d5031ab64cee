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


# ---- bars for ill-conditioned units (sharp attention, long iterations) ----
# The method amplifies any rounding by the conditioning of its landmark block,
# which grows steeply as attention sharpens or the iteration runs past the
# paper's counts.  There the bar of a unit is derived from the float64
# oracle's own response to rounding at the precision the GPU path works in:
# no evaluation at that precision can be held closer to the oracle.

# Relative rounding of the derived factors (landmarks, G_L^n, G_U^n, Y): hi +
# lo pairs keep 16 significant bits in bf16; in fp16 they keep 22 for entries
# of at least 2^-3 of fp16's normal range, but the low part of smaller
# entries (most of G_L^n and G_U^n under sharp attention) falls into fp16's
# subnormal range and keeps fewer, so 16 bits is taken for both.
FACTOR_EPS = {"bf16": 2.0 ** -17, "f16": 2.0 ** -17}


def landmark_sensitivity(q, k, v, m: int, iters: int, eps: float, reps: int = 2, seed: int = 0) -> np.ndarray:
    """Per unit, the oracle's largest relative output change over `reps`
    draws when every landmark coordinate of Qbar and Kbar moves by exactly
    eps relative (each token of a segment scaled by 1 + eps*xi, xi = +-1 per
    segment and feature: the segment mean scales the same way), as rounding
    the landmarks to eps does.  Segment landmarks; float64 throughout."""
    qu, ku, vu = (units_view(torch.as_tensor(x)).double().numpy() for x in (q, k, v))
    U, N, d = qu.shape
    ref = oracle.nystra_attention(qu, ku, vu, m, iters)
    rng = np.random.default_rng(seed)

    def move(x):
        xi = rng.choice([-1.0, 1.0], size=(U, m, 1, d))
        return (x.reshape(U, m, N // m, d) * (1.0 + eps * xi)).reshape(U, N, d)

    out = np.zeros(U)
    for _ in range(reps):
        out = np.maximum(out, per_unit_rel(oracle.nystra_attention(move(qu), move(ku), vu, m, iters), ref))
    return out


def io_ulp_sensitivity(q, k, v, m: int, iters: int, reps: int = 2, seed: int = 0) -> np.ndarray:
    """Per unit, the oracle's largest relative output change over `reps`
    draws when every element of Q, K and V moves one ulp of its I/O type up
    or down (at random)."""
    q, k, v = (torch.as_tensor(x) for x in (q, k, v))
    qu, ku, vu = (units_view(x) for x in (q, k, v))
    ref = oracle.nystra_attention(qu, ku, vu, m, iters)
    g = torch.Generator().manual_seed(seed)

    def move(x):
        up = torch.nextafter(x, torch.full_like(x, float("inf")))
        dn = torch.nextafter(x, torch.full_like(x, -float("inf")))
        return torch.where(torch.rand(x.shape, generator=g) < 0.5, up, dn)

    out = np.zeros(qu.shape[0])
    for _ in range(reps):
        out = np.maximum(out, per_unit_rel(oracle.nystra_attention(move(qu), move(ku), move(vu), m, iters), ref))
    return out


def nystra_float32(q, k, v, m: int, iters: int) -> np.ndarray:
    """Algorithm 1 (segment landmarks, the stabilised blocks of Sec. 2.2, the
    iteration of Razavi et al.) evaluated in float32 with numpy: the accuracy
    any fp32 evaluation of the method reaches, for the fp32 I/O bars."""
    qu, ku, vu = (units_view(torch.as_tensor(x)).float().numpy() for x in (q, k, v))
    U, N, d = qu.shape
    f = np.float32
    s = f(1.0 / np.sqrt(d))
    qb = qu.reshape(U, m, N // m, d).mean(2, dtype=f)
    kb = ku.reshape(U, m, N // m, d).mean(2, dtype=f)
    SL = s * (qu @ kb.transpose(0, 2, 1))
    SU = s * (qb @ ku.transpose(0, 2, 1))
    SA = s * (qb @ kb.transpose(0, 2, 1))
    mU = SU.max(-1, keepdims=True)
    GL = np.exp(SL - SL.max(-1, keepdims=True))
    GU = np.exp(SU - mU)
    A = np.exp(SA - mU)
    Z = A.transpose(0, 2, 1) / (np.abs(A).sum(1).max(-1) * np.abs(A).sum(2).max(-1))[:, None, None]
    eye = np.eye(m, dtype=f)
    for _ in range(iters):
        X = A @ Z
        Z = f(0.25) * (Z @ (f(13) * eye - X @ (f(15) * eye - X @ (f(7) * eye - X))))
    P = GL @ Z
    num = P @ (GU @ vu)
    den = P @ GU.sum(-1, keepdims=True)
    return (num / den).astype(np.float64)
