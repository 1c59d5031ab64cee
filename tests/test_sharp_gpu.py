"""GPU parity as attention sharpens: Q and K scaled by s (logit standard
deviation s^2; the configurations' inputs have about 1).

The method amplifies rounding by the conditioning of its landmark block
G_A^n, which grows steeply with s: at s = 2 a few units in a hundred are so
ill-conditioned that moving each landmark coordinate by one part in 2^17
moves the float64 oracle's own output by 10% to 300%.  On such a unit no
evaluation that carries the factors with 16 significant bits can be held to a
fixed bar, so each unit's bar is the larger of the fixed one and the oracle's
own response to rounding at the GPU path's working precision (tests/parity.py
defines the perturbations); every other unit keeps the fixed bar.  Every path
must stay finite wherever the oracle is.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_08520_gb300 import binding, workloads
from tests.parity import (FACTOR_EPS, TOL, landmark_sensitivity, nystra_float32, per_unit_rel, units_view)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2506_08520_gb300 import build
    build.build()


def _sharp(units, N, d, dtype, s, seed):
    q, k, v = workloads.random_qkv(units, N, d, "f32", seed=seed)
    T = workloads.DTYPES[dtype]
    return (q * s).to(T), (k * s).to(T), v.to(T)


def _errors(q, k, v, m, iters, factors="pairs"):
    out = binding.nystra(q.cuda(), k.cuda(), v.cuda(), m=m, iters=iters, factors=factors)
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    got = units_view(out.cpu()).double().numpy()
    ref = oracle.nystra_attention(units_view(q), units_view(k), units_view(v), m, iters)
    return got, ref


# Every tensor-core kernel family with 16-bit I/O: the stage-pool kernel
# (8x8 windows), the team kernel (16x16), the streaming kernel (32x32), each
# with the one-warp core (m <= 16) and, where it has one, the distributed core
# (m = 32); the grouped kernel (m = 32 at 8x8 and, with d_h = 32, at 16x16;
# every m = 64).
FAMILIES = [
    # N, d, m, dtype, units
    (64, 30, 16, "bf16", 48), (64, 32, 8, "f16", 48),
    (256, 30, 16, "bf16", 32), (256, 32, 8, "f16", 32), (256, 30, 32, "bf16", 32),
    (1024, 30, 16, "bf16", 12), (1024, 32, 16, "f16", 12), (1024, 30, 32, "bf16", 12),
    (64, 30, 32, "bf16", 48), (256, 32, 32, "f16", 32),
    (64, 30, 64, "bf16", 32), (256, 30, 64, "bf16", 32), (1024, 32, 64, "f16", 12),
]


@pytest.mark.parametrize("N,d,m,dtype,units", FAMILIES)
def test_paired_factors_at_logit_std_4(N, d, m, dtype, units):
    # s = 2.  The derived factors are hi + lo pairs (FACTOR_EPS relative
    # rounding); a unit's bar is max(fixed bar, the oracle's change when its
    # landmarks are rounded once to that precision).
    q, k, v = _sharp(units, N, d, dtype, 2.0, N * 3 + m + d + 7)
    got, ref = _errors(q, k, v, m, 6)
    assert np.isfinite(got).all()
    err = per_unit_rel(got, ref)
    delta = landmark_sensitivity(q, k, v, m, 6, FACTOR_EPS[dtype])
    bar = np.maximum(TOL[dtype], delta)
    worst = int(np.argmax(err / bar))
    print(f"N={N} m={m} {dtype}: max err {err.max():.2e}, {int((err > TOL[dtype]).sum())} of {units} units above "
          f"{TOL[dtype]} (their landmark sensitivity {delta[err > TOL[dtype]]})")
    assert (err <= bar).all(), f"unit {worst}: err {err[worst]:.3e} > bar {bar[worst]:.3e}"
    # the bulk holds the fixed bar
    assert np.median(err) <= TOL[dtype] / 4


@pytest.mark.parametrize("N,d,m", [(64, 30, 16), (64, 32, 8), (256, 30, 16), (48, 20, 12)])
def test_fp32_at_logit_std_4(N, d, m):
    # fp32 I/O: the 8x8 tensor-core path splits inputs and factors into bf16
    # pairs, the SIMT path (other shapes) is fp32 throughout.  A unit's bar is
    # max(1e-4, 4 x the error of the same algorithm evaluated in float32),
    # and, on the tensor-core path, 2 x its landmark sensitivity at the pairs'
    # 2^-17 (inputs and factors are both rounded to pairs).
    q, k, v = _sharp(16, N, d, "f32", 2.0, N + m + d)
    got, ref = _errors(q, k, v, m, 6)
    assert np.isfinite(got).all()
    err = per_unit_rel(got, ref)
    e32 = per_unit_rel(nystra_float32(q, k, v, m, 6), ref)
    bar = np.maximum(TOL["f32"], 4.0 * e32)
    if N == 64 and m <= 16:
        bar = np.maximum(bar, 2.0 * landmark_sensitivity(q, k, v, m, 6, 2.0 ** -17))
    worst = int(np.argmax(err / bar))
    print(f"f32 N={N} m={m}: max err {err.max():.2e}, float32 evaluation {e32.max():.2e}")
    assert (err <= bar).all(), f"unit {worst}: err {err[worst]:.3e} > bar {bar[worst]:.3e}"


@pytest.mark.parametrize("factors", ["pairs", "16"])
@pytest.mark.parametrize("s", [3.0, 4.0, 6.0])
@pytest.mark.parametrize("N,d,m,dtype", [(64, 30, 16, "bf16"), (64, 32, 8, "f16"), (256, 30, 16, "bf16"),
                                         (256, 30, 32, "bf16"), (1024, 30, 16, "bf16"), (1024, 32, 32, "f16"),
                                         (64, 30, 32, "bf16"), (256, 32, 32, "f16"), (256, 30, 64, "bf16"),
                                         (1024, 32, 64, "bf16"), (64, 30, 16, "f32"), (256, 30, 16, "f32")])
def test_finite_wherever_the_oracle_is(N, d, m, dtype, s, factors):
    # logit std up to 36: exponentials of whole rows of G_A^n fall far below
    # fp32's range unless the scale enters the exponent first; no path may
    # return inf or NaN where the float64 oracle is finite
    if dtype == "f32" and factors == "16":
        pytest.skip("NYSTRA_FACTORS_16 concerns 16-bit I/O only")
    q, k, v = _sharp(8, N, d, dtype, s, N + m + d + int(s))
    got, ref = _errors(q, k, v, m, 6, factors)
    fin = np.isfinite(ref).all(axis=(1, 2))
    assert np.isfinite(got[fin]).all()


@pytest.mark.parametrize("N,d,m,dtype", [(64, 30, 16, "bf16"), (64, 32, 8, "f16"), (256, 30, 16, "bf16"),
                                         (1024, 30, 16, "bf16"), (1024, 32, 32, "f16"), (256, 32, 32, "bf16"),
                                         (256, 30, 64, "bf16")])
def test_factors16_within_the_bar_for_soft_attention(N, d, m, dtype):
    # NYSTRA_FACTORS_16 rounds the derived factors to the I/O type: the bar
    # holds for logit std up to about 1.5 (s = 1.25), as nystra.h states
    q, k, v = _sharp(16, N, d, dtype, 1.25, N + m + d + 3)
    got, ref = _errors(q, k, v, m, 6, "16")
    err = per_unit_rel(got, ref)
    assert err.max() <= TOL[dtype], f"max rel err {err.max():.3e} at unit {int(np.argmax(err))}"


def test_factors16_is_the_single_rounding_path():
    # the two factor precisions are different kernels: on soft inputs both
    # meet the bar, and the paired factors are at least as close to the oracle
    q, k, v = _sharp(48, 1024, 30, "bf16", 1.0, 11)
    got2, ref = _errors(q, k, v, 16, 6, "pairs")
    got1, _ = _errors(q, k, v, 16, 6, "16")
    e2, e1 = per_unit_rel(got2, ref), per_unit_rel(got1, ref)
    assert not np.array_equal(got1, got2)
    assert e2.max() <= TOL["bf16"] and e1.max() <= TOL["bf16"]
    assert np.median(e2) <= np.median(e1)
