"""The multi-core CPU path (libnystra_host.so, fp32) against the float64
oracle on the same inputs: PnP-Nystra within the fp32 bar of 1e-4 per unit
(max relative Frobenius error) at the paper's iteration counts, exact
attention within 1e-5, over both landmark poolings, several shapes, ragged
sizes and edge cases; results independent of the thread count; argument
checks."""
import pytest
import torch

import oracle
from paper_2506_08520_gb300 import binding, build, host, workloads
from tests.parity import per_unit_rel


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build_host()


def _units(x):
    return x.reshape(-1, x.shape[-2], x.shape[-1])


def _qkv(units, N, d, seed, scale=1.0):
    q, k, v = workloads.random_qkv(units, N, d, "f32", seed=seed, scale=scale)
    return tuple(x.reshape(1, units, N, d).contiguous() for x in (q, k, v))


CASES = [  # units, N, d, m, iters, pooling
    (6, 64, 30, 16, 6, "segments"),
    (4, 64, 32, 8, 6, "segments"),
    (3, 256, 30, 16, 6, "segments"),
    (2, 256, 32, 32, 4, "segments"),
    (2, 1024, 30, 16, 6, "segments"),
    (2, 1024, 30, 64, 6, "segments"),
    (3, 48, 20, 12, 6, "segments"),     # ragged: no power of two anywhere
    (3, 10, 7, 5, 3, "segments"),
    (5, 64, 30, 16, 0, "segments"),     # Z_0 only
    (5, 64, 30, 16, 1, "segments"),
    (4, 64, 30, 16, 6, "patches"),      # 2x2 patches of the 8x8 window
    (2, 256, 30, 16, 6, "patches"),     # 4x4 patches of 16x16
    (2, 144, 12, 16, 6, "patches"),     # 3x3 patches of 12x12
    (3, 64, 30, 64, 6, "segments"),     # m = N: every token its own landmark
]


@pytest.mark.parametrize("units,N,d,m,iters,pool", CASES)
def test_host_nystra_matches_the_oracle(units, N, d, m, iters, pool):
    q, k, v = _qkv(units, N, d, seed=units * 31 + N + d + m + iters)
    got = host.nystra(q, k, v, m, iters, pool)
    ref = oracle.nystra_attention(_units(q), _units(k), _units(v), m, iters, pool)
    err = per_unit_rel(_units(got).double().numpy(), ref)
    assert err.max() <= 1e-4, f"max rel err {err.max():.3e} at unit {int(err.argmax())}"


@pytest.mark.parametrize("units,N,d", [(4, 64, 30), (2, 256, 32), (1, 1024, 30), (3, 10, 7)])
def test_host_exact_matches_the_oracle(units, N, d):
    q, k, v = _qkv(units, N, d, seed=N + d)
    got = host.exact(q, k, v)
    ref = oracle.exact_attention(_units(q), _units(k), _units(v))
    err = per_unit_rel(_units(got).double().numpy(), ref)
    assert err.max() <= 1e-5, f"max rel err {err.max():.3e}"


def test_host_workload_sample_matches_the_oracle():
    # the 1280x720 map with 32x32 windows, m = 16: a sample of its units
    wl = workloads.WORKLOADS["sr720p-w32-m16-bf16"]
    q, k, v = (x[:3].float().contiguous() for x in workloads.make_qkv(wl))
    got = host.nystra(q, k, v, wl.m, wl.iters)
    ref = oracle.nystra_attention(_units(q), _units(k), _units(v), wl.m, wl.iters)
    err = per_unit_rel(_units(got).double().numpy(), ref)
    assert err.max() <= 1e-4, f"max rel err {err.max():.3e}"


def test_host_results_do_not_depend_on_the_thread_count():
    q, k, v = _qkv(12, 256, 30, seed=4)
    a = host.nystra(q, k, v, 16, 6, n_threads=1)
    b = host.nystra(q, k, v, 16, 6, n_threads=4)
    assert torch.equal(a, b)
    assert torch.equal(host.exact(q, k, v, n_threads=1), host.exact(q, k, v, n_threads=3))


def test_host_units_are_independent():
    q, k, v = _qkv(6, 64, 30, seed=8)
    perm = torch.tensor([3, 0, 5, 1, 4, 2])
    a = host.nystra(q, k, v, 16, 6)
    b = host.nystra(*(x[:, perm].contiguous() for x in (q, k, v)), 16, 6)
    assert torch.equal(a[:, perm], b)


def test_host_nystra_tracks_exact_attention_with_many_landmarks():
    # m = N with a converged iteration recovers exact attention (the oracle's
    # pin, here on the CPU path itself)
    q, k, v = _qkv(3, 16, 8, seed=2, scale=0.5)
    ny = host.nystra(q, k, v, 16, 40)
    ex = host.exact(q, k, v)
    err = per_unit_rel(_units(ny).double().numpy(), _units(ex).double().numpy())
    assert err.max() <= 1e-4, f"max rel err {err.max():.3e}"


def test_host_argument_validation():
    L = host.lib()
    P = 1 << 20
    ok, inv = binding.NYSTRA_OK, binding.NYSTRA_EINVAL
    f = L.nystra_attention_host
    assert f(P, 2 * P, 3 * P, 64 * P, 0, 2, 64, 30, 16, 6, 0, 0) == ok       # empty: no-op
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 15, 6, 0, 0) == inv      # m does not divide N
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 2048, 30, 16, 6, 0, 0) == inv    # N > 1024
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 65, 16, 6, 0, 0) == inv      # d_h > 64
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 101, 0, 0) == inv    # iterations
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 8, 6, 1, 0) == inv       # 8 landmarks are no square grid
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 6, 2, 0) == inv      # no such pooling
    assert f(0, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 6, 0, 0) == inv      # null input
    assert f(P, 2 * P, 3 * P, P + 64, 4, 2, 64, 30, 16, 6, 0, 0) == inv      # out overlaps q
    g = L.exact_window_attention_host
    assert g(P, 2 * P, 3 * P, 64 * P, 0, 2, 64, 30, 0) == ok
    assert g(P, 2 * P, 3 * P, 64 * P, 4, 2, 0, 30, 0) == inv
    assert g(P, 2 * P, 3 * P, 2 * P + 4, 4, 2, 64, 30, 0) == inv
    assert host.threads() >= 1
    with pytest.raises(ValueError):
        host.nystra(*(torch.zeros(1, 1, 64, 30, dtype=torch.bfloat16) for _ in range(3)))


def test_host_exp_is_within_two_ulp_of_exp():
    # the CPU path's own exponential (Cody-Waite reduction, degree-7 Taylor
    # polynomial) against float64 exp rounded to float32, over the softmax's
    # argument range (x <= 0: scores minus their row maximum) into the
    # subnormal results, and a little above 0
    import numpy as np
    x = np.concatenate([np.linspace(-104.0, 2.0, 2_000_003), -np.logspace(-8, 0, 10_001),
                        np.linspace(-1e-3, 1e-3, 10_001)]).astype(np.float32)
    y = host.exp(torch.from_numpy(x)).numpy()
    ref = np.exp(x.astype(np.float64))
    ref32 = ref.astype(np.float32)
    ulp = np.spacing(ref32).astype(np.float64)  # float32 spacing (2^-149 in the subnormal range)
    err = np.abs(y.astype(np.float64) - ref) / ulp
    assert err.max() <= 2.0, (float(err.max()), float(x[err.argmax()]))
    # exact and special values
    sp = torch.tensor([0.0, -0.0, float("-inf"), -105.0, -1e30, float("nan"), -103.9], dtype=torch.float32)
    ys = host.exp(sp)
    assert ys[0] == 1.0 and ys[1] == 1.0
    assert ys[2] == 0.0 and ys[3] == 0.0 and ys[4] == 0.0
    assert torch.isnan(ys[5])
    assert 0.0 < ys[6] < 1e-44  # a subnormal result, not flushed
    assert host.exp(torch.zeros(0)).numel() == 0


def test_host_library_exports_every_declared_symbol():
    import ctypes
    import os
    import re
    hdr = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                            "nystra_host.h")).read()
    names = re.findall(r"NYSTRA_API\s+[\w\s\*]+?\b(\w+)\s*\(", hdr)
    assert {"nystra_attention_host", "exact_window_attention_host", "nystra_host_threads"} <= set(names)
    raw = ctypes.CDLL(host.LIB_PATH)
    for name in names:
        assert hasattr(raw, name), f"{name} declared in nystra_host.h but not exported"


@pytest.mark.parametrize("N,m,pool,per_window", [(64, 16, "segments", False), (256, 16, "segments", True),
                                                 (256, 16, "patches", False), (64, 8, "segments", True)])
def test_host_score_bias_matches_the_oracle(N, m, pool, per_window):
    # a relative-position bias (one per head, or one per window and head) pooled
    # into its landmark blocks on the CPU, then PnP-Nystra with it
    nw, heads, d = 3, 2, 30
    w = int(round(N ** 0.5))
    q, k, v = (x.reshape(nw, heads, N, d).contiguous()
               for x in workloads.random_qkv(nw * heads, N, d, "f32", seed=N + m))
    b = torch.from_numpy(workloads.relpos_bias(w, heads, seed=7)).float()  # [heads, N, N]
    if per_window:
        b = (b[None] + 0.5 * torch.randn(nw, heads, N, N, generator=torch.Generator().manual_seed(3))).reshape(
            nw * heads, N, N).contiguous()
    pooled = host.pool_bias(b.contiguous(), m, pool)
    got = host.nystra_biased(q, k, v, pooled, m, 6, pool)
    full = b.reshape(-1, heads, N, N) if per_window else b[None]
    ref = oracle.nystra_attention(q, k, v, m, 6, pool, full.double().numpy())
    err = per_unit_rel(_units(got).double().numpy(), _units(torch.from_numpy(ref)).numpy())
    assert err.max() <= 1e-4, f"max rel err {err.max():.3e}"


def test_host_bias_pooling_is_the_landmark_mean():
    # integer biases: the pooled blocks are exact means over each landmark's tokens
    N, m = 16, 4
    b = torch.arange(N * N, dtype=torch.float32).reshape(1, N, N) % 7
    L, U, A = host.pool_bias(b, m)
    seg = torch.arange(N) // (N // m)
    for j in range(m):
        assert torch.allclose(L[0, :, j], b[0][:, seg == j].mean(1))
        assert torch.allclose(U[0, j, :], b[0][seg == j, :].mean(0))
        for i in range(m):
            assert torch.allclose(A[0, i, j], b[0][seg == i][:, seg == j].mean())


def test_host_bias_argument_validation():
    L = host.lib()
    P = 1 << 20
    inv = binding.NYSTRA_EINVAL
    f = L.nystra_attention_bias_host
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 6, 0, 8 * P, 9 * P, 10 * P, 3, 0) == inv   # bias windows
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 6, 0, 0, 9 * P, 10 * P, 1, 0) == inv       # missing block
    assert f(P, 2 * P, 3 * P, 64 * P, 4, 2, 64, 30, 16, 6, 0, 64 * P, 9 * P, 10 * P, 1, 0) == inv  # overlaps out
    g = L.nystra_pool_bias_host
    assert g(P, 1, 64, 15, 0, 2 * P, 3 * P, 4 * P, 0) == inv     # m does not divide N
    assert g(P, 1, 64, 16, 0, P, 3 * P, 4 * P, 0) == inv         # output overlaps the bias
    assert g(P, 0, 64, 16, 0, 2 * P, 3 * P, 4 * P, 0) == binding.NYSTRA_OK
