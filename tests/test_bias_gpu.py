"""Additive score bias on the GPU (relative-position bias, shifted-window masks)
against the float64 oracle: the landmark pooling of the bias, and PnP-Nystra
with a bias shared by all windows or given per window."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_08520_gb300 import binding, workloads
from tests.parity import TOL, per_unit_rel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2506_08520_gb300 import build
    build.build()


@pytest.mark.parametrize("N,m,pool", [(64, 16, "segments"), (64, 8, "segments"), (64, 16, "patches"),
                                      (256, 16, "patches"), (256, 32, "segments"), (1024, 16, "patches"),
                                      (48, 12, "segments")])
def test_pool_bias_matches_the_oracle(N, m, pool):
    rng = np.random.default_rng(N + m)
    B = rng.standard_normal((3, N, N)).astype(np.float32)
    bL, bU, bA = binding.pool_bias(torch.from_numpy(B).cuda(), m, pool)
    torch.cuda.synchronize()
    for n in range(3):
        rL, rU, rA = oracle.pool_bias(B[n], m, pool)
        for got, ref in ((bL[n], rL), (bU[n], rU), (bA[n], rA)):
            np.testing.assert_allclose(got.cpu().double().numpy(), ref, rtol=1e-5, atol=1e-5)


def _swin_bias(w, heads, rng, scale=0.5):
    """Relative-position bias of a w x w window: a table of (2w-1)^2 offsets per head."""
    table = scale * rng.standard_normal(((2 * w - 1) ** 2, heads))
    r, c = np.divmod(np.arange(w * w), w)
    idx = (r[:, None] - r[None, :] + w - 1) * (2 * w - 1) + (c[:, None] - c[None, :] + w - 1)
    return table[idx].transpose(2, 0, 1)  # [heads, N, N]


def _shift_masks(n_windows, w, rng):
    """Masks like those of shifted windows: tokens of different regions do not
    attend to each other (-100, finite); every other window is unmasked."""
    N = w * w
    masks = np.zeros((n_windows, N, N))
    for i in range(0, n_windows, 2):
        region = (np.arange(N) % w >= w // 2).astype(int) + 2 * (np.arange(N) // w >= rng.integers(1, w))
        masks[i] = np.where(region[:, None] == region[None, :], 0.0, -100.0)
    return masks


CASES = [  # n_windows, heads, N, d, m, pool, per-window masks
    (6, 3, 64, 30, 16, "segments", False),
    (6, 3, 64, 30, 16, "patches", True),
    (4, 2, 64, 32, 8, "segments", True),
    (3, 2, 256, 30, 16, "patches", False),
    (3, 2, 256, 30, 16, "segments", True),
    (2, 2, 1024, 30, 16, "patches", False),
    (2, 2, 256, 32, 32, "segments", False),
    (3, 2, 64, 30, 64, "segments", False),
]


@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16"])
@pytest.mark.parametrize("nw,heads,N,d,m,pool,masked", CASES)
def test_biased_attention_matches_the_oracle(nw, heads, N, d, m, pool, masked, dtype):
    rng = np.random.default_rng(nw * 100 + N + m)
    w = int(round(N ** 0.5))
    q, k, v = workloads.random_qkv(nw * heads, N, d, dtype, seed=N + d + m)
    q, k, v = (x.reshape(nw, heads, N, d) for x in (q, k, v))
    bias = _swin_bias(w, heads, rng)[None]                       # [1, heads, N, N]
    if masked:
        bias = bias + _shift_masks(nw, w, rng)[:, None]          # [nw, heads, N, N]
    pooled = binding.pool_bias(torch.from_numpy(bias.astype(np.float32)).cuda().contiguous(), m, pool)
    out = binding.nystra_biased(q.cuda(), k.cuda(), v.cuda(), pooled, m, 6, landmarks=pool)
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    # the oracle takes the fp32-rounded bias the GPU was given
    b32 = np.broadcast_to(bias.astype(np.float32).astype(np.float64), (nw, heads, N, N))
    ref = oracle.nystra_attention(q, k, v, m, 6, pool, b32)
    err = per_unit_rel(out.double().cpu().numpy(), ref)
    assert err.max() <= TOL[dtype], f"max rel err {err.max():.3e} at unit {int(err.argmax())}"
    # the bias matters: without it the output is far off
    plain = oracle.nystra_attention(q, k, v, m, 6, pool)
    assert per_unit_rel(plain, ref).max() > 0.05


def test_zero_bias_equals_the_unbiased_call():
    q, k, v = (x.cuda() for x in workloads.random_qkv(8, 64, 30, "bf16", seed=4))
    q, k, v = (x.reshape(4, 2, 64, 30) for x in (q, k, v))
    pooled = binding.pool_bias(torch.zeros(2, 64, 64, device="cuda"), 16)
    a = binding.nystra_biased(q, k, v, pooled, 16, 6)
    b = binding.nystra(q, k, v, 16, 6)
    torch.cuda.synchronize()
    err = per_unit_rel(a.double().cpu().numpy(), b.double().cpu().numpy())
    assert err.max() <= TOL["bf16"]


@pytest.mark.parametrize("name", ["swinir256-bf16-relpos", "sr720p-w16-m16-bf16-relpos",
                                  "sr720p-w32-m16-bf16-relpos"])
def test_relpos_workloads(name):
    from tests.parity import sample_units
    wl = workloads.WORKLOADS[name]
    q, k, v = workloads.make_qkv(wl)
    bias = workloads.make_bias(wl)
    pooled = binding.pool_bias(bias.cuda(), wl.m, wl.landmarks)
    out = binding.nystra_biased(q.cuda(), k.cuda(), v.cuda(), pooled, wl.m, wl.iters).cpu()
    idx = sample_units(wl.units, 192)
    qu, ku, vu, ou = (x.reshape(-1, wl.N, wl.d) for x in (q, k, v, out))
    b = bias.double().numpy()[idx % wl.heads]  # unit u is head u % heads
    ref = oracle.nystra_attention(qu[idx], ku[idx], vu[idx], wl.m, wl.iters, wl.landmarks, b)
    err = per_unit_rel(ou[idx].double().numpy(), ref)
    print(f"{name}: max rel err {err.max():.3e}")
    assert err.max() <= TOL[wl.dtype]
