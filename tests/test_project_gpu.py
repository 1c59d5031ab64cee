"""The Q/K/V projection of Eq. 1 on the fifth-generation tensor cores
(nystra_project_qkv, tcgen05 MMAs with tensor-memory accumulators) against
the float64 oracle's projection.  The kernel accumulates the products of the
16-bit inputs in fp32 and rounds once to the I/O type, so every element is
within one unit in the last place of the oracle's exactly rounded value, and
almost all are equal to it; on integer inputs, whose sums fp32 holds exactly,
the two agree bit for bit.  Then the projections feed nystra_attention and
are compared with the oracle's PnP-Nystra of the projected tokens and with the
fused entry point."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_08520_gb300 import binding, workloads
from tests.parity import TOL, per_unit_rel

pytestmark = pytest.mark.gpu

TORCH = {"bf16": torch.bfloat16, "f16": torch.float16}
ULP = {"bf16": 2.0 ** -7, "f16": 2.0 ** -10}  # spacing relative to the leading power of two


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2506_08520_gb300 import build
    build.build()


def _project(x, w, b, heads):
    q, k, v = binding.project_qkv(x.cuda(), w.cuda(), heads, None if b is None else b.cuda())
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    return tuple(t.cpu() for t in (q, k, v))


def _check_rounding(got, ref, x, w, heads, dtype):
    """Each element within one ulp (of its I/O type, at the oracle's value) plus
    the fp32 accumulation bound; at least 99% equal to the rounded oracle."""
    C = x.shape[-1]
    # sum_c |x_c w_oc| per output element, as a bound on fp32 accumulation error
    ax = x.double().abs().numpy()
    aw = w.double().abs().numpy()
    mag = ax @ aw.T  # [nw, N, 3C]
    mag = mag.reshape(mag.shape[0], mag.shape[1], 3, heads, C // heads).transpose(2, 0, 3, 1, 4)
    rounded = 0
    total = 0
    for i in range(3):
        g = got[i].double().numpy()
        r = ref[i]
        ulp = ULP[dtype] * np.exp2(np.floor(np.log2(np.maximum(np.abs(r), 1e-30))))
        bound = ulp + C * 2.0 ** -22 * mag[i]
        bad = np.abs(g - r) > bound
        assert not bad.any(), (f"part {'QKV'[i]}: {int(bad.sum())} elements beyond one ulp, worst "
                               f"{float(np.max(np.abs(g - r) - bound)):.3e}")
        rt = torch.from_numpy(r).to(TORCH[dtype]).double().numpy()
        rounded += int((g == rt).sum())
        total += g.size
    assert rounded >= 0.99 * total, f"only {rounded}/{total} elements equal the rounded oracle"


CASES = [  # n_windows, N, heads, d_h, dtype, projection bias
    (2, 64, 6, 30, "bf16", True),     # SwinIR: C = 180, two heads per CTA, a partial last k-block
    (3, 64, 1, 32, "bf16", False),    # Uformer stage 1: C = 32, one head
    (2, 64, 8, 32, "f16", True),      # Uformer stage 4: C = 256
    (3, 64, 3, 30, "bf16", True),     # C = 90: 4-byte granules (C % 4 != 0), a half-empty head pair
    (5, 32, 2, 2, "f16", True),       # N = 32, d_h = 2
    (7, 96, 4, 16, "bf16", True),     # a tile of 128 rows straddling windows, a ragged last tile
    (1, 1024, 6, 30, "f16", False),   # one 32x32 window
    (2, 64, 12, 32, "bf16", True),    # C = 384, the widest: one head per CTA
    (2, 256, 5, 24, "bf16", True),    # 16x16 windows, odd head count
]


@pytest.mark.parametrize("nw,N,heads,d,dtype,with_b", CASES)
def test_projection_matches_the_oracle(nw, N, heads, d, dtype, with_b):
    x, w, b = workloads.random_x_wqkv(nw, N, heads, d, dtype, seed=nw * 13 + N + heads + d, with_bias=with_b)
    got = _project(x, w, b, heads)
    ref = oracle.project_qkv(x, w, b, heads)
    _check_rounding(got, ref, x, w, heads, dtype)


@pytest.mark.parametrize("dtype", ["bf16", "f16"])
def test_projection_is_exact_on_integers(dtype):
    # integer tokens and weights in [-3, 3] and a bias of halves: every sum is
    # exact in fp32 and float64, so the kernel's one rounding is the oracle's
    rng = np.random.default_rng(5)
    nw, N, heads, d = 3, 64, 6, 30
    C = heads * d
    x = torch.from_numpy(rng.integers(-3, 4, (nw, N, C)).astype(np.float32)).to(TORCH[dtype])
    w = torch.from_numpy(rng.integers(-3, 4, (3 * C, C)).astype(np.float32)).to(TORCH[dtype])
    b = torch.from_numpy(rng.integers(-8, 9, 3 * C).astype(np.float32) / 2)
    got = _project(x, w, b, heads)
    ref = oracle.project_qkv(x, w, b, heads)
    for i in range(3):
        rt = torch.from_numpy(ref[i]).to(TORCH[dtype])
        assert torch.equal(got[i], rt), f"part {'QKV'[i]}: {int((got[i] != rt).sum())} elements differ"


def test_projection_layout_by_permutation_weights():
    # w_qkv row o holds a single 1 at column perm[o]: Q, K, V are gathers of
    # token features, exactly, in the head-split layout
    rng = np.random.default_rng(9)
    nw, N, heads, d = 2, 64, 6, 30
    C = heads * d
    x = torch.from_numpy(rng.standard_normal((nw, N, C))).to(torch.bfloat16)
    perm = rng.integers(0, C, 3 * C)
    w = torch.zeros(3 * C, C, dtype=torch.bfloat16)
    w[np.arange(3 * C), perm] = 1
    got = _project(x, w, None, heads)
    xs = x.double().numpy()
    for i in range(3):
        feats = xs[..., perm[i * C:(i + 1) * C]].reshape(nw, N, heads, d).transpose(0, 2, 1, 3)
        assert np.array_equal(got[i].double().numpy(), feats), f"part {'QKV'[i]} is not the gather"


def test_projection_repeated_calls_are_identical():
    x, w, b = workloads.random_x_wqkv(40, 64, 6, 30, "bf16", seed=3)
    a = _project(x, w, b, 6)
    c = _project(x, w, b, 6)
    for i in range(3):
        assert torch.equal(a[i], c[i])


def test_projection_zero_windows_is_a_no_op():
    x = torch.zeros(0, 64, 180, dtype=torch.bfloat16, device="cuda")
    w = torch.zeros(540, 180, dtype=torch.bfloat16, device="cuda")
    q, k, v = binding.project_qkv(x, w, 6)
    torch.cuda.synchronize()
    assert q.shape == (0, 6, 64, 30) and binding.status() == binding.NYSTRA_OK


@pytest.mark.parametrize("name", ["sr720p-w32-m16-bf16-qkv", "sr720p-w16-m16-bf16-qkv", "swinir256-bf16-qkv"])
def test_projection_full_size_sampled_windows(name):
    wl = workloads.WORKLOADS[name]
    x, w = workloads.make_x_wqkv(wl)
    q, k, v = binding.project_qkv(x.cuda(), w.cuda(), wl.heads)
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    rng = np.random.default_rng(0)
    idx = np.unique(np.concatenate([[0, wl.n_windows - 1], rng.choice(wl.n_windows, 6, replace=False)]))
    got = tuple(t[idx].cpu() for t in (q, k, v))
    ref = oracle.project_qkv(x[idx], w, None, wl.heads)
    _check_rounding(got, ref, x[idx], w, wl.heads, wl.dtype)


@pytest.mark.parametrize("N,m", [(64, 16), (256, 16), (1024, 16), (1024, 32)])
def test_projection_then_attention(N, m):
    # project, then nystra_attention: the oracle's PnP-Nystra of the projected
    # tokens within the bar, and the fused entry point's result within 1e-2
    x, w, b = workloads.random_x_wqkv(4, N, 6, 30, "bf16", seed=N + m)
    xd, wd, bd = x.cuda(), w.cuda(), b.cuda()
    q, k, v = binding.project_qkv(xd, wd, 6, bd)
    out = binding.nystra(q, k, v, m, 6)
    fused = binding.nystra_qkv(xd, wd, 6, m, 6, b_qkv=bd)
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    ref = oracle.nystra_attention_qkv(x, w, b, 6, m, 6)
    err = per_unit_rel(out.cpu().double().numpy(), ref)
    assert err.max() <= TOL["bf16"], f"max rel err {err.max():.3e}"
    agree = per_unit_rel(out.cpu().double().numpy(), fused.cpu().double().numpy())
    assert agree.max() <= 1e-2, f"two-pass and fused paths differ by {agree.max():.3e}"
