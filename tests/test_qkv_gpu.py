"""The fused Q/K/V projection front end on the GPU against the float64
oracle (the projections of Eq. 1, then PnP-Nystra).  The oracle projects
without rounding; the kernel rounds Q, K, V to the I/O type as an unfused
projection would store them, and over the paper's 0-6 iterations the same bar
holds with that rounding."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_08520_gb300 import binding, workloads
from tests.parity import TOL, per_unit_rel, sample_units

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2506_08520_gb300 import build
    build.build()


def _run(x, w, b, heads, m, iters=6, pool="segments", pooled=None):
    out = binding.nystra_qkv(x.cuda(), w.cuda(), heads, m, iters, b_qkv=None if b is None else b.cuda(),
                             pooled=pooled, landmarks=pool)
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    return out.cpu()


CASES = [  # n_windows, heads, d_h, m, pooling, dtype, projection bias
    (5, 6, 30, 16, "segments", "bf16", True),     # SwinIR heads: C = 180, a partial last k-step
    (7, 1, 32, 16, "segments", "bf16", False),    # Uformer stage 1: C = 32
    (3, 8, 32, 16, "segments", "f16", True),      # Uformer stage 4: C = 256
    (4, 3, 30, 8, "segments", "f16", False),      # m = 8
    (4, 6, 30, 16, "patches", "bf16", True),      # square-patch landmarks
    (3, 2, 16, 16, "segments", "bf16", True),     # d_h = 16: two empty n-tiles
    (3, 11, 32, 16, "segments", "bf16", True),    # C = 352, the widest
    (2, 2, 32, 8, "segments", "f16", True),       # C = 64: the widest with shared stages
    (3, 2, 30, 16, "patches", "bf16", True),      # shared stages, square patches
    (2, 5, 6, 8, "segments", "f16", True),        # C = 30: C % 4 != 0
    (2, 176, 2, 8, "segments", "bf16", True),     # more heads than SMs: CTAs beyond one wave
    (1, 6, 30, 16, "segments", "bf16", False),    # one window
]


@pytest.mark.parametrize("nw,heads,d,m,pool,dtype,with_b", CASES)
def test_fused_projection_matches_the_oracle(nw, heads, d, m, pool, dtype, with_b):
    x, w, b = workloads.random_x_wqkv(nw, 64, heads, d, dtype, seed=nw * 7 + heads + d + m, with_bias=with_b)
    out = _run(x, w, b, heads, m, pool=pool)
    ref = oracle.nystra_attention_qkv(x, w, b, heads, m, 6, pool)
    err = per_unit_rel(out.double().numpy(), ref)
    assert err.max() <= TOL[dtype], f"max rel err {err.max():.3e} at unit {int(err.argmax())}"


@pytest.mark.parametrize("iters", [0, 1, 4])
def test_fused_projection_iteration_counts(iters):
    x, w, b = workloads.random_x_wqkv(3, 64, 6, 30, "bf16", seed=iters)
    out = _run(x, w, b, 6, 16, iters)
    err = per_unit_rel(out.double().numpy(), oracle.nystra_attention_qkv(x, w, b, 6, 16, iters))
    assert err.max() <= TOL["bf16"]


def test_fused_projection_at_the_iteration_limit_is_finite():
    """Beyond the paper's 4-6 steps the iteration nears the pseudo-inverse of
    nearly singular G_A^n blocks, and the method's own output moves by up to
    ~100% when Q, K, V move by one rounding of the I/O type (the float64
    oracle shows it: 7 of 103,680 bf16 values one ulp apart change a unit's
    output by 10% at 12 steps, by 1e-4 at 6).  A fused projection rounds its
    own Q, K, V, so at 12 steps only finiteness is fixed."""
    x, w, b = workloads.random_x_wqkv(12, 64, 6, 30, "bf16", seed=12)
    out = _run(x, w, b, 6, 16, 12)
    assert torch.isfinite(out.float()).all()


def test_bias_only_projection_gives_the_value_bias():
    """W = 0: every token projects to the bias and the output is b_V's head
    slice (rounded to the I/O type), whatever the landmarks and iterations."""
    nw, heads, d = 3, 6, 30
    C = heads * d
    b = torch.randn(3 * C, generator=torch.Generator().manual_seed(5))
    x = torch.randn(nw, 64, C).bfloat16()
    out = _run(x, torch.zeros(3 * C, C, dtype=torch.bfloat16), b, heads, 16).double()
    want = b[2 * C:].bfloat16().double().reshape(1, heads, 1, d).expand(nw, heads, 64, d)
    assert torch.allclose(out, want, rtol=1e-2, atol=1e-3)


def test_fused_equals_projecting_first():
    """The fused call and the unfused path (Q, K, V projected in fp32, rounded
    to bf16, then nystra_attention) agree to the rounding of Q, K, V."""
    nw, heads, d = 16, 6, 30
    x, w, b = workloads.random_x_wqkv(nw, 64, heads, d, "bf16", seed=9)
    fused = _run(x, w, b, heads, 16).double()
    y = (x.cuda().float() @ w.cuda().float().T + b.cuda()).bfloat16()
    q, k, v = (y.reshape(nw, 64, 3, heads, d)[:, :, i].transpose(1, 2).contiguous() for i in range(3))
    unfused = binding.nystra(q, k, v, 16, 6).cpu().double()
    err = per_unit_rel(fused.numpy(), unfused.numpy())
    assert err.max() <= 1e-2, f"max rel err {err.max():.3e}"


def test_permuted_windows_give_permuted_outputs_bit_for_bit():
    nw, heads, d = 40, 6, 30
    x, w, b = workloads.random_x_wqkv(nw, 64, heads, d, "bf16", seed=11)
    perm = torch.from_numpy(np.random.default_rng(0).permutation(nw))
    a = _run(x, w, b, heads, 16)
    p = _run(x[perm].contiguous(), w, b, heads, 16)
    assert torch.equal(a[perm], p)


def test_fused_projection_with_a_score_bias():
    nw, heads, d, m = 6, 3, 30, 16
    x, w, b = workloads.random_x_wqkv(nw, 64, heads, d, "bf16", seed=13)
    B = torch.from_numpy(workloads.relpos_bias(8, heads, seed=14))
    pooled = binding.pool_bias(B.cuda(), m)
    out = _run(x, w, b, heads, m, pooled=pooled)
    ref = oracle.nystra_attention_qkv(x, w, b, heads, m, 6, "segments", B.double().numpy()[None])
    err = per_unit_rel(out.double().numpy(), ref)
    assert err.max() <= TOL["bf16"]
    assert per_unit_rel(oracle.nystra_attention_qkv(x, w, b, heads, m, 6), ref).max() > 0.02  # the bias matters


@pytest.mark.parametrize("name", ["swinir256-bf16-qkv", "uformer-s1-qkv", "uformer-s4-qkv", "sr720p-w8-m16-f16-qkv",
                                  "swinir256-bf16-relpos-qkv", "sr720p-w16-m16-bf16-qkv", "sr720p-w32-m16-bf16-qkv",
                                  "sr720p-w32-m32-bf16-qkv", "sr720p-w16-m16-bf16-relpos-qkv"])
def test_fused_workloads(name):
    """Full-size workloads in the launch configuration the benchmark times,
    checked on sampled units (first, last, strided and random)."""
    wl = workloads.WORKLOADS[name]
    x, w = workloads.make_x_wqkv(wl)
    pooled, B = None, workloads.make_bias(wl)
    if B is not None:
        pooled = binding.pool_bias(B.cuda(), wl.m, wl.landmarks)
    out = binding.nystra_qkv(x.cuda(), w.cuda(), wl.heads, wl.m, wl.iters, pooled=pooled, landmarks=wl.landmarks)
    torch.cuda.synchronize()
    assert binding.status() == binding.NYSTRA_OK
    idx = sample_units(wl.units, 96)
    win, head = idx // wl.heads, idx % wl.heads
    q, k, v = oracle.project_qkv(x[torch.from_numpy(np.unique(win))], w, None, wl.heads)
    pos = np.searchsorted(np.unique(win), win)
    bias = None if B is None else B.double().numpy()[head]
    ref = oracle.nystra_attention(q[pos, head], k[pos, head], v[pos, head], wl.m, wl.iters, wl.landmarks, bias)
    got = out.reshape(wl.units, wl.N, wl.d)[torch.from_numpy(idx)].cpu().double().numpy()
    err = per_unit_rel(got, ref)
    print(f"{name}: max rel err {err.max():.3e}")
    assert err.max() <= TOL[wl.dtype]


def _window_masks(n_windows, w=8, seed=0):
    """Shifted-window-like masks: tokens of different regions do not attend to
    each other (-100, finite); every other window is unmasked."""
    rng = np.random.default_rng(seed)
    N = w * w
    masks = np.zeros((n_windows, N, N))
    for i in range(0, n_windows, 2):
        region = (np.arange(N) % w >= w // 2).astype(int) + 2 * (np.arange(N) // w >= rng.integers(1, w))
        masks[i] = np.where(region[:, None] == region[None, :], 0.0, -100.0)
    return masks


@pytest.mark.parametrize("heads,d,dtype,per_window", [(2, 30, "bf16", False),   # shared stages (C = 60)
                                                      (2, 30, "f16", True),     # shared stages, per-window masks
                                                      (6, 30, "bf16", True)])   # private stages, per-window masks
def test_fused_projection_score_bias_variants(heads, d, dtype, per_window):
    nw, m = 4, 16
    x, w, b = workloads.random_x_wqkv(nw, 64, heads, d, dtype, seed=heads * 10 + d)
    B = workloads.relpos_bias(8, heads, seed=15)[None].astype(np.float64)       # [1, heads, N, N]
    if per_window:
        B = B + _window_masks(nw)[:, None]                                       # [nw, heads, N, N]
    B32 = np.ascontiguousarray(B.astype(np.float32))
    pooled = binding.pool_bias(torch.from_numpy(B32).cuda(), m)
    out = _run(x, w, b, heads, m, pooled=pooled)
    ref = oracle.nystra_attention_qkv(x, w, b, heads, m, 6, "segments",
                                      np.broadcast_to(B32.astype(np.float64), (nw, heads, 64, 64)))
    err = per_unit_rel(out.double().numpy(), ref)
    assert err.max() <= TOL[dtype], f"max rel err {err.max():.3e} at unit {int(err.argmax())}"


@pytest.mark.parametrize("m,pool,bias", [(16, "segments", "window"), (8, "segments", None), (16, "patches", None),
                                         (8, "segments", "head")])
def test_shared_stage_handoff_over_many_windows(m, pool, bias):
    """C = 60 <= 64: two warps share each Q/K/V stage and hand it over through
    the stage's bounded mbarrier.  4096 windows give every CTA dozens of
    windows, so every warp waits on the hand-off many times: with a per-window
    score bias, with m = 8 and with square patches.  Sampled units against
    the oracle."""
    nw, heads, d = 4096, 2, 30
    x, w, b = workloads.random_x_wqkv(nw, 64, heads, d, "bf16", seed=m + len(pool) + (0 if bias is None else 7))
    pooled, B = None, None
    if bias is not None:
        B = workloads.relpos_bias(8, heads, seed=3)[None].astype(np.float32)      # [1, heads, N, N]
        if bias == "window":
            B = np.ascontiguousarray(B + _window_masks(nw, seed=4)[:, None].astype(np.float32))
        pooled = binding.pool_bias(torch.from_numpy(B).cuda(), m, pool)
    out = _run(x, w, b, heads, m, pool=pool, pooled=pooled)
    idx = sample_units(nw * heads, 160)
    win, head = idx // heads, idx % heads
    uw = np.unique(win)
    q, k, v = oracle.project_qkv(x[torch.from_numpy(uw)], w, b, heads)
    pos = np.searchsorted(uw, win)
    bsl = None
    if B is not None:
        bsl = B.astype(np.float64)[win if B.shape[0] > 1 else np.zeros_like(win), head]
    ref = oracle.nystra_attention(q[pos, head], k[pos, head], v[pos, head], m, 6, pool, bsl)
    got = out.reshape(nw * heads, 64, d)[torch.from_numpy(idx)].double().numpy()
    err = per_unit_rel(got, ref)
    assert err.max() <= TOL["bf16"], f"max rel err {err.max():.3e} at sampled unit {int(idx[err.argmax()])}"


def test_fused_projection_with_16bit_factors():
    """NYSTRA_FACTORS_16 on the fused path: the same bar on soft inputs, and
    a different (single-rounding) kernel from the default."""
    x, w, b = workloads.random_x_wqkv(6, 64, 6, 30, "bf16", seed=21)
    ref = oracle.nystra_attention_qkv(x, w, b, 6, 16, 6)
    outs = []
    for factors in ("pairs", "16"):
        o = binding.nystra_qkv(x.cuda(), w.cuda(), 6, 16, 6, b_qkv=b.cuda(), factors=factors)
        torch.cuda.synchronize()
        assert binding.status() == binding.NYSTRA_OK
        outs.append(o.cpu())
        assert per_unit_rel(o.cpu().double().numpy(), ref).max() <= TOL["bf16"]
    assert not torch.equal(outs[0], outs[1])


@pytest.mark.parametrize("s", [2.0, 4.0])
def test_fused_projection_sharp_attention_is_finite(s):
    """W_Q, W_K scaled by s (logit std s^2): finite wherever the oracle is."""
    x, w, b = workloads.random_x_wqkv(8, 64, 6, 30, "bf16", seed=int(s) + 30)
    C = 180
    w = w.clone()
    w[:2 * C] = (w[:2 * C].float() * s).bfloat16()
    out = _run(x, w, b, 6, 16)
    ref = oracle.nystra_attention_qkv(x, w, b, 6, 16, 6)
    fin = np.isfinite(ref).all(axis=(-2, -1))
    assert np.isfinite(out.double().numpy()[fin]).all()


# 16x16 and 32x32 windows (the streaming structure, chunks projected in place)
LARGE = [  # n_windows, N, heads, d_h, m, pooling, dtype, projection bias
    (3, 256, 6, 30, 16, "segments", "bf16", True),    # SwinIR heads, C = 180
    (5, 256, 1, 32, 8, "segments", "f16", False),     # one head, C = 32
    (2, 256, 3, 30, 16, "patches", "bf16", True),     # square patches (4x4 of 4x4 tokens)
    (2, 1024, 6, 30, 16, "segments", "bf16", True),
    (2, 1024, 4, 32, 32, "segments", "bf16", True),   # m = 32: the two-warp core
    (2, 1024, 2, 16, 16, "patches", "f16", True),     # square patches (4x4 of 8x8 tokens)
    (1, 1024, 11, 32, 16, "segments", "bf16", True),  # C = 352, the widest
    (3, 256, 8, 32, 16, "segments", "f16", True),     # C = 256
    (2, 1024, 5, 6, 8, "segments", "bf16", True),     # C = 30: a partial k-step
]


@pytest.mark.parametrize("nw,N,heads,d,m,pool,dtype,with_b", LARGE)
def test_fused_projection_large_windows(nw, N, heads, d, m, pool, dtype, with_b):
    x, w, b = workloads.random_x_wqkv(nw, N, heads, d, dtype, seed=nw * 5 + N + heads + d + m, with_bias=with_b)
    out = _run(x, w, b, heads, m, pool=pool)
    ref = oracle.nystra_attention_qkv(x, w, b, heads, m, 6, pool)
    err = per_unit_rel(out.double().numpy(), ref)
    assert err.max() <= TOL[dtype], f"max rel err {err.max():.3e} at unit {int(err.argmax())}"


@pytest.mark.parametrize("N", [256, 1024])
def test_fused_large_windows_equal_projecting_first(N):
    """The fused call and the unfused path (projected in fp32, rounded to bf16,
    then nystra_attention) agree to the rounding of Q, K, V."""
    nw, heads, d = 3, 6, 30
    x, w, b = workloads.random_x_wqkv(nw, N, heads, d, "bf16", seed=N)
    fused = _run(x, w, b, heads, 16).double()
    y = (x.cuda().float() @ w.cuda().float().T + b.cuda()).bfloat16()
    q, k, v = (y.reshape(nw, N, 3, heads, d)[:, :, i].transpose(1, 2).contiguous() for i in range(3))
    unfused = binding.nystra(q, k, v, 16, 6).cpu().double()
    assert per_unit_rel(fused.numpy(), unfused.numpy()).max() <= 1e-2


@pytest.mark.parametrize("N,per_window", [(256, False), (1024, True)])
def test_fused_large_windows_with_a_score_bias(N, per_window):
    nw, heads, d, m = 3, 2, 30, 16
    w_ = int(round(N ** 0.5))
    x, w, b = workloads.random_x_wqkv(nw, N, heads, d, "bf16", seed=N + 3)
    B = workloads.relpos_bias(w_, heads, seed=5)[None].astype(np.float32)       # [1, heads, N, N]
    if per_window:
        B = np.ascontiguousarray(B + np.random.default_rng(1).normal(0, 0.5, (nw, 1, N, N)).astype(np.float32))
    pooled = binding.pool_bias(torch.from_numpy(B).cuda(), m)
    out = _run(x, w, b, heads, m, pooled=pooled)
    ref = oracle.nystra_attention_qkv(x, w, b, heads, m, 6, "segments",
                                      np.broadcast_to(B.astype(np.float64), (nw, heads, N, N)))
    err = per_unit_rel(out.double().numpy(), ref)
    assert err.max() <= TOL["bf16"], f"max rel err {err.max():.3e}"


def test_fused_large_windows_many_windows_and_16bit_factors():
    """Enough windows that every team of every CTA processes several units
    (both buffers of the double-buffered state, both task orders' steady
    state); both factor precisions on soft inputs.  Sampled units."""
    nw, N, heads, d, m = 600, 256, 2, 30, 16
    x, w, b = workloads.random_x_wqkv(nw, N, heads, d, "bf16", seed=77)
    idx = sample_units(nw * heads, 96)
    win, head = idx // heads, idx % heads
    uw = np.unique(win)
    q, k, v = oracle.project_qkv(x[torch.from_numpy(uw)], w, b, heads)
    pos = np.searchsorted(uw, win)
    ref = oracle.nystra_attention(q[pos, head], k[pos, head], v[pos, head], m, 6)
    for factors in ("pairs", "16"):
        out = binding.nystra_qkv(x.cuda(), w.cuda(), heads, m, 6, b_qkv=b.cuda(), factors=factors)
        torch.cuda.synchronize()
        assert binding.status() == binding.NYSTRA_OK
        got = out.reshape(nw * heads, N, d)[torch.from_numpy(idx)].cpu().double().numpy()
        assert per_unit_rel(got, ref).max() <= TOL["bf16"], factors
