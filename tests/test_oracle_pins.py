"""Pins for the float64 oracle against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: each test checks a closed form,
a brute-force evaluation, a special case that reduces to a textbook routine,
or an identity the method must satisfy, chosen so that a dropped term, a
wrong sign or index, or a transposed operand in the oracle fails one of them.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2506_08520_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_examples.json")


def _rng(seed):
    return np.random.default_rng(seed)


def _rel(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


# --------------------------------------------------------------------------
# Worked examples (tests/golden): hand-derived values.
# --------------------------------------------------------------------------
def _cases():
    with open(GOLDEN) as f:
        return {c["name"]: c for c in json.load(f)["cases"]}


def test_golden_exact_two_tokens():
    c = _cases()["exact_two_tokens"]
    out = oracle.exact_attention(np.array(c["q"])[None], np.array(c["k"])[None], np.array(c["v"])[None])
    np.testing.assert_allclose(out[0], np.array(c["exact_out"]), rtol=0, atol=1e-14)


def test_golden_single_landmark():
    c = _cases()["nystra_single_landmark"]
    out = oracle.nystra_attention(np.array(c["q"])[None], np.array(c["k"])[None],
                                  np.array(c["v"])[None], c["m"], c["iters"])
    np.testing.assert_allclose(out[0], np.array(c["nystra_out"]), rtol=0, atol=1e-14)


def test_golden_pinv_one_step():
    c = _cases()["pinv_iteration_diagonal"]
    Z = oracle.pinv_iteration(np.array(c["A"]), c["iters"])
    np.testing.assert_allclose(Z, np.array(c["Z1"]), rtol=0, atol=1e-15)


# --------------------------------------------------------------------------
# Exact attention, Eq. (1) / Eq. (2).
# --------------------------------------------------------------------------
def test_exact_attention_bruteforce():
    """Triple loop straight from Eq. 1 with math.exp, no max shift."""
    rng = _rng(11)
    U, N, d = 3, 5, 3
    q, k, v = (rng.standard_normal((U, N, d)) for _ in range(3))
    out = oracle.exact_attention(q, k, v)
    for u in range(U):
        for i in range(N):
            w = [math.exp(sum(q[u, i, c] * k[u, j, c] for c in range(d)) / math.sqrt(d)) for j in range(N)]
            z = sum(w)
            for c in range(d):
                ref = sum(w[j] * v[u, j, c] for j in range(N)) / z
                assert abs(out[u, i, c] - ref) < 1e-13


def test_exact_attention_kernel_form():
    """Eq. 2: O = (G V) / (G 1) with G = exp(QK^T/sqrt(d)) unshifted."""
    rng = _rng(12)
    q, k, v = (0.7 * rng.standard_normal((4, 32, 16)) for _ in range(3))
    G = np.exp(q @ k.transpose(0, 2, 1) / np.sqrt(16))
    ref = (G @ v) / G.sum(-1, keepdims=True)
    assert _rel(oracle.exact_attention(q, k, v), ref) < 1e-13


# --------------------------------------------------------------------------
# Step 1: landmarks (segment indexing must be exact).
# --------------------------------------------------------------------------
def test_landmarks_integer_exact():
    """Integer tokens and power-of-two segment length: means are exact."""
    rng = _rng(13)
    N, d = 64, 5
    x = rng.integers(-50, 50, size=(N, d)).astype(np.float64)
    for m in (1, 2, 8, 16, 64):
        L = N // m
        ref = np.array([[sum(x[t, c] for t in range(j * L, (j + 1) * L)) / L for c in range(d)]
                        for j in range(m)])
        assert np.array_equal(oracle.landmarks(x, m), ref)
    assert np.array_equal(oracle.landmarks(x, N), x)


def test_landmarks_segment_permutations():
    """Permuting tokens inside a segment permutes output rows; across segments it does not."""
    rng = _rng(14)
    N, d, m = 32, 8, 4
    q, k, v = (rng.standard_normal((N, d)) for _ in range(3))
    base = oracle.nystra_attention(q[None], k[None], v[None], m, 6)[0]
    perm = np.arange(N)
    perm[8:16] = perm[8:16][::-1]           # inside segment 1 (L = 8)
    out = oracle.nystra_attention(q[perm][None], k[perm][None], v[perm][None], m, 6)[0]
    np.testing.assert_allclose(out, base[perm], rtol=1e-10, atol=1e-12)
    swap = np.arange(N)
    swap[[7, 8]] = swap[[8, 7]]             # across segments 0 and 1
    out2 = oracle.nystra_attention(q[swap][None], k[swap][None], v[swap][None], m, 6)[0]
    assert np.abs(out2 - base[swap]).max() > 1e-6


# --------------------------------------------------------------------------
# Step 4: the iterative pseudo-inverse.
# --------------------------------------------------------------------------
def _gan(seed, N=64, d=30, m=16):
    rng = _rng(seed)
    q, k, v = (rng.standard_normal((N, d)) for _ in range(3))
    return oracle.nystra_stages(q, k, v, m, 0)["GAn"]


def test_iteration_start():
    """Z_0 = A^T / (||A||_1 ||A||_inf) and the start is convergent (rho(I - A Z_0) < 1)."""
    A = _gan(15)
    Z0 = oracle.pinv_iteration(A, 0)
    ref = A.T / (np.linalg.norm(A, 1) * np.linalg.norm(A, np.inf))
    np.testing.assert_allclose(Z0, ref, rtol=1e-14, atol=0)
    E0 = np.eye(len(A)) - A @ Z0
    assert np.max(np.abs(np.linalg.eigvals(E0))) < 1.0


def test_iteration_residual_recursion():
    """With E_k = I - A Z_k the update gives E_{k+1} = 3/4 E_k^3 + 1/4 E_k^4 exactly."""
    for seed in (16, 17):
        A = _gan(seed)
        I = np.eye(len(A))
        for kk in range(6):
            E = I - A @ oracle.pinv_iteration(A, kk)
            En = I - A @ oracle.pinv_iteration(A, kk + 1)
            pred = 0.75 * np.linalg.matrix_power(E, 3) + 0.25 * np.linalg.matrix_power(E, 4)
            assert np.abs(En - pred).max() < 1e-9 * max(1.0, np.abs(E).max())


def test_iteration_converges_to_moore_penrose():
    """Run to convergence the iteration reaches numpy's SVD pseudo-inverse,
    for a nonsingular core block and for a rank-deficient one."""
    A = _gan(18, m=8)
    Z = oracle.pinv_iteration(A, 80)
    np.testing.assert_allclose(Z, np.linalg.inv(A), rtol=1e-7, atol=1e-7 * np.abs(Z).max())
    # Rank 5 of 8 with singular values 3..1.  On the null space the update maps
    # round-off x -> 13x/4, so stop once the range has converged (3^k growth of
    # the residual exponent) and long before 3.25^k round-off growth matters.
    rng = _rng(19)
    U, _ = np.linalg.qr(rng.standard_normal((8, 8)))
    W, _ = np.linalg.qr(rng.standard_normal((8, 8)))
    B = U[:, :5] @ np.diag([3.0, 2.5, 2.0, 1.5, 1.0]) @ W[:, :5].T
    Zb = oracle.pinv_iteration(B, 12)
    P = np.linalg.pinv(B)
    np.testing.assert_allclose(Zb, P, atol=1e-9 * np.abs(P).max())
    np.testing.assert_allclose(B @ Zb @ B, B, atol=1e-9 * np.abs(B).max())
    np.testing.assert_allclose(Zb @ B @ Zb, Zb, atol=1e-9 * np.abs(Zb).max())


# --------------------------------------------------------------------------
# Steps 2-3: the kernel blocks and their stabilisation.
# --------------------------------------------------------------------------
def _extended(q, k, m):
    """G~ = exp(Q~ K~^T / sqrt(d)) built directly from its definition (Eq. 3)."""
    N, d = q.shape
    qb = q.reshape(m, N // m, d).mean(1)
    kb = k.reshape(m, N // m, d).mean(1)
    Qt, Kt = np.vstack([qb, q]), np.vstack([kb, k])
    return np.exp(Qt @ Kt.T / np.sqrt(d))


def test_blocks_match_extended_matrix():
    """G_A^n, G_U^n scaled by exp(m_U) and G_L^n by exp(m_L) are the blocks of G~."""
    rng = _rng(20)
    N, d, m = 48, 12, 6
    q, k, v = (rng.standard_normal((N, d)) for _ in range(3))
    st = oracle.nystra_stages(q, k, v, m, 6)
    Gt = _extended(q, k, m)
    eU, eL = np.exp(st["mU"])[:, None], np.exp(st["mL"])[:, None]
    np.testing.assert_allclose(st["GAn"] * eU, Gt[:m, :m], rtol=1e-12)
    np.testing.assert_allclose(st["GUn"] * eU, Gt[:m, m:], rtol=1e-12)
    np.testing.assert_allclose(st["GLn"] * eL, Gt[m:, :m], rtol=1e-12)
    # row maxima are the maxima of the log-scores the paper names (Sec. 2.2)
    np.testing.assert_allclose(np.exp(st["mU"]), Gt[:m, m:].max(1), rtol=1e-12)
    np.testing.assert_allclose(np.exp(st["mL"]), Gt[m:, :m].max(1), rtol=1e-12)


def test_stable_form_equals_unnormalised_form():
    """Eq. 8 (stabilised) with a converged inverse equals Eq. 7
    evaluated without any stabilisation, G^ = G_L G_A^+ G_U with an SVD pinv."""
    rng = _rng(21)
    N, d, m = 64, 16, 8
    q, k, v = (0.8 * rng.standard_normal((N, d)) for _ in range(3))
    Gt = _extended(q, k, m)
    GA, GU, GL = Gt[:m, :m], Gt[:m, m:], Gt[m:, :m]
    Gh = GL @ np.linalg.pinv(GA) @ GU
    ref = (Gh @ v) / (Gh @ np.ones(N))[:, None]
    out = oracle.nystra_attention(q[None], k[None], v[None], m, 80)[0]
    assert _rel(out, ref) < 1e-9


# --------------------------------------------------------------------------
# Special cases that reduce to exact attention.
# --------------------------------------------------------------------------
def test_every_token_a_landmark_is_exact_attention():
    """m = N: G_L = G_U = G and G_A = G, so G^ = G and the output is Eq. 1."""
    rng = _rng(22)
    U, N, d = 3, 16, 8
    q, k, v = (0.5 * rng.standard_normal((U, N, d)) for _ in range(3))
    ref = oracle.exact_attention(q, k, v)
    out = oracle.nystra_attention(q, k, v, N, 80)
    assert _rel(out, ref) < 1e-8


def test_corollary_exact_recovery():
    """Tokens constant within each segment make rank(G~) = m, so G^ = G (Corollary 2.2)."""
    rng = _rng(23)
    N, d, m = 64, 8, 8
    L = N // m
    qs, ks = rng.standard_normal((m, d)), rng.standard_normal((m, d))
    q, k = np.repeat(qs, L, axis=0), np.repeat(ks, L, axis=0)
    v = rng.standard_normal((N, d))
    assert np.linalg.matrix_rank(_extended(q, k, m), tol=1e-9) == m
    ref = oracle.exact_attention(q[None], k[None], v[None])
    out = oracle.nystra_attention(q[None], k[None], v[None], m, 80)
    assert _rel(out, ref) < 1e-8


def test_single_landmark_is_mean_query_attention():
    """m = 1: every output row is the exact attention of the mean query."""
    rng = _rng(24)
    N, d = 32, 6
    q, k, v = (rng.standard_normal((N, d)) for _ in range(3))
    out = oracle.nystra_attention(q[None], k[None], v[None], 1, 6)[0]
    w = np.exp(q.mean(0) @ k.T / np.sqrt(d))
    ref = (w @ v) / w.sum()
    np.testing.assert_allclose(out, np.broadcast_to(ref, (N, d)), rtol=1e-12, atol=1e-13)


# --------------------------------------------------------------------------
# Invariances that hold at any iteration count (Z need not be converged).
# --------------------------------------------------------------------------
def test_value_shift_and_scale():
    """O_N and O_D share P and G_U^n, so V + 1c^T -> O + 1c^T and aV -> aO."""
    rng = _rng(25)
    U, N, d, m = 4, 64, 30, 16
    q, k, v = (rng.standard_normal((U, N, d)) for _ in range(3))
    c = rng.standard_normal(d)
    base = oracle.nystra_attention(q, k, v, m, 6)
    shifted = oracle.nystra_attention(q, k, v + c, m, 6)
    np.testing.assert_allclose(shifted, base + c, rtol=1e-9, atol=1e-9)
    scaled = oracle.nystra_attention(q, k, -2.5 * v, m, 6)
    np.testing.assert_allclose(scaled, -2.5 * base, rtol=1e-12, atol=1e-12)


def test_units_are_independent():
    rng = _rng(26)
    U, N, d, m = 6, 32, 8, 4
    q, k, v = (rng.standard_normal((U, N, d)) for _ in range(3))
    base = oracle.nystra_attention(q, k, v, m, 6)
    p = rng.permutation(U)
    assert np.array_equal(oracle.nystra_attention(q[p], k[p], v[p], m, 6), base[p])
    for u in range(U):
        assert np.array_equal(oracle.nystra_attention(q[u:u + 1], k[u:u + 1], v[u:u + 1], m, 6)[0], base[u])


def test_invalid_m_rejected():
    q = np.zeros((1, 10, 4))
    for m in (0, 3, 11):
        with pytest.raises(ValueError):
            oracle.nystra_attention(q, q, q, m, 6)


# --------------------------------------------------------------------------
# Lemma 2.1 (spectral bound) in an explicit-constant form, and Table 6's trend.
# --------------------------------------------------------------------------
def _lemma_terms(q, k, m):
    Gt = _extended(q, k, m)
    GA, GU, GL, G = Gt[:m, :m], Gt[:m, m:], Gt[m:, :m], Gt[m:, m:]
    GAi = np.linalg.inv(GA)
    S = G - GL @ GAi @ GU
    sv_t = np.linalg.svd(Gt, compute_uv=False)
    sv_a = np.linalg.svd(GA, compute_uv=False)
    return S, sv_t, sv_a, GL @ GAi, GAi @ GU


@pytest.mark.parametrize("seed,lowrank", [(27, False), (28, True)])
def test_lemma_bound_explicit_constant(seed, lowrank):
    """Block LDU of G~ gives min(||S||, s_m(G_A)) <= (1+||G_L G_A^-1||)(1+||G_A^-1 G_U||) s_{m+1}(G~),
    S = G - G_L G_A^-1 G_U; the oracle's converged G^ reproduces S."""
    wl = workloads.Workload("t", 2, 1, 64, 16, 8, 6, "f32", seed, "lowrank" if lowrank else "iid")
    q, k, v = (x.double().numpy()[0, 0] for x in workloads.make_qkv(wl))
    m = 8
    S, sv_t, sv_a, LA, AU = _lemma_terms(q, k, m)
    lhs = min(np.linalg.norm(S, 2), sv_a[m - 1])
    rhs = (1 + np.linalg.norm(LA, 2)) * (1 + np.linalg.norm(AU, 2)) * sv_t[m]
    assert lhs <= rhs * (1 + 1e-9)
    # The oracle's converged stages rebuild G^ = M_L G_L^n Z G_U^n (Sec. 2.2, with
    # Z = (G_A^n)^-1 = G_A^-1 M_U), and its error is exactly the Schur complement S.
    st = oracle.nystra_stages(q, k, v, m, 200)
    Gh = (np.exp(st["mL"])[:, None] * st["GLn"]) @ st["Z"] @ st["GUn"]
    G = _extended(q, k, m)[m:, m:]
    assert _rel(Gh, G - S) < 1e-6
    print("empirical C = ||S|| s_m(G_A) / s_{m+1}(G~) =", np.linalg.norm(S, 2) * sv_a[m - 1] / sv_t[m])


def test_table6_trend_more_landmarks_and_iterations():
    """More landmarks (at 6 iterations) and more iterations (at m=16) move the
    output towards exact attention on low-rank inputs (Table 6's trend)."""
    wl = workloads.Workload("t", 8, 2, 256, 32, 16, 6, "f32", 3, "lowrank")
    q, k, v = (x.double().numpy().reshape(-1, 256, 32) for x in workloads.make_qkv(wl))
    ex = oracle.exact_attention(q, k, v)
    err_m = [_rel(oracle.nystra_attention(q, k, v, m, 6), ex) for m in (8, 16, 32)]
    err_i = [_rel(oracle.nystra_attention(q, k, v, 16, it), ex) for it in (1, 3, 6)]
    print("err vs m (8,16,32):", err_m, " err vs iters (1,3,6):", err_i)
    assert err_m[0] > err_m[2]
    assert err_i[0] > err_i[2]


# --------------------------------------------------------------------------
# Step 1, the other reading of "average pooling over non-overlapping windows":
# square patches of a square window.
# --------------------------------------------------------------------------
def _patch_major(w, p):
    """Token order that lists patch 0's tokens first, then patch 1's, ... (row-major patches)."""
    b = w // p
    return np.array([(pr * b + r) * w + pc * b + c
                     for pr in range(p) for pc in range(p) for r in range(b) for c in range(b)])


@pytest.mark.parametrize("w,p", [(8, 4), (8, 2), (16, 4), (16, 8), (32, 4), (8, 8), (8, 1)])
def test_patch_landmarks_integer_exact(w, p):
    """Integer tokens: patch means equal the mean over the b x b block of the w x w grid."""
    rng = _rng(31 + w + p)
    N, d, b = w * w, 3, w // p
    x = rng.integers(-40, 40, size=(N, d)).astype(np.float64)
    ref = x.reshape(p, b, p, b, d).mean(axis=(1, 3)).reshape(p * p, d)
    assert np.array_equal(oracle.landmarks(x, p * p, "patches"), ref)


@pytest.mark.parametrize("w,p", [(8, 4), (16, 4), (16, 8)])
def test_patches_are_segments_of_the_patch_major_order(w, p):
    """Patch pooling of a window equals segment pooling after reordering its tokens
    patch by patch; attention is equivariant under the token reordering."""
    rng = _rng(41 + w + p)
    N, d, m = w * w, 6, p * p
    q, k, v = (rng.standard_normal((2, N, d)) for _ in range(3))
    pm = _patch_major(w, p)
    assert sorted(pm) == list(range(N))
    out = oracle.nystra_attention(q, k, v, m, 6, "patches")
    seg = oracle.nystra_attention(q[:, pm], k[:, pm], v[:, pm], m, 6)
    np.testing.assert_allclose(out[:, pm], seg, rtol=1e-11, atol=1e-12)
    for u in range(2):
        np.testing.assert_array_equal(oracle.landmarks(q[u], m, "patches"), oracle.landmarks(q[u, pm], m))


def test_patch_permutations():
    """Swapping tokens inside a patch permutes output rows; across patches it does not."""
    rng = _rng(43)
    w, p, d = 8, 2, 5
    N, m = w * w, p * p
    q, k, v = (rng.standard_normal((N, d)) for _ in range(3))
    base = oracle.nystra_attention(q[None], k[None], v[None], m, 6, "patches")[0]
    inside = np.arange(N)
    inside[[0, 3 * w + 3]] = inside[[3 * w + 3, 0]]  # both in patch (0, 0) (b = 4)
    out = oracle.nystra_attention(q[inside][None], k[inside][None], v[inside][None], m, 6, "patches")[0]
    np.testing.assert_allclose(out, base[inside], rtol=1e-10, atol=1e-12)
    across = np.arange(N)
    across[[3, 4]] = across[[4, 3]]  # same segment of 16 tokens, different patches
    out2 = oracle.nystra_attention(q[across][None], k[across][None], v[across][None], m, 6, "patches")[0]
    assert np.abs(out2 - base[across]).max() > 1e-6


def test_patch_special_cases():
    """m = N (1 x 1 patches) and m = 1 (one patch) coincide with the segment reading."""
    rng = _rng(44)
    N, d = 16, 4
    q, k, v = (0.5 * rng.standard_normal((2, N, d)) for _ in range(3))
    for m in (1, N):
        np.testing.assert_array_equal(oracle.nystra_attention(q, k, v, m, 6, "patches"),
                                      oracle.nystra_attention(q, k, v, m, 6))


def test_patch_corollary_exact_recovery():
    """Tokens constant within each square patch: rank(G~) = m and G^ = G (Corollary 2.2)."""
    rng = _rng(45)
    w, p, d = 8, 4, 6
    b, m = w // p, p * p
    qs, ks = rng.standard_normal((p, p, d)), rng.standard_normal((p, p, d))
    up = lambda x: np.repeat(np.repeat(x, b, axis=0), b, axis=1).reshape(w * w, d)
    q, k = up(qs), up(ks)
    v = rng.standard_normal((w * w, d))
    ref = oracle.exact_attention(q[None], k[None], v[None])
    out = oracle.nystra_attention(q[None], k[None], v[None], m, 80, "patches")
    assert _rel(out, ref) < 1e-8
    seg = oracle.nystra_attention(q[None], k[None], v[None], m, 80)
    assert _rel(seg, ref) > 1e-3  # the segment reading does not see the patch structure


@pytest.mark.parametrize("N,m", [(64, 8), (48, 16), (64, 9), (256, 36)])
def test_patch_shapes_that_do_not_tile_are_rejected(N, m):
    x = np.zeros((1, N, 4))
    with pytest.raises(ValueError):
        oracle.nystra_attention(x, x, x, m, 6, "patches")


# --------------------------------------------------------------------------
# An additive score bias (window attention's relative-position bias and
# masks): each landmark block sees the mean bias over its landmarks' tokens.
# --------------------------------------------------------------------------
def test_exact_attention_with_bias_bruteforce():
    rng = _rng(51)
    N, d = 6, 3
    q, k, v = (rng.standard_normal((N, d)) for _ in range(3))
    B = rng.standard_normal((N, N))
    ref = np.empty((N, d))
    for i in range(N):
        w = [math.exp(sum(q[i, c] * k[j, c] for c in range(d)) / math.sqrt(d) + B[i, j]) for j in range(N)]
        for c in range(d):
            ref[i, c] = sum(w[j] * v[j, c] for j in range(N)) / sum(w)
    np.testing.assert_allclose(oracle.exact_attention(q[None], k[None], v[None], B)[0], ref, rtol=1e-12)


def _landmark_ids(N, m, pool):
    if pool == "segments":
        return np.arange(N) // (N // m)
    w, p = int(round(N ** 0.5)), int(round(m ** 0.5))
    b = w // p
    r, c = np.divmod(np.arange(N), w)
    return (r // b) * p + c // b


@pytest.mark.parametrize("pool,N,m", [("segments", 64, 16), ("segments", 32, 4), ("patches", 64, 16),
                                      ("patches", 256, 16), ("patches", 64, 4)])
def test_pool_bias_is_the_mean_over_landmark_tokens(pool, N, m):
    rng = _rng(52 + N + m)
    B = rng.standard_normal((N, N))
    BL, BU, BA = oracle.pool_bias(B, m, pool)
    ids = _landmark_ids(N, m, pool)
    for j in range(m):
        np.testing.assert_allclose(BL[:, j], B[:, ids == j].mean(axis=1), rtol=1e-12, atol=1e-14)
        np.testing.assert_allclose(BU[j], B[ids == j].mean(axis=0), rtol=1e-12, atol=1e-14)
        for i in range(m):
            np.testing.assert_allclose(BA[i, j], B[np.ix_(ids == i, ids == j)].mean(), rtol=1e-12, atol=1e-14)


def test_zero_bias_changes_nothing():
    rng = _rng(53)
    q, k, v = (rng.standard_normal((2, 64, 8)) for _ in range(3))
    for pool in ("segments", "patches"):
        np.testing.assert_array_equal(oracle.nystra_attention(q, k, v, 16, 6, pool, np.zeros((64, 64))),
                                      oracle.nystra_attention(q, k, v, 16, 6, pool))


def test_row_constant_bias_cancels():
    """B[i][t] = c_i shifts whole rows of S_L, S_U and S_A with their maxima: G^n is unchanged."""
    rng = _rng(54)
    N, d = 64, 8
    q, k, v = (rng.standard_normal((2, N, d)) for _ in range(3))
    B = np.repeat(3.0 * rng.standard_normal((N, 1)), N, axis=1)
    for pool in ("segments", "patches"):
        np.testing.assert_allclose(oracle.nystra_attention(q, k, v, 16, 6, pool, B),
                                   oracle.nystra_attention(q, k, v, 16, 6, pool), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(oracle.exact_attention(q, k, v, B), oracle.exact_attention(q, k, v),
                               rtol=1e-10, atol=1e-12)


def test_bias_with_every_token_a_landmark_is_exact_biased_attention():
    rng = _rng(55)
    U, N, d = 2, 16, 6
    q, k, v = (0.5 * rng.standard_normal((U, N, d)) for _ in range(3))
    B = 0.5 * rng.standard_normal((U, N, N))
    ref = oracle.exact_attention(q, k, v, B)
    assert _rel(oracle.nystra_attention(q, k, v, N, 80, "segments", B), ref) < 1e-8
    assert _rel(oracle.nystra_attention(q, k, v, N, 80, "patches", B), ref) < 1e-8


def test_block_constant_bias_exact_recovery():
    """Tokens constant per segment and a bias constant per pair of segments keep
    rank(G~) = m, so a converged inverse recovers exact biased attention."""
    rng = _rng(56)
    N, d, m = 64, 8, 8
    L = N // m
    q = np.repeat(rng.standard_normal((m, d)), L, axis=0)
    k = np.repeat(rng.standard_normal((m, d)), L, axis=0)
    v = rng.standard_normal((N, d))
    B = np.kron(rng.standard_normal((m, m)), np.ones((L, L)))
    ref = oracle.exact_attention(q[None], k[None], v[None], B)
    assert _rel(oracle.nystra_attention(q[None], k[None], v[None], m, 80, "segments", B), ref) < 1e-8
    # the bias matters: dropping it moves the output
    assert _rel(oracle.nystra_attention(q[None], k[None], v[None], m, 80), ref) > 1e-3


# --------------------------------------------------------------------------
# The projections of Eq. (1) (the fused Q/K/V front end).
# --------------------------------------------------------------------------
def _perm_weights(rng, C):
    perms = [rng.permutation(C) for _ in range(3)]
    w = np.zeros((3 * C, C))
    for i, p in enumerate(perms):
        w[i * C + np.arange(C), p] = 1.0
    return w, perms


def test_projection_with_permutation_weights_gathers_columns():
    """Row o of w_qkv holding a single 1 at column p[o] makes output feature o
    the token feature p[o], exactly: this fixes which of w or its transpose
    multiplies, the Q/K/V order of the stacked rows and the head split."""
    rng = _rng(60)
    nw, N, heads, d = 3, 16, 3, 4
    C = heads * d
    x = rng.standard_normal((nw, N, C))
    w, perms = _perm_weights(rng, C)
    for got, p in zip(oracle.project_qkv(x, w, None, heads), perms):
        for h in range(heads):
            np.testing.assert_array_equal(got[:, h], x[:, :, p[h * d:(h + 1) * d]])


def test_projection_bias_only_gives_the_value_bias():
    """W = 0: every token of a window projects to the bias, all scores are
    equal, and attention of identical values returns that value; the Nystrom
    blocks are all-ones, whose pseudo-inverse J/m^2 the iteration starts at and
    keeps.  So O = b_V's head slice exactly, for any m, pooling and iteration count."""
    rng = _rng(61)
    nw, N, heads, d = 2, 64, 2, 6
    C = heads * d
    x = rng.standard_normal((nw, N, C))
    b = rng.standard_normal(3 * C)
    want = np.broadcast_to(b[2 * C:].reshape(heads, 1, d), (nw, heads, N, d))
    for m, pool, iters in ((16, "segments", 6), (4, "patches", 3), (64, "segments", 0)):
        out = oracle.nystra_attention_qkv(x, np.zeros((3 * C, C)), b, heads, m, iters, pool)
        np.testing.assert_allclose(out, want, rtol=1e-12, atol=1e-12)


def test_projection_scaled_identities_reduce_to_split_heads():
    """w_qkv = [I; 2I; -I] makes Q, 2Q, -Q the heads of x itself (a reshape,
    no arithmetic), so the fused result is PnP-Nystra of those slices."""
    rng = _rng(62)
    nw, N, heads, d = 2, 64, 3, 8
    C = heads * d
    x = rng.standard_normal((nw, N, C))
    I = np.eye(C)
    xs = x.reshape(nw, N, heads, d).transpose(0, 2, 1, 3)
    got = oracle.nystra_attention_qkv(x, np.vstack([I, 2 * I, -I]), None, heads, 16, 6)
    np.testing.assert_allclose(got, oracle.nystra_attention(xs, 2 * xs, -xs, 16, 6), rtol=0, atol=1e-13)


def test_projection_reproduces_the_projected_workload_recipe():
    """The fused-projection workload hands the oracle the very draws the
    SwinIR-like recipe multiplies (Q, K, V = X W with W [in, out]), so its
    projections equal that recipe's Q, K, V."""
    wl = workloads.WORKLOADS["swinir256-bf16"].with_(n_windows=3)
    X, W = workloads._tokens_and_weights(wl)
    for got, ref in zip(oracle.project_qkv(X, W, None, wl.heads), workloads._proj(wl)):
        np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_projection_shapes_are_checked():
    with pytest.raises(ValueError):
        oracle.project_qkv(np.zeros((1, 4, 6)), np.zeros((18, 4)), None, 3)
    with pytest.raises(ValueError):
        oracle.project_qkv(np.zeros((1, 4, 6)), np.zeros((18, 6)), None, 4)
