"""Stage-by-stage parity of the tensor-core path for 8x8 windows.

The test-only stage dump runs, for one unit, the device functions of the
N = 64 kernel and returns every intermediate of Algorithm 1 in fp32.  Each
stage is held against the float64 oracle with a bound derived from the
rounding that stage performs (I/O-type landmarks and G^n blocks, fp32
accumulation), and the later stages are also checked "feed-forward": the
oracle's step applied to the GPU's own previous stage, so that each step's
arithmetic is isolated from the error it inherits."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_08520_gb300 import binding, workloads
from tests.parity import TOL

pytestmark = pytest.mark.gpu

TORCH = {"f32": torch.float32, "bf16": torch.bfloat16, "f16": torch.float16}
# Relative rounding unit of the values the path rounds to the I/O type (for
# fp32 I/O: the bf16 hi + lo operand split, 2^-16).
U = {"f32": 2.0 ** -16, "bf16": 2.0 ** -8, "f16": 2.0 ** -11}


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2506_08520_gb300 import build
    build.build()


def _stages(q, k, v, m, iters, unit, landmarks="segments"):
    qd, kd, vd = (x.cuda() for x in (q, k, v))
    st = binding.debug_stages(qd, kd, vd, m, iters, unit, landmarks=landmarks)
    return {n: x.double().numpy() for n, x in st.items()}


def _unit(x, u):
    return x.reshape(-1, x.shape[-2], x.shape[-1])[u].double().numpy()


def _relf(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


# ---------------------------------------------------------------- step 1
@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16"])
@pytest.mark.parametrize("m,d", [(16, 30), (8, 32), (16, 8)])
def test_segment_indexing_is_bit_exact(dtype, m, d):
    # Token i of the window carries i + c in column c: the mean of segment j
    # (tokens jL .. jL+L-1, L = 64/m) is jL + (L-1)/2 + c, exact in every I/O
    # type, so any wrong token-to-segment assignment changes a value.
    N, L = 64, 64 // m
    x = (torch.arange(N, dtype=torch.float64)[:, None] + torch.arange(d, dtype=torch.float64)[None, :])
    x = x.to(TORCH[dtype]).reshape(1, 1, N, d).contiguous()
    st = _stages(x, x.flip(-2).contiguous(), x, m, 6, 0)
    j = np.arange(m)[:, None]
    c = np.arange(d)[None, :]
    want_q = j * L + (L - 1) / 2 + c
    want_k = (N - 1) - (j * L + (L - 1) / 2) + c  # the same tokens in reverse order
    assert np.array_equal(st["qbar"], want_q)
    assert np.array_equal(st["kbar"], want_k)


@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16"])
def test_landmarks_of_integer_tokens_equal_the_oracle_exactly(dtype):
    # Integers in [-8, 8] and L in {4, 8}: every segment mean is a multiple
    # of 1/8 below 8 in magnitude, exact in each I/O type.
    g = torch.Generator().manual_seed(17)
    for m in (8, 16):
        x = torch.randint(-8, 9, (3, 2, 64, 30), generator=g).to(TORCH[dtype])
        for u in (0, 5):
            st = _stages(x, x, x, m, 6, u)
            ref = oracle.landmarks(_unit(x, u), m)
            assert np.array_equal(st["qbar"], ref)
            assert np.array_equal(st["kbar"], ref)


@pytest.mark.parametrize("dtype", ["bf16", "f16"])
@pytest.mark.parametrize("d", [30, 32, 8])
def test_patch_indexing_is_bit_exact(dtype, d):
    # Token (r, s) of the 8x8 window carries 8r + s + c in column c: the mean
    # of 2x2 patch (pr, pc) is 8 (2 pr + 1/2) + 2 pc + 1/2 + c, exact in both
    # 16-bit types (at most 89.5 = 179/2).
    N = 64
    x = (torch.arange(N, dtype=torch.float64)[:, None] + torch.arange(d, dtype=torch.float64)[None, :])
    x = x.to(TORCH[dtype]).reshape(1, 1, N, d).contiguous()
    st = _stages(x, x, x, 16, 6, 0, landmarks="patches")
    j = np.arange(16)[:, None]
    want = 8 * (2 * (j // 4) + 0.5) + 2 * (j % 4) + 0.5 + np.arange(d)[None, :]
    assert np.array_equal(st["qbar"], want)
    assert np.array_equal(st["kbar"], want)
    g = torch.Generator().manual_seed(18)
    xi = torch.randint(-8, 9, (2, 3, 64, d), generator=g).to(TORCH[dtype])
    for u in (0, 4):
        st = _stages(xi, xi, xi, 16, 6, u, landmarks="patches")
        assert np.array_equal(st["qbar"], oracle.landmarks(_unit(xi, u), 16, "patches"))


@pytest.mark.parametrize("dtype", ["bf16", "f16"])
def test_patch_stage_dump_matches_the_product_kernel(dtype):
    q, k, v = workloads.random_qkv(3, 64, 30, dtype, seed=21)
    full = binding.nystra(q.cuda(), k.cuda(), v.cuda(), 16, 6, landmarks="patches").cpu()
    for u in range(3):
        st = _stages(q, k, v, 16, 6, u, landmarks="patches")
        assert np.array_equal(_unit(full, u), st["out"])
        ref = oracle.nystra_stages(_unit(q, u), _unit(k, u), _unit(v, u), 16, 6, "patches")
        assert _relf(st["out"], ref["out"]) <= TOL[dtype]


# ------------------------------------------------------------ steps 2-7
CASES = [(16, 30, 6), (8, 32, 6), (16, 8, 6), (16, 30, 0), (16, 30, 1)]


@pytest.mark.parametrize("dtype", ["f32", "bf16", "f16"])
@pytest.mark.parametrize("m,d,iters", CASES)
def test_stages_against_oracle(dtype, m, d, iters):
    q, k, v = workloads.random_qkv(4, 64, d, dtype, seed=100 + m + d + iters)
    u_t = U[dtype]
    s = 1.0 / np.sqrt(d)
    for unit in (0, 3):
        st = _stages(q, k, v, m, iters, unit)
        Q, K, V = _unit(q, unit), _unit(k, unit), _unit(v, unit)
        ref = oracle.nystra_stages(Q, K, V, m, iters)

        # step 1: landmarks, fp32 sums of the (split, for fp32 I/O) tokens,
        # rounded once to the I/O type
        u_sum = 2.0 ** -16 if dtype == "f32" else 2.0 ** -20
        for name, X in (("qbar", Q), ("kbar", K)):
            r = ref[name]
            bound = u_t * np.abs(r) + u_sum * oracle.landmarks(np.abs(X), m) + 1e-12
            assert np.all(np.abs(st[name] - r) <= bound), name

        # steps 2-3: G_L^n = exp(S_L - m_L).  S_L uses the rounded Kbar
        # (|dS_ij| <= s sum_c |q_ic| |kbar_jc| u), the shift m_L moves by at
        # most the row's largest |dS|, and G_L^n is rounded to the I/O type.
        a_l = s * (np.abs(Q) @ np.abs(ref["kbar"]).T).max(axis=1, keepdims=True)
        bound = 2.0 * (2.0 * a_l * u_t + u_t) * ref["GLn"] + 1e-6
        assert np.all(np.abs(st["GLn"] - ref["GLn"]) <= bound), "G_L^n"

        # m_U over all N keys, from the rounded Qbar
        a_u = s * (np.abs(ref["qbar"]) @ np.abs(K).T).max(axis=1)
        assert np.all(np.abs(st["mU"] - ref["mU"]) <= 2.0 * a_u * u_t + 1e-5), "m_U"

        # step 5: W = G_U^n [V | 1]; G_U^n carries the m_U error twice over
        # and is rounded to the I/O type before the product
        V1 = np.concatenate([V, np.ones((64, 1))], axis=1)
        w_ref = ref["GUn"] @ V1
        eps = 2.0 * (4.0 * a_u * u_t + u_t)
        w_bound = (eps[:, None] * ref["GUn"]) @ np.abs(V1) + 1e-5
        assert np.all(np.abs(st["W"] - w_ref) <= w_bound), "W"

        # step 3: G_A^n = exp(S_A - m_U) from both rounded landmark sets
        a_a = s * (np.abs(ref["qbar"]) @ np.abs(ref["kbar"]).T).max(axis=1, keepdims=True)
        ga_bound = 2.0 * (2.0 * a_a * u_t + 2.0 * a_u[:, None] * u_t) * ref["GAn"] + 1e-6
        assert np.all(np.abs(st["GAn"] - ref["GAn"]) <= ga_bound), "G_A^n"

        # step 4, feed-forward: the oracle's iteration on the GPU's own G_A^n.
        # The GPU iterates on fp16 two-term splits (about 2^-22 per operand);
        # along directions of small singular values that have not converged a
        # step's error grows by up to 13/4 per later step: 2^-22 (13/4)^6 is
        # about 3e-4.
        z_ff = oracle.pinv_iteration(st["GAn"], iters)
        e_z = _relf(st["Z"], z_ff)
        assert e_z <= 1e-3, f"Z vs the oracle's iteration on the GPU's G_A^n: {e_z:.2e}"

        # step 6, feed-forward: Y = Z W, split-tf32 products (about 2^-21 per
        # product) with fp32 accumulation, bounded elementwise through |Z||W|
        zw = st["Z"] @ st["W"]
        assert np.all(np.abs(st["Y"] - zw) <= 2.0 ** -18 * (np.abs(st["Z"]) @ np.abs(st["W"])) + 1e-30), "Y = Z W"

        # step 7, feed-forward: O from the GPU's own G_L^n and Y.  The kernel
        # rounds Y to the I/O type (split bf16 for fp32 I/O), accumulates in
        # fp32 and rounds O; bound each ratio through |G_L^n| |Y|.
        G, Y = st["GLn"], st["Y"]
        num, den = G @ Y[:, :d], G @ Y[:, d]
        o_ff = num / den[:, None]
        e_num = u_t * (G @ np.abs(Y[:, :d]))
        e_den = u_t * (G @ np.abs(Y[:, d]))
        o_bound = 2.0 * ((e_num + np.abs(o_ff) * e_den[:, None]) / np.abs(den)[:, None] + u_t * np.abs(o_ff))
        assert np.all(np.abs(st["out"] - o_ff) <= o_bound + 1e-30), "O feed-forward"

        # end to end against the oracle, and against the product kernel
        assert _relf(st["out"], ref["out"]) <= TOL[dtype]
        full = binding.nystra(q.cuda(), k.cuda(), v.cuda(), m, iters)
        torch.cuda.synchronize()
        assert np.array_equal(_unit(full.cpu(), unit), st["out"]), "stage dump differs from nystra_attention"


def test_stage_dump_on_a_side_stream_matches():
    q, k, v = (x.cuda() for x in workloads.random_qkv(2, 64, 30, "bf16", seed=9))
    a = binding.debug_stages(q, k, v, 16, 6, 1)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        b = binding.debug_stages(q, k, v, 16, 6, 1, stream=s)
    for name in a:
        assert torch.equal(a[name], b[name]), name
