// Tensor-core PnP-Nystra kernel for 64-token windows (8x8 windows), 16-bit I/O.
//
// One warp owns one (window, head) unit at a time; a CTA holds WARPS such
// warps, each with a private shared-memory slice, and the grid is persistent
// (warps stride over units).  Per unit:
//   stage   one mbarrier-tracked 1-D bulk copy each for Q, K, V (the unit's
//           N*d_h elements are contiguous), bounded wait;
//   front   landmarks Qbar, Kbar (segment means, Algorithm 1 step 1);
//           S_U = Qbar K^T on the tensor cores, row max m_U over all N keys,
//           G_U^n = exp(S_U - m_U) kept in registers and reused directly as the
//           A operand of W = G_U^n [V | 1] (step 6's right factor);
//           S_L = Q Kbar^T, m_L, G_L^n = exp(S_L - m_L) parked in shared memory
//           as ready-made MMA fragments.  Q, K, V are now consumed, so the next
//           unit's bulk copy is issued here and overlaps everything below;
//   back    G_A^n = exp(Qbar Kbar^T - m_U), Z_0 = A^T/(||A||_1 ||A||_inf) and
//           `iters` steps Z <- Z (13I - X(15I - X(7I - X)))/4, X = A Z (step 4),
//           Y = Z W, then O = (G_L^n Y_:d) / (G_L^n Y_d) (steps 5-7), written
//           straight from registers.
// Products with 64-token or d_h extents use mma.sync in the I/O dtype with fp32
// accumulation.  The m x m iteration and Y = Z W use split-tf32 mma.sync (three
// tf32 products per term, close to fp32: the iteration's round-off is amplified
// by ||A|| ||Z||, which grows with the iteration count).
//
// The iteration runs in registers.  Two facts make that possible:
//  * an MMA result (C layout: lane holds columns 2t, 2t+1) feeds the next MMA's
//    A operand unchanged if the k index is permuted consistently for both
//    operands (k-slot t <-> column 2t, k-slot t+4 <-> column 2t+1);
//  * X = A Z_k and every polynomial in X are symmetric (Z_0 = a A^T, and each
//    update multiplies by a polynomial in X), so the B fragment of such a matrix
//    is the lane's own C-layout values of its transpose.  The computed X is
//    symmetrised, (X + X^T)/2, each step to keep this exact for X itself.
// Z (the B operand of A Z) and X (for its transpose) go through shared memory
// once per step; everything else stays in registers.  Scores are kept in the
// log2 domain (scaled by log2(e)/sqrt(d_h)) so each exponential is one FFMA
// and one ex2.
#include "common.cuh"
#include "ptx.cuh"

namespace nystra {

__device__ unsigned int g_fault_w64;  // bit 0: a bounded wait gave up

namespace {

constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s bound on any single wait

template <int M, int NCOL>
struct Layout64 {
    static constexpr int N = 64;
    static constexpr int MT = (M + 15) / 16;           // landmark m-tiles
    static constexpr int MP = MT * 16;                 // padded landmark count
    static constexpr int LS = 40;                      // Qbar/Kbar row stride (16-bit elements)
    static constexpr int SM = MP + 4;                  // fp32 core-matrix row stride
    static constexpr int WS = NCOL + 4;                // fp32 W row stride
    static constexpr int YS = (M < 16 ? 16 : M) + 8;   // Y^T row stride (16-bit elements)
    static constexpr int KTL = (M >= 16) ? M / 16 : 1; // k-steps of O = G_L^n Y
    static constexpr size_t STAGE = 3 * N * 32 * 2;    // Q, K, V for d_h <= 32
    static constexpr size_t QBAR = STAGE;
    static constexpr size_t KBAR = QBAR + MP * LS * 2;
    static constexpr size_t GLF = KBAR + MP * LS * 2;
    static constexpr size_t MATA = GLF + (N / 16) * KTL * 32 * 16;
    static constexpr size_t MATZ = MATA + MP * SM * 4;
    static constexpr size_t WBUF = MATZ + MP * SM * 4;
    static constexpr size_t YT = WBUF + MP * WS * 4;
    static constexpr size_t BAR = YT + ((NCOL * YS * 2 + 15) / 16) * 16;
    static constexpr size_t WARP_BYTES = ((BAR + 16 + 127) / 128) * 128;
};

template <typename T>
__device__ __forceinline__ uint32_t ld32(const T* p) {
    return *reinterpret_cast<const uint32_t*>(p);
}

// C-layout fragments of an MP x MP fp32 matrix: f[i][n][e] is row
// 16i + g + 8(e >> 1), column 8n + 2t + (e & 1).
template <int MT>
using Frag = float[MT][2 * MT][4];

template <int MT>
__device__ __forceinline__ void frag_zero(Frag<MT>& f) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n) f[i][n][0] = f[i][n][1] = f[i][n][2] = f[i][n][3] = 0.f;
}

// T = alpha I - D, in place.
template <int MT>
__device__ __forceinline__ void frag_shift(Frag<MT>& f, float alpha, int g, int t) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const bool diag = (16 * i + 8 * (e >> 1) + g) == (8 * n + (e & 1) + 2 * t);
                f[i][n][e] = (diag ? alpha : 0.f) - f[i][n][e];
            }
}

template <int MT>
using FragLo = uint32_t[MT][2 * MT][4];

template <int MT>
__device__ __forceinline__ void frag_lo(const Frag<MT>& f, FragLo<MT>& lo) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) lo[i][n][e] = tf32_lo(f[i][n][e]);
}

// D = A B (MP x MP, fp32 accumulate) on split-tf32 tensor cores.
//   afrag(i, kk, hi[4], lo[4]) gives the A operand registers of m-tile i,
//     k-step kk (k permuted as described in the header);
//   bfrag(kk, j, y[2]) gives the B operand values of k-step kk, n-tile j.
// Even and odd k-steps accumulate separately, halving each chain of
// dependent MMAs.
template <int MT, typename AF, typename BF>
__device__ __forceinline__ void mm_tc(AF afrag, BF bfrag, Frag<MT>& D) {
    float acc[2][MT][2 * MT][4];
#pragma unroll
    for (int p = 0; p < 2; ++p)
#pragma unroll
        for (int i = 0; i < MT; ++i)
#pragma unroll
            for (int j = 0; j < 2 * MT; ++j) acc[p][i][j][0] = acc[p][i][j][1] = acc[p][i][j][2] = acc[p][i][j][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < 2 * MT; ++kk) {
        uint32_t ah[MT][4], al[MT][4];
#pragma unroll
        for (int i = 0; i < MT; ++i) afrag(i, kk, ah[i], al[i]);
#pragma unroll
        for (int j = 0; j < 2 * MT; ++j) {
            float y[2];
            bfrag(kk, j, y);
            const uint32_t bh0 = __float_as_uint(y[0]), bh1 = __float_as_uint(y[1]);
            const uint32_t bl0 = tf32_lo(y[0]), bl1 = tf32_lo(y[1]);
#pragma unroll
            for (int i = 0; i < MT; ++i) {
                float(&c)[4] = acc[kk & 1][i][j];
                mma_tf32(c, al[i][0], al[i][1], al[i][2], al[i][3], bh0, bh1);
                mma_tf32(c, ah[i][0], ah[i][1], ah[i][2], ah[i][3], bl0, bl1);
                mma_tf32(c, ah[i][0], ah[i][1], ah[i][2], ah[i][3], bh0, bh1);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int j = 0; j < 2 * MT; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) D[i][j][e] = acc[0][i][j][e] + acc[1][i][j][e];
}

// A operand (k-permuted) straight from C-layout fragments with precomputed low parts.
template <int MT>
struct AFromFrag {
    const Frag<MT>& f;
    const FragLo<MT>& lo;
    __device__ __forceinline__ void operator()(int i, int kk, uint32_t (&h)[4], uint32_t (&l)[4]) const {
        h[0] = __float_as_uint(f[i][kk][0]); l[0] = lo[i][kk][0];
        h[1] = __float_as_uint(f[i][kk][2]); l[1] = lo[i][kk][2];
        h[2] = __float_as_uint(f[i][kk][1]); l[2] = lo[i][kk][1];
        h[3] = __float_as_uint(f[i][kk][3]); l[3] = lo[i][kk][3];
    }
};
// B operand of a symmetric matrix from its own C-layout fragments.
template <int MT>
struct BFromSymFrag {
    const Frag<MT>& f;
    __device__ __forceinline__ void operator()(int kk, int j, float (&y)[2]) const {
        y[0] = f[j >> 1][kk][(j & 1) * 2];
        y[1] = f[j >> 1][kk][(j & 1) * 2 + 1];
    }
};
// B operand of a row-major fp32 matrix in shared memory (row stride S).
template <int S>
struct BFromSmem {
    const float* m;
    int g, t;
    __device__ __forceinline__ void operator()(int kk, int j, float (&y)[2]) const {
        y[0] = m[(8 * kk + 2 * t) * S + 8 * j + g];
        y[1] = m[(8 * kk + 2 * t + 1) * S + 8 * j + g];
    }
};

template <int MT, int SM>
__device__ __forceinline__ void frag_store(const Frag<MT>& f, float* S, int g, int t) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n) {
            const int r = 16 * i + g, c = 8 * n + 2 * t;
            *reinterpret_cast<float2*>(S + r * SM + c) = make_float2(f[i][n][0], f[i][n][1]);
            *reinterpret_cast<float2*>(S + (r + 8) * SM + c) = make_float2(f[i][n][2], f[i][n][3]);
        }
}

template <typename T, int M, int NCOL, int WARPS>
__global__ void __launch_bounds__(WARPS * 32, 1)
nystra_w64_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                  T* __restrict__ out, long long n_units, int d, int iters, float sl2) {
    using Lay = Layout64<M, NCOL>;
    using Op = Mma16<T>;
    constexpr int N = 64, MT = Lay::MT, MP = Lay::MP, LS = Lay::LS, SM = Lay::SM, WS = Lay::WS,
                  YS = Lay::YS, KTL = Lay::KTL, NTO = NCOL / 8;
    constexpr int L = N / M;  // tokens per landmark segment

    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;
    unsigned char* base = smem_raw + (size_t)warp * Lay::WARP_BYTES;
    const int nd = N * d;
    T* Qs = reinterpret_cast<T*>(base);
    T* Ks = Qs + nd;
    T* Vs = Qs + 2 * nd;
    T* qbar = reinterpret_cast<T*>(base + Lay::QBAR);
    T* kbar = reinterpret_cast<T*>(base + Lay::KBAR);
    unsigned char* glf = base + Lay::GLF;
    float* mA = reinterpret_cast<float*>(base + Lay::MATA);
    float* mZ = reinterpret_cast<float*>(base + Lay::MATZ);
    float* mW = reinterpret_cast<float*>(base + Lay::WBUF);
    T* yT = reinterpret_cast<T*>(base + Lay::YT);
    uint64_t* bar = reinterpret_cast<uint64_t*>(base + Lay::BAR);

    const long long stride = (long long)gridDim.x * WARPS;
    long long u = (long long)blockIdx.x * WARPS + warp;
    const uint32_t tile_bytes = (uint32_t)(nd * sizeof(T));

    auto issue = [&](long long unit) {
        const size_t off = (size_t)unit * nd;
        mbar_arrive_expect_tx(bar, 3u * tile_bytes);
        bulk_g2s(Qs, q + off, tile_bytes, bar);
        bulk_g2s(Ks, k + off, tile_bytes, bar);
        bulk_g2s(Vs, v + off, tile_bytes, bar);
    };

    if (lane == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    __syncwarp();
    if (u < n_units && lane == 0) issue(u);
    uint32_t phase = 0;

    for (; u < n_units; u += stride) {
        const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(bar, phase, kWaitNs));
        if (!ok) {
            if (lane == 0) atomicOr(&g_fault_w64, 1u);
            break;
        }
        phase ^= 1u;

        // ---------------- front: landmarks (Algorithm 1 step 1) ----------------
        {
            const float invL = 1.f / (float)L;
            const int dp = d >> 1;
#pragma unroll 2
            for (int idx = lane; idx < MP * 16; idx += 32) {
                const int j = idx >> 4, p = idx & 15;
                float ax = 0.f, ay = 0.f, bx = 0.f, by = 0.f;
                if (j < M && p < dp) {
#pragma unroll
                    for (int r = 0; r < L; ++r) {
                        const int off = (j * L + r) * d + 2 * p;
                        const float2 a = Op::unpack(ld32(Qs + off));
                        const float2 b = Op::unpack(ld32(Ks + off));
                        ax += a.x; ay += a.y; bx += b.x; by += b.y;
                    }
                    ax *= invL; ay *= invL; bx *= invL; by *= invL;
                }
                *reinterpret_cast<uint32_t*>(qbar + j * LS + 2 * p) = Op::pack(ax, ay);
                *reinterpret_cast<uint32_t*>(kbar + j * LS + 2 * p) = Op::pack(bx, by);
            }
        }
        __syncwarp();

        // ------- front: S_U, m_U, G_U^n (registers), W = G_U^n [V | 1] -------
        // B fragments of [V | 1 | 0] (k = tokens, n = columns) by 8x8 transposes.
        uint32_t vb[8][NTO];
#pragma unroll
        for (int a = 0; a < 8; ++a)
#pragma unroll
            for (int b = 0; b < NTO; ++b) {
                const int c0 = 8 * b + 2 * t;
                const uint32_t x = c0 < d ? ld32(Vs + (8 * a + g) * d + c0) : (c0 == d ? Op::kOne : 0u);
                vb[a][b] = movmatrix_trans(x);
            }
        float mU[MT][2];  // row maxima of S_U, log2 domain
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            uint32_t aq[2][4];
#pragma unroll
            for (int kk = 0; kk < 2; ++kk) {
                const T* r0 = qbar + (16 * mt + g) * LS + 16 * kk + 2 * t;
                aq[kk][0] = ld32(r0);
                aq[kk][1] = ld32(r0 + 8 * LS);
                aq[kk][2] = ld32(r0 + 8);
                aq[kk][3] = ld32(r0 + 8 * LS + 8);
            }
            float s[8][4];
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
                const T* kr = Ks + (8 * nt + g) * d;
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
                    const int c0 = 16 * kk + 2 * t, c1 = c0 + 8;
                    const uint32_t b0 = c0 < d ? ld32(kr + c0) : 0u;
                    const uint32_t b1 = c1 < d ? ld32(kr + c1) : 0u;
                    Op::k16(s[nt], aq[kk], b0, b1);
                }
            }
            float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
                mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
            }
            mx0 = quad_max(mx0) * sl2;
            mx1 = quad_max(mx1) * sl2;
            mU[mt][0] = mx0;
            mU[mt][1] = mx1;
            const bool v0 = (16 * mt + g) < M, v1 = (16 * mt + g + 8) < M;
            auto e0 = [&](float x) { return ex2(fmaf(x, sl2, -mx0)); };
            auto e1 = [&](float x) { return ex2(fmaf(x, sl2, -mx1)); };
            float w[NTO][4];
#pragma unroll
            for (int j = 0; j < NTO; ++j) w[j][0] = w[j][1] = w[j][2] = w[j][3] = 0.f;
#pragma unroll
            for (int kt = 0; kt < 4; ++kt) {
                uint32_t a[4];
                a[0] = v0 ? Op::pack(e0(s[2 * kt][0]), e0(s[2 * kt][1])) : 0u;
                a[1] = v1 ? Op::pack(e1(s[2 * kt][2]), e1(s[2 * kt][3])) : 0u;
                a[2] = v0 ? Op::pack(e0(s[2 * kt + 1][0]), e0(s[2 * kt + 1][1])) : 0u;
                a[3] = v1 ? Op::pack(e1(s[2 * kt + 1][2]), e1(s[2 * kt + 1][3])) : 0u;
#pragma unroll
                for (int j = 0; j < NTO; ++j) Op::k16(w[j], a, vb[2 * kt][j], vb[2 * kt + 1][j]);
            }
#pragma unroll
            for (int j = 0; j < NTO; ++j) {
                const int r = 16 * mt + g, c = 8 * j + 2 * t;
                *reinterpret_cast<float2*>(mW + r * WS + c) = make_float2(w[j][0], w[j][1]);
                *reinterpret_cast<float2*>(mW + (r + 8) * WS + c) = make_float2(w[j][2], w[j][3]);
            }
        }

        // ------------- front: S_L, G_L^n fragments (shared memory) -------------
        {
            constexpr int NTL = M / 8;
            uint32_t bk[NTL][2][2];
#pragma unroll
            for (int j = 0; j < NTL; ++j)
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
                    const T* kr = kbar + (8 * j + g) * LS + 16 * kk + 2 * t;
                    bk[j][kk][0] = ld32(kr);
                    bk[j][kk][1] = ld32(kr + 8);
                }
#pragma unroll
            for (int tm = 0; tm < 4; ++tm) {
                uint32_t a[2][4];
                const T* q0 = Qs + (16 * tm + g) * d;
                const T* q1 = q0 + 8 * d;
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
                    const int c0 = 16 * kk + 2 * t, c1 = c0 + 8;
                    a[kk][0] = c0 < d ? ld32(q0 + c0) : 0u;
                    a[kk][1] = c0 < d ? ld32(q1 + c0) : 0u;
                    a[kk][2] = c1 < d ? ld32(q0 + c1) : 0u;
                    a[kk][3] = c1 < d ? ld32(q1 + c1) : 0u;
                }
                float sl[NTL][4];
#pragma unroll
                for (int j = 0; j < NTL; ++j) {
                    sl[j][0] = sl[j][1] = sl[j][2] = sl[j][3] = 0.f;
#pragma unroll
                    for (int kk = 0; kk < 2; ++kk) Op::k16(sl[j], a[kk], bk[j][kk][0], bk[j][kk][1]);
                }
                float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
                for (int j = 0; j < NTL; ++j) {
                    mx0 = fmaxf(mx0, fmaxf(sl[j][0], sl[j][1]));
                    mx1 = fmaxf(mx1, fmaxf(sl[j][2], sl[j][3]));
                }
                mx0 = quad_max(mx0) * sl2;
                mx1 = quad_max(mx1) * sl2;
                auto e0 = [&](float x) { return ex2(fmaf(x, sl2, -mx0)); };
                auto e1 = [&](float x) { return ex2(fmaf(x, sl2, -mx1)); };
                if constexpr (M >= 16) {
#pragma unroll
                    for (int kk = 0; kk < KTL; ++kk) {
                        uint4 f;
                        f.x = Op::pack(e0(sl[2 * kk][0]), e0(sl[2 * kk][1]));
                        f.y = Op::pack(e1(sl[2 * kk][2]), e1(sl[2 * kk][3]));
                        f.z = Op::pack(e0(sl[2 * kk + 1][0]), e0(sl[2 * kk + 1][1]));
                        f.w = Op::pack(e1(sl[2 * kk + 1][2]), e1(sl[2 * kk + 1][3]));
                        reinterpret_cast<uint4*>(glf)[(tm * KTL + kk) * 32 + lane] = f;
                    }
                } else {
                    uint2 f;
                    f.x = Op::pack(e0(sl[0][0]), e0(sl[0][1]));
                    f.y = Op::pack(e1(sl[0][2]), e1(sl[0][3]));
                    reinterpret_cast<uint2*>(glf)[tm * 32 + lane] = f;
                }
            }
        }
        __syncwarp();

        // Q, K, V are consumed: prefetch the next unit into the stage.
        {
            const long long un = u + stride;
            if (un < n_units && lane == 0) {
                fence_proxy_async_smem();
                issue(un);
            }
        }

        // ------------- back: G_A^n (fragments), norms, Z_0 -------------
        Frag<MT> Zc, Ac;
        FragLo<MT> Aclo;
        {
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
                uint32_t aq[2][4];
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
                    const T* r0 = qbar + (16 * mt + g) * LS + 16 * kk + 2 * t;
                    aq[kk][0] = ld32(r0);
                    aq[kk][1] = ld32(r0 + 8 * LS);
                    aq[kk][2] = ld32(r0 + 8);
                    aq[kk][3] = ld32(r0 + 8 * LS + 8);
                }
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n) {
                    float sa[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                    for (int kk = 0; kk < 2; ++kk) {
                        const T* kr = kbar + (8 * n + g) * LS + 16 * kk + 2 * t;
                        Op::k16(sa, aq[kk], ld32(kr), ld32(kr + 8));
                    }
                    const int r0 = 16 * mt + g, r1 = r0 + 8, c = 8 * n + 2 * t;
                    Ac[mt][n][0] = (r0 < M && c < M) ? ex2(fmaf(sa[0], sl2, -mU[mt][0])) : 0.f;
                    Ac[mt][n][1] = (r0 < M && c + 1 < M) ? ex2(fmaf(sa[1], sl2, -mU[mt][0])) : 0.f;
                    Ac[mt][n][2] = (r1 < M && c < M) ? ex2(fmaf(sa[2], sl2, -mU[mt][1])) : 0.f;
                    Ac[mt][n][3] = (r1 < M && c + 1 < M) ? ex2(fmaf(sa[3], sl2, -mU[mt][1])) : 0.f;
                }
            }
            // ||A||_inf (max row sum) and ||A||_1 (max column sum); A > 0.
            float rmax = 0.f, cmax = 0.f;
#pragma unroll
            for (int i = 0; i < MT; ++i) {
                float r0 = 0.f, r1 = 0.f;
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n) {
                    r0 += Ac[i][n][0] + Ac[i][n][1];
                    r1 += Ac[i][n][2] + Ac[i][n][3];
                }
                r0 += __shfl_xor_sync(0xffffffffu, r0, 1);
                r0 += __shfl_xor_sync(0xffffffffu, r0, 2);
                r1 += __shfl_xor_sync(0xffffffffu, r1, 1);
                r1 += __shfl_xor_sync(0xffffffffu, r1, 2);
                rmax = fmaxf(rmax, fmaxf(r0, r1));
            }
#pragma unroll
            for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    float c = 0.f;
#pragma unroll
                    for (int i = 0; i < MT; ++i) c += Ac[i][n][e] + Ac[i][n][e + 2];
                    c += __shfl_xor_sync(0xffffffffu, c, 4);
                    c += __shfl_xor_sync(0xffffffffu, c, 8);
                    c += __shfl_xor_sync(0xffffffffu, c, 16);
                    cmax = fmaxf(cmax, c);
                }
            const float alpha = 1.f / (warp_max(rmax) * warp_max(cmax));
            frag_store<MT, SM>(Ac, mA, g, t);
            __syncwarp();
            // Z_0 = alpha A^T: C-layout element (r, c) is alpha * A[c][r].
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int r = 16 * i + g + 8 * (e >> 1), c = 8 * n + 2 * t + (e & 1);
                        Zc[i][n][e] = alpha * mA[c * SM + r];
                    }
            frag_store<MT, SM>(Zc, mZ, g, t);
            frag_lo<MT>(Ac, Aclo);
            __syncwarp();
        }

        // ---------------- back: pseudo-inverse iteration (step 4) ----------------
#pragma unroll 1
        for (int it = 0; it < iters; ++it) {
            Frag<MT> X, Tm, P;
            FragLo<MT> Xlo;
            mm_tc<MT>(AFromFrag<MT>{Ac, Aclo}, BFromSmem<SM>{mZ, g, t}, X);  // X = A Z
            // X is symmetric in exact arithmetic; make the computed one exactly
            // symmetric, (X + X^T)/2, so that every polynomial below is one in a
            // single symmetric matrix.  (Without this, reading B fragments of
            // X^T instead of X lets the antisymmetric round-off grow by up to
            // 13/4 per step in the not-yet-converged directions.)  Z is no longer
            // needed in shared memory, so its slot holds X for the transpose.
            __syncwarp();
            frag_store<MT, SM>(X, mZ, g, t);
            __syncwarp();
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int r = 16 * i + g + 8 * (e >> 1), c = 8 * n + 2 * t + (e & 1);
                        X[i][n][e] = 0.5f * (X[i][n][e] + mZ[c * SM + r]);
                        Tm[i][n][e] = X[i][n][e];
                    }
            frag_lo<MT>(X, Xlo);
            frag_shift<MT>(Tm, 7.f, g, t);                                   // 7I - X
            mm_tc<MT>(AFromFrag<MT>{X, Xlo}, BFromSymFrag<MT>{Tm}, P);     // X (7I - X)
            frag_shift<MT>(P, 15.f, g, t);                                   // 15I - ...
            mm_tc<MT>(AFromFrag<MT>{X, Xlo}, BFromSymFrag<MT>{P}, Tm);     // X (15I - ...)
            frag_shift<MT>(Tm, 13.f, g, t);                                  // 13I - ...
            {
                FragLo<MT> Zlo;
                frag_lo<MT>(Zc, Zlo);
                mm_tc<MT>(AFromFrag<MT>{Zc, Zlo}, BFromSymFrag<MT>{Tm}, P);  // Z (13I - ...)
            }
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                    for (int e = 0; e < 4; ++e) Zc[i][n][e] = 0.25f * P[i][n][e];
            __syncwarp();
            frag_store<MT, SM>(Zc, mZ, g, t);
            __syncwarp();
        }

        // ---------------- back: Y = Z W, Y^T as 16-bit B operand ----------------
        {
            float y[MT][NTO][4];
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int j = 0; j < NTO; ++j) y[i][j][0] = y[i][j][1] = y[i][j][2] = y[i][j][3] = 0.f;
            FragLo<MT> Zlo;
            frag_lo<MT>(Zc, Zlo);
#pragma unroll
            for (int kk = 0; kk < 2 * MT; ++kk) {
                uint32_t ah[MT][4], al[MT][4];
#pragma unroll
                for (int i = 0; i < MT; ++i) AFromFrag<MT>{Zc, Zlo}(i, kk, ah[i], al[i]);
#pragma unroll
                for (int j = 0; j < NTO; ++j) {
                    const float y0 = mW[(8 * kk + 2 * t) * WS + 8 * j + g];
                    const float y1 = mW[(8 * kk + 2 * t + 1) * WS + 8 * j + g];
                    const uint32_t bh0 = __float_as_uint(y0), bh1 = __float_as_uint(y1);
                    const uint32_t bl0 = tf32_lo(y0), bl1 = tf32_lo(y1);
#pragma unroll
                    for (int i = 0; i < MT; ++i) {
                        mma_tf32(y[i][j], al[i][0], al[i][1], al[i][2], al[i][3], bh0, bh1);
                        mma_tf32(y[i][j], ah[i][0], ah[i][1], ah[i][2], ah[i][3], bl0, bl1);
                        mma_tf32(y[i][j], ah[i][0], ah[i][1], ah[i][2], ah[i][3], bh0, bh1);
                    }
                }
            }
            // fp16 has a narrow range: scale Y by a power of two.  Numerator and
            // denominator columns share the factor, so it cancels in step 7.
            float scale = 1.f;
            if (Op::kNarrowRange) {
                float ymax = 0.f;
#pragma unroll
                for (int i = 0; i < MT; ++i)
#pragma unroll
                    for (int j = 0; j < NTO; ++j)
#pragma unroll
                        for (int e = 0; e < 4; ++e) ymax = fmaxf(ymax, fabsf(y[i][j][e]));
                ymax = warp_max(ymax);
                if (ymax > 0.f) scale = exp2f((float)(14 - ilogbf(ymax)));
            }
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int j = 0; j < NTO; ++j) {
                    const int r = 16 * i + g, c = 8 * j + 2 * t;
                    yT[c * YS + r] = from_f32<T>(y[i][j][0] * scale);
                    yT[(c + 1) * YS + r] = from_f32<T>(y[i][j][1] * scale);
                    yT[c * YS + r + 8] = from_f32<T>(y[i][j][2] * scale);
                    yT[(c + 1) * YS + r + 8] = from_f32<T>(y[i][j][3] * scale);
                }
        }
        __syncwarp();

        // ---------------- back: O = (G_L^n Y_:d) / (G_L^n Y_d) ----------------
        {
            uint32_t by[KTL][NTO][2];
#pragma unroll
            for (int kk = 0; kk < KTL; ++kk)
#pragma unroll
                for (int j = 0; j < NTO; ++j) {
                    const T* yr = yT + (8 * j + g) * YS + 16 * kk + 2 * t;
                    by[kk][j][0] = ld32(yr);
                    by[kk][j][1] = (M >= 16) ? ld32(yr + 8) : 0u;
                }
            const int jd = d >> 3, td = (d & 7) >> 1;
            const int src = (lane & ~3) | td;
            T* obase = out + (size_t)u * nd;
#pragma unroll
            for (int tm = 0; tm < 4; ++tm) {
                float o[NTO][4];
#pragma unroll
                for (int j = 0; j < NTO; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
                if constexpr (M >= 16) {
#pragma unroll
                    for (int kk = 0; kk < KTL; ++kk) {
                        const uint4 f = reinterpret_cast<const uint4*>(glf)[(tm * KTL + kk) * 32 + lane];
                        const uint32_t a[4] = {f.x, f.y, f.z, f.w};
#pragma unroll
                        for (int j = 0; j < NTO; ++j) Op::k16(o[j], a, by[kk][j][0], by[kk][j][1]);
                    }
                } else {
                    const uint2 f = reinterpret_cast<const uint2*>(glf)[tm * 32 + lane];
#pragma unroll
                    for (int j = 0; j < NTO; ++j) Op::k8(o[j], f.x, f.y, by[0][j][0]);
                }
                float d0 = 0.f, d1 = 0.f;
#pragma unroll
                for (int j = 0; j < NTO; ++j)
                    if (j == jd) {
                        d0 = o[j][0];
                        d1 = o[j][2];
                    }
                const float i0 = 1.f / __shfl_sync(0xffffffffu, d0, src);
                const float i1 = 1.f / __shfl_sync(0xffffffffu, d1, src);
                T* o0 = obase + (16 * tm + g) * d;
                T* o1 = o0 + 8 * d;
#pragma unroll
                for (int j = 0; j < NTO; ++j) {
                    const int c = 8 * j + 2 * t;
                    if (c < d) {
                        *reinterpret_cast<uint32_t*>(o0 + c) = Op::pack(o[j][0] * i0, o[j][1] * i0);
                        *reinterpret_cast<uint32_t*>(o1 + c) = Op::pack(o[j][2] * i1, o[j][3] * i1);
                    }
                }
            }
        }
        __syncwarp();
    }
}

template <typename T, int M, int NCOL, int WARPS>
cudaError_t launch_cfg(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                       int iters, cudaStream_t stream) {
    auto kern = nystra_w64_kernel<T, M, NCOL, WARPS>;
    const size_t smem = (size_t)WARPS * Layout64<M, NCOL>::WARP_BYTES;
    static int s_blocks = 0;  // persistent grid size (device-wide), set on first use
    if (s_blocks == 0) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        int dev = 0, sms = 0, per_sm = 0;
        if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
        if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
        if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, WARPS * 32, smem)) != cudaSuccess)
            return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        s_blocks = sms * per_sm;
    }
    const long long want = (n_units + WARPS - 1) / WARPS;
    const long long grid = want < s_blocks ? want : s_blocks;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<(unsigned)grid, WARPS * 32, smem, stream>>>((const T*)q, (const T*)k, (const T*)v, (T*)out, n_units,
                                                      d, iters, sl2);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const void* q, const void* k, const void* v, void* out, long long n_units, int d, int m,
                     int iters, cudaStream_t stream) {
    const bool wide = d > 30;  // the ones column needs a fifth n-tile when d_h = 32
    switch (m) {
        case 8:
            return wide ? launch_cfg<T, 8, 40, 9>(q, k, v, out, n_units, d, iters, stream)
                        : launch_cfg<T, 8, 32, 9>(q, k, v, out, n_units, d, iters, stream);
        case 16:
            return wide ? launch_cfg<T, 16, 40, 9>(q, k, v, out, n_units, d, iters, stream)
                        : launch_cfg<T, 16, 32, 9>(q, k, v, out, n_units, d, iters, stream);
        default:
            return wide ? launch_cfg<T, 32, 40, 5>(q, k, v, out, n_units, d, iters, stream)
                        : launch_cfg<T, 32, 32, 5>(q, k, v, out, n_units, d, iters, stream);
    }
}

}  // namespace
}  // namespace nystra

namespace nystra_host {
bool nystra_w64_supports(int N, int d, int m, int dtype) {
    return (dtype == 1 || dtype == 2) && N == 64 && d >= 2 && d <= 32 && (d % 2) == 0 &&
           (m == 8 || m == 16 || m == 32);
}

cudaError_t launch_nystra_w64(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                              int m, int iters, int dtype, cudaStream_t stream) {
    using namespace nystra;
    if (dtype == 1) return launch_t<__nv_bfloat16>(q, k, v, out, n_units, d, m, iters, stream);
    return launch_t<__half>(q, k, v, out, n_units, d, m, iters, stream);
}

unsigned int take_fault_word_w64(cudaError_t* err) {
    unsigned int w = 0, zero = 0;
    *err = cudaMemcpyFromSymbol(&w, nystra::g_fault_w64, sizeof(w));
    if (*err == cudaSuccess && w != 0) *err = cudaMemcpyToSymbol(nystra::g_fault_w64, &zero, sizeof(zero));
    return w;
}
}  // namespace nystra_host
