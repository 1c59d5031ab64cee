// Tensor-core PnP-Nystra: the per-phase device functions shared by every
// tensor-core kernel, and the grouped kernel.  Windows of N = 64, 256 or 1024
// tokens (8x8, 16x16, 32x32), m in {8, 16, 32, 64}, even d_h <= 32, 16-bit
// I/O (fp32 I/O through the operand policy Opnd<float>, used by the 8x8 pool
// kernel).  Included by one translation unit per N (nystra_tc_n*.cu), which
// also includes the kernel for its common case: nystra_pool.cuh (8x8, m <=
// 16), nystra_team.cuh (16x16, m <= 32), nystra_stream.cuh (32x32, m <= 32).
// Compile-time options of those kernels: square-patch landmarks (Pooling,
// PW > 0) and an additive score bias (BIAS, m <= 16).
//
// Phases of one (window, head) unit:
//   stage    bulk copies of Q, K, V rows (contiguous in HBM) into shared
//            memory; bounded mbarrier waits.
//   front    landmarks (Algorithm 1 step 1) of the segments a warp owns
//            (segments never straddle warps: N/m <= TPW); S_L = Q Kbar^T and
//            G_L^n = exp(S_L - m_L) parked as MMA fragments [P1];
//            S_U = Qbar K^T with a running row max across 64-token chunks,
//            G_U^n fed straight from registers into W_r = G_U^n [V | 1],
//            rescaled online when the max grows.
//   combine  (several token warps) partial (W_r, m_r) merged in a fixed
//            order: m_U = max_r m_r, W = sum_r exp(m_r - m_U) W_r, which is
//            exactly G_U^n [V | 1] with the max over all N keys.
//   core     G_A^n = exp(Qbar Kbar^T - m_U), Z_0 = A^T/(||A||_1 ||A||_inf),
//            `iters` steps Z <- Z(13I - X(15I - X(7I - X)))/4 with X = A Z
//            (step 4), Y = Z W stored as a 16-bit B operand: core_warp (one
//            warp, in registers, m <= 16) or dist_core (m/16 warps).
//   output   O = (G_L^n Y_:d) / (G_L^n Y_d) (steps 5-7), staged row-major and
//            written with one bulk store (rows of 60 bytes would otherwise be
//            written as partial sectors); [P2] S_L and G_L^n recomputed from
//            a still-resident Q.
//
// Grouped kernel (nystra_tc_kernel; every m = 32 or 64 the three kernels
// above do not take).  A group of token warps owns one unit at a time, plus
// helper warps when the distributed core needs more warps than there are
// token warps; a CTA holds GROUPS groups and the grid is persistent.  The
// next unit's Q and K are copied after the combine ([P2]: K only, Q after the
// output), V once the output store has read its staging.  P1 ("G_L parked")
// is used when it fits as many groups as P2.
//
// Arithmetic.  Products with token or d_h extents use mma.sync in the I/O
// type with fp32 accumulation.  The m x m iteration needs close to fp32
// accuracy (its round-off is amplified by ||A|| ||Z||, which grows with the
// iteration count): it uses fp16 two-term splits (x = hi + lo, three k16
// products lo*hi + hi*lo + hi*hi, 22 significant bits), with Z rescaled by a
// power of two every step to stay in fp16's range.  Y = Z W uses split-tf32
// (W's range is not bounded).  The iteration carries the symmetric
// X = A Z_k next to Z (X_{k+1} = X_k T3/4, equal to A Z_{k+1}), so every
// product has a symmetric or transposed right factor, and X is made exactly
// symmetric (lower triangle mirrored) after each update, which keeps
// antisymmetric round-off from growing by up to 13/4 per step in directions
// that have not converged.  Scores are kept in the log2 domain (scaled by
// log2(e)/sqrt(d_h)), so each exponential is one FFMA and one ex2.
#pragma once

#include "common.cuh"
#include "ptx.cuh"

namespace nystra {
namespace tc {

constexpr uint64_t kWaitNs = 2000000000ull;  // 2 s bound on any single wait
constexpr float kLog2e = 1.4426950408889634f;  // score bias into the log2 domain of ex2
constexpr size_t kSmemLimit = 232448;        // opt-in dynamic shared memory per CTA

// 2^e as an fp32 bit pattern (e clamped to the normal range [-126, 127]).
__device__ __forceinline__ float pow2i(int e) {
    e = e < -126 ? -126 : (e > 127 ? 127 : e);
    return __int_as_float((e + 127) << 23);
}

// Token order of staged rows within a 64-token chunk (rows of d_h 16-bit
// values, contiguous).  A fragment load has lane (g, t) read word t (+ a
// constant) of row g of an 8-row tile; row i of tile j is token ctok<RS>(j, i)
// of the chunk: every RS-th token, tiles interleaved within groups of 8 RS
// tokens.  With w = d_h / 2 words per row the 8 rows of a tile start 4 words
// apart modulo 32, so the 32 lanes read 32 distinct banks, when RS = 4 for odd
// w (d_h = 30: 15-word rows, which collide two by two in token order) and
// RS = 2 for w = 2 mod 4; otherwise token order itself is conflict-free or no
// order is (w = 0 mod 8).  A contraction over tokens only needs its two
// operands in the same order, and each output row goes back to its own token,
// so the kernels pick the order freely.  Rows g and g + 8 of a 16-row tile tm
// are tiles 2 tm and 2 tm + 1: tokens mtok<RS>(tm, g) and that + mrow<RS>().
constexpr int row_step(int d) { return d <= 0 ? 1 : ((d / 2) % 2 == 1 ? 4 : ((d / 2) % 4 == 2 ? 2 : 1)); }
template <int RS>
__device__ __forceinline__ int ctok(int j, int i) {
    return 8 * RS * (j / RS) + (j % RS) + RS * i;
}
template <int RS>
__device__ __forceinline__ int mtok(int tm, int g) {
    return ctok<RS>(2 * tm, g);
}
template <int RS>
__host__ __device__ constexpr int mrow() {
    return RS == 1 ? 8 : 1;
}
static_assert(row_step(30) == 4 && row_step(28) == 2 && row_step(32) == 1 && row_step(0) == 1, "row steps");

// Shared scratch of the distributed core (m = 32, 64; see dist_core): two
// matrices of fp16 pairs (hi plane, then lo plane; rows padded to m + 8
// halves so ldmatrix is conflict-free) and an auxiliary float area.
template <int M>
struct DistScratch {
    static constexpr int CW = M / 16, SS = M + 8;
    static constexpr size_t PLANE = (size_t)M * SS * 2;
    static constexpr size_t MAT = 2 * PLANE;
    static constexpr size_t AUX = ((size_t)CW * M * 4 + 4 * CW * 4 + 15) / 16 * 16;  // column sums, maxima
    static constexpr size_t BYTES = ((2 * MAT + AUX + 127) / 128) * 128;
};

template <typename T, int M>
struct GlPark;  // parked G_L^n fragments (defined with the front phase)

template <typename T, int M, int NCOL, int TPW, int WPU, bool GLS, int CW = 1>
struct Layout {
    static constexpr int N = TPW * WPU;
    static constexpr int GW = WPU > CW ? WPU : CW;       // warps per group (token warps first)
    static constexpr int NCH = TPW / 64;                 // 64-token chunks per warp
    static constexpr int DS = (NCOL == 32) ? 30 : 32;    // staged row width bound (d_h <= DS)
    static constexpr int MT = (M + 15) / 16;             // landmark m-tiles
    static constexpr int MP = MT * 16;                   // padded landmark count
    static constexpr int LS = LmS<T>::LS;                // Qbar/Kbar row stride
    static constexpr int WS = NCOL + 4;                  // fp32 W row stride
    static constexpr int YS = YtS<T, M>::YS;             // Y^T row stride
    static constexpr int KTL = (M >= 16) ? M / 16 : 1;   // k-steps of O = G_L^n Y
    static constexpr int GLB = GlPark<T, M>::BYTES;      // bytes per lane per G_L fragment
    // per-warp private memory: stage (Q, K, V rows of the warp), G_L fragments
    static constexpr size_t STAGE = 3 * (size_t)TPW * DS * 2;
    static constexpr size_t GLF = STAGE;
    static constexpr size_t WARP_BYTES = ((GLF + (GLS ? (size_t)NCH * 4 * KTL * 32 * GLB : 0) + 127) / 128) * 128;
    // A warp's partial W (fp32 MP x NCOL, row stride WS, then MP row maxima)
    // lives in its stage right after the Q rows, once K and V are consumed.
    static constexpr size_t WPART = (size_t)TPW * DS * 2;
    static_assert(WPU == 1 || (size_t)MP * WS * 4 + MP * 4 <= 2 * (size_t)TPW * DS * 2,
                  "W partial must fit in K+V");
    // Distributed core (CW > 1): its scratch is group memory, or, with long
    // stages (TPW >= 256), the first two token warps' K/V rows (consumed by
    // the combine before the core starts; the next unit's K and V are copied
    // after the core).
    static constexpr bool SCR_IN_STAGE = (CW > 1) && (TPW >= 256);
    static constexpr bool SCR_IN_GROUP = (CW > 1) && !SCR_IN_STAGE;
    static constexpr size_t SCR_BYTES = SCR_IN_GROUP ? DistScratch<(M > 16 ? M : 32)>::BYTES : 0;
    static_assert(!SCR_IN_STAGE || (WPU >= 2 && DistScratch<(M > 16 ? M : 32)>::MAT +
                                                       DistScratch<(M > 16 ? M : 32)>::AUX <=
                                                   2 * (size_t)TPW * DS * 2),
                  "scratch must fit in two warps' K/V rows");
    static constexpr size_t QB_BYTES = LmS<T>::bytes(MP);
    static constexpr size_t YT_BYTES = YtS<T, M>::bytes(NCOL);
    // Per-group shared memory.  Y^T is written by the core once it has read
    // Qbar, W and m_U for the last time, so it overlays them when no warp can
    // write the next unit's landmarks or W while another still reads Y^T:
    // with one warp per unit, or when G_L^n is recomputed (the output is
    // followed by a group barrier before the next unit's Q lands); with the
    // distributed core, whose scratch starts after every core warp has read
    // its Qbar rows, the scratch overlays Qbar and Y^T overlays W and m_U.
    //   one-warp core:     Qbar | W | m_U | Kbar (| Y^T) | bars
    //   distributed core:  W | m_U | Kbar | bars | Qbar (inside the scratch)
    static constexpr bool YT_OVERLAY = SCR_IN_GROUP || (WPU == 1) || !GLS;
    static constexpr size_t G_W = SCR_IN_GROUP ? 0 : QB_BYTES;  // fp32 MP x WS
    static constexpr size_t G_MU = G_W + MP * WS * 4;           // m_U, log2 domain
    static constexpr size_t G_KBAR = ((G_MU + MP * 4 + 15) / 16) * 16;
    static constexpr size_t G_BAR = SCR_IN_GROUP ? ((G_KBAR + QB_BYTES + 15) / 16) * 16
                                                 : (((YT_OVERLAY ? G_KBAR + QB_BYTES : G_KBAR + QB_BYTES + YT_BYTES) +
                                                     15) / 16) * 16;
    static constexpr size_t G_BAR_END = G_BAR + 16 * WPU;  // two mbarriers per token warp
    static constexpr size_t G_QBAR = SCR_IN_GROUP ? ((G_BAR_END + 16 + 127) / 128) * 128 : 0;
    static constexpr size_t G_YT = SCR_IN_GROUP ? G_W : (YT_OVERLAY ? G_QBAR : G_KBAR + QB_BYTES);
    static_assert(!YT_OVERLAY || YT_BYTES <= (SCR_IN_GROUP ? G_KBAR : G_KBAR - G_QBAR),
                  "Y^T must fit over the regions it overlays");
    static constexpr size_t G_SCR = SCR_IN_GROUP ? G_QBAR : ((G_BAR_END + 16 + 127) / 128) * 128;
    static constexpr size_t GROUP_BYTES =
        ((SCR_IN_GROUP ? G_QBAR + (SCR_BYTES > QB_BYTES ? SCR_BYTES : QB_BYTES) : G_SCR) + 127) / 128 * 128;
    static constexpr size_t PER_GROUP = GROUP_BYTES + WPU * WARP_BYTES;
};

// C-layout fragments of an MP x MP fp32 matrix: f[i][n][e] is row
// 16i + g + 8(e >> 1), column 8n + 2t + (e & 1).
template <int MT>
using Frag = float[MT][2 * MT][4];
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
// ---- fp16 two-term split products for the m x m iteration ----
// A operand registers (m16n8k16 row layout) of every m-tile i and k-step kk,
// each register split into hi and lo halves.
template <int MT>
using HFrag = H2Pair[MT][MT][4];

// A operand from C-layout fragments: k-step kk spans n-tiles 2kk and 2kk+1.
template <int MT>
__device__ __forceinline__ void to_hfrag(const Frag<MT>& c, HFrag<MT>& a) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int kk = 0; kk < MT; ++kk) {
            a[i][kk][0] = split_h2(c[i][2 * kk][0], c[i][2 * kk][1]);
            a[i][kk][1] = split_h2(c[i][2 * kk][2], c[i][2 * kk][3]);
            a[i][kk][2] = split_h2(c[i][2 * kk + 1][0], c[i][2 * kk + 1][1]);
            a[i][kk][3] = split_h2(c[i][2 * kk + 1][2], c[i][2 * kk + 1][3]);
        }
}

// Multiply fragments by 2^e with e chosen so that max |f| lands in
// [2^10, 2^11) (fp16 headroom for the products); returns e (0 if f == 0).
template <int MT>
__device__ __forceinline__ int frag_normalise(Frag<MT>& f) {
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) mx = fmaxf(mx, fabsf(f[i][n][e]));
    mx = warp_max_nonneg(mx);
    if (!(mx > 0.f) || !(mx < INFINITY)) return 0;
    const int e = 10 - ilogbf(mx);
    const float s = pow2i(e);
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
            for (int k = 0; k < 4; ++k) f[i][n][k] *= s;
    return e;
}

// ---- symmetric operands in registers ----
// A operand register r of m-tile i, k-step kk holds the 8x8 block
// (2i + (r & 1), 2kk + (r >> 1)): row g, columns 2t and 2t + 1 of it.  The
// B operand of P^T is P's own A operand registers: k-step kk, n-tile j uses
// registers (j & 1) and 2 + (j & 1) of m-tile j >> 1.

// prmt selector that mirrors the lower triangle of a diagonal 8x8 block:
// element (g, 2t) keeps the lane's value when g >= 2t, else takes the
// transpose's, element (g, 2t + 1) likewise with g >= 2t + 1.
__device__ __forceinline__ uint32_t tril_selector(int g, int t) {
    return ((g >= 2 * t) ? 0x10u : 0x54u) | (((g >= 2 * t + 1) ? 0x32u : 0x76u) << 8);
}

template <int MT>
__device__ __forceinline__ H2Pair split_reg(const Frag<MT>& c, int i, int kk, int r, float s) {
    const int n = 2 * kk + (r >> 1), e = 2 * (r & 1);
    return split_h2(s * c[i][n][e], s * c[i][n][e + 1]);
}

// A operand of s*C split into fp16 pairs.
template <int MT>
__device__ __forceinline__ void to_hfrag_scaled(const Frag<MT>& c, HFrag<MT>& a, float s) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int kk = 0; kk < MT; ++kk)
#pragma unroll
            for (int r = 0; r < 4; ++r) a[i][kk][r] = split_reg<MT>(c, i, kk, r, s);
}

// A operand of the exactly symmetric matrix defined by the lower triangle of
// s*C: blocks below the diagonal are split from C, diagonal blocks mirror
// their lower triangle, blocks above are transposes of their mirror blocks.
// Taking one triangle removes the antisymmetric round-off of a product of
// symmetric factors before it can grow.
template <int MT>
__device__ __forceinline__ void sym_hfrag(const Frag<MT>& c, HFrag<MT>& a, uint32_t sel, float s) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int kk = 0; kk < MT; ++kk)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int R = 2 * i + (r & 1), C = 2 * kk + (r >> 1);
                if (R >= C) a[i][kk][r] = split_reg<MT>(c, i, kk, r, s);
                if (R == C) {
                    a[i][kk][r].hi = prmt(a[i][kk][r].hi, movmatrix_trans(a[i][kk][r].hi), sel);
                    a[i][kk][r].lo = prmt(a[i][kk][r].lo, movmatrix_trans(a[i][kk][r].lo), sel);
                }
            }
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int kk = 0; kk < MT; ++kk)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int R = 2 * i + (r & 1), C = 2 * kk + (r >> 1);
                if (R < C) {
                    const H2Pair src = a[C >> 1][R >> 1][(C & 1) + 2 * (R & 1)];
                    a[i][kk][r] = H2Pair{movmatrix_trans(src.hi), movmatrix_trans(src.lo)};
                }
            }
}

// A operand of P^T from P's A operand (8x8 block transposes).
template <int MT>
__device__ __forceinline__ void transpose_hfrag(const HFrag<MT>& a, HFrag<MT>& b) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int kk = 0; kk < MT; ++kk)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int R = 2 * i + (r & 1), C = 2 * kk + (r >> 1);
                const H2Pair src = a[C >> 1][R >> 1][(C & 1) + 2 * (R & 1)];
                b[i][kk][r] = H2Pair{movmatrix_trans(src.hi), movmatrix_trans(src.lo)};
            }
}

// D += A P^T with fp16 two-term split operands, the small terms lo*hi and
// hi*lo first, then hi*hi.
template <int MT>
__device__ __forceinline__ void mm_hT_acc(const HFrag<MT>& A, const HFrag<MT>& P, Frag<MT>& D) {
    using H = Mma16<__half>;
#pragma unroll
    for (int kk = 0; kk < MT; ++kk)
#pragma unroll
        for (int j = 0; j < 2 * MT; ++j) {
            const H2Pair b0 = P[j >> 1][kk][j & 1], b1 = P[j >> 1][kk][2 + (j & 1)];
#pragma unroll
            for (int i = 0; i < MT; ++i) {
                const uint32_t ahi[4] = {A[i][kk][0].hi, A[i][kk][1].hi, A[i][kk][2].hi, A[i][kk][3].hi};
                const uint32_t alo[4] = {A[i][kk][0].lo, A[i][kk][1].lo, A[i][kk][2].lo, A[i][kk][3].lo};
                H::k16(D[i][j], alo, b0.hi, b1.hi);
                H::k16(D[i][j], ahi, b0.lo, b1.lo);
                H::k16(D[i][j], ahi, b0.hi, b1.hi);
            }
        }
}

// D = s I.
template <int MT>
__device__ __forceinline__ void frag_diag(Frag<MT>& D, float s, int g, int t) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int j = 0; j < 2 * MT; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e)
                D[i][j][e] = ((16 * i + 8 * (e >> 1) + g) == (8 * j + (e & 1) + 2 * t)) ? s : 0.f;
}

// D += s (hi + lo) of the split A operand P, element by element (fp32): C-layout
// element (i, n, e) is half (e & 1) of register (e >> 1) | ((n & 1) << 1) of
// P's m-tile i, k-step n / 2.
template <int MT>
__device__ __forceinline__ void frag_add_h(Frag<MT>& D, const HFrag<MT>& P, float s) {
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const H2Pair x = P[i][n >> 1][h | ((n & 1) << 1)];
                const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&x.hi));
                const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&x.lo));
                D[i][n][2 * h] = fmaf(s, a.x + b.x, D[i][n][2 * h]);
                D[i][n][2 * h + 1] = fmaf(s, a.y + b.y, D[i][n][2 * h + 1]);
            }
}

// Largest |D| over the warp.
template <int MT>
__device__ __forceinline__ float frag_absmax(const Frag<MT>& D) {
    float mx = 0.f;
#pragma unroll
    for (int i = 0; i < MT; ++i)
#pragma unroll
        for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) mx = fmaxf(mx, fabsf(D[i][n][e]));
    return warp_max_nonneg(mx);
}

// Largest value over the warp (any sign).
__device__ __forceinline__ float warp_max_f(float x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}

// Exponent e with 2^e x in [2^10, 2^11) (0 when x is 0 or not finite): an
// fp16 pair of a matrix scaled so keeps 22 significant bits for every entry
// down to 2^-13 of its largest one.
__device__ __forceinline__ int h2_exponent(float x) { return (x > 0.f && x < INFINITY) ? 10 - ilogbf(x) : 0; }

// S_L for one 16-token tile of the stage and its G_L^n fragments (A operand
// of O = G_L^n Y, k = landmarks).  q0: row g of the tile (token mtok<RS>(tm,
// g) of its chunk); row g + 8 lies mrow<RS>() rows further on.
// BIAS: bl points at row g of the tile in the N x M block B_L of the score
// bias (row stride M); log2(e) B_L enters the exponent beside the scaled score.
template <typename T, int M, int KTL, bool BIAS = false, int RS = 1>
__device__ __forceinline__ void gl_tile(const T* q0, const T* kbar, int d, int g, int t, float sl2,
                                        typename Opnd<T>::DReg (&f)[KTL][4], const float* bl = nullptr) {
    using O = Opnd<T>;
    using R = typename O::Reg;
    constexpr int NTL = M / 8, LS = LmS<T>::LS, LO = LmS<T>::LO;
    R a[2][4];
    const T* q1 = q0 + mrow<RS>() * d;
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
        const int c0 = 16 * kk + 2 * t, c1 = c0 + 8;
        a[kk][0] = c0 < d ? O::ld(q0 + c0) : O::zero();
        a[kk][1] = c0 < d ? O::ld(q1 + c0) : O::zero();
        a[kk][2] = c1 < d ? O::ld(q0 + c1) : O::zero();
        a[kk][3] = c1 < d ? O::ld(q1 + c1) : O::zero();
    }
    float sl[NTL][4];
#pragma unroll
    for (int j = 0; j < NTL; ++j) {
        sl[j][0] = sl[j][1] = sl[j][2] = sl[j][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const T* kr = kbar + (8 * j + g) * LS + 16 * kk + 2 * t;
            O::mma(sl[j], a[kk], DSt<T>::ld(kr, LO), DSt<T>::ld(kr + 8, LO));
        }
    }
    if constexpr (BIAS) {  // scores in the log2 domain, bias included: e0/e1 below take them as they are
#pragma unroll
        for (int j = 0; j < NTL; ++j) {
            const float2 b0 = __ldg(reinterpret_cast<const float2*>(bl + 8 * j + 2 * t));
            const float2 b1 = __ldg(reinterpret_cast<const float2*>(bl + mrow<RS>() * M + 8 * j + 2 * t));
            sl[j][0] = fmaf(sl[j][0], sl2, kLog2e * b0.x);
            sl[j][1] = fmaf(sl[j][1], sl2, kLog2e * b0.y);
            sl[j][2] = fmaf(sl[j][2], sl2, kLog2e * b1.x);
            sl[j][3] = fmaf(sl[j][3], sl2, kLog2e * b1.y);
        }
    }
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int j = 0; j < NTL; ++j) {
        mx0 = fmaxf(mx0, fmaxf(sl[j][0], sl[j][1]));
        mx1 = fmaxf(mx1, fmaxf(sl[j][2], sl[j][3]));
    }
    const float ssl = BIAS ? 1.f : sl2;
    mx0 = quad_max(mx0) * ssl;
    mx1 = quad_max(mx1) * ssl;
    auto e0 = [&](float x) { return ex2(fmaf(x, ssl, -mx0)); };
    auto e1 = [&](float x) { return ex2(fmaf(x, ssl, -mx1)); };
    if constexpr (M >= 16) {
#pragma unroll
        for (int kk = 0; kk < KTL; ++kk) {
            f[kk][0] = O::dpk(e0(sl[2 * kk][0]), e0(sl[2 * kk][1]));
            f[kk][1] = O::dpk(e1(sl[2 * kk][2]), e1(sl[2 * kk][3]));
            f[kk][2] = O::dpk(e0(sl[2 * kk + 1][0]), e0(sl[2 * kk + 1][1]));
            f[kk][3] = O::dpk(e1(sl[2 * kk + 1][2]), e1(sl[2 * kk + 1][3]));
        }
    } else {
        f[0][0] = O::dpk(e0(sl[0][0]), e0(sl[0][1]));
        f[0][1] = O::dpk(e1(sl[0][2]), e1(sl[0][3]));
        f[0][2] = f[0][3] = O::dzero();
    }
}

// Parked G_L^n fragments: per lane and 16-token tile, KTL x 4 operand
// registers (m >= 16) or 2 (m = 8): single 16-bit registers (Single16 I/O:
// one or a half 16-byte vector per k-step) or hi + lo pairs (two or one).
template <typename T, int M>
struct GlPark {
    using R = typename Opnd<T>::DReg;
    static constexpr bool kPair = sizeof(R) == 8;
    static constexpr int REGS = (M >= 16) ? 4 : 2;              // registers per k-step
    static constexpr int BYTES = REGS * (int)sizeof(R);          // per lane per k-step
    static __device__ __forceinline__ void put(uint32_t* glf, int slot, const R (&f)[4]) {
        if constexpr (!kPair) {
            if constexpr (M >= 16)
                reinterpret_cast<uint4*>(glf)[slot] = make_uint4(f[0], f[1], f[2], f[3]);
            else
                reinterpret_cast<uint2*>(glf)[slot] = make_uint2(f[0], f[1]);
        } else if constexpr (M >= 16) {
            reinterpret_cast<uint4*>(glf)[2 * slot] = make_uint4(f[0].hi, f[1].hi, f[2].hi, f[3].hi);
            reinterpret_cast<uint4*>(glf)[2 * slot + 1] = make_uint4(f[0].lo, f[1].lo, f[2].lo, f[3].lo);
        } else {
            reinterpret_cast<uint4*>(glf)[slot] = make_uint4(f[0].hi, f[1].hi, f[0].lo, f[1].lo);
        }
    }
    static __device__ __forceinline__ void get(const uint32_t* glf, int slot, R (&f)[4]) {
        if constexpr (!kPair) {
            if constexpr (M >= 16) {
                const uint4 x = reinterpret_cast<const uint4*>(glf)[slot];
                f[0] = x.x; f[1] = x.y; f[2] = x.z; f[3] = x.w;
            } else {
                const uint2 x = reinterpret_cast<const uint2*>(glf)[slot];
                f[0] = x.x; f[1] = x.y; f[2] = f[3] = 0u;
            }
        } else {
            const uint4* p = reinterpret_cast<const uint4*>(glf);
            if constexpr (M >= 16) {
                const uint4 h = p[2 * slot], l = p[2 * slot + 1];
                f[0] = {h.x, l.x};
                f[1] = {h.y, l.y};
                f[2] = {h.z, l.z};
                f[3] = {h.w, l.w};
            } else {
                const uint4 x = p[slot];
                f[0] = {x.x, x.z};
                f[1] = {x.y, x.w};
                f[2] = f[3] = R{0u, 0u};
            }
        }
    }
};

// Landmark means of the segments one warp owns (Algorithm 1 step 1) on the
// tensor cores, transposed: xbar^T = X^T P^T with the staged tokens X as
// the A operand (features x tokens; fragments are 8x8 transposes of the
// row-major stage) and the averaging matrix P^T (P[j][t] = 1/L when token t
// lies in segment j; exact in 16 bits since L is a power of two) as B.  A
// 16-token k-step only meets the n-tiles of its own segments, so a warp
// issues 2 x TPW/16 products (x2 when L = 1).
//
// landmarks_acc adds one 64-token chunk X (tokens tok0..tok0+63 of the warp's
// range) to the accumulators c (features x the warp's LPW segments);
// landmarks_put stores the means as rows j0.. of xbar (LmS layout: hi + lo
// 16-bit pairs, or fp32 for fp32 I/O); columns >= d come out as zeros.
//
// PW > 0 pools square patches instead of segments: the window is PW tokens
// wide, a landmark averages a B x B patch (B^2 = L) and the patches of a
// patch row are numbered left to right.  A warp's token range starts on a
// patch-row boundary, so its landmarks are again LPW consecutive rows.
template <int L, int PW>
struct Pooling {
    static constexpr int B = (L == 1) ? 1 : (L == 4) ? 2 : (L == 16) ? 4 : (L == 64) ? 8 : (L == 256) ? 16 : 0;
    static constexpr int P = PW > 0 ? PW / (B > 0 ? B : 1) : 0;  // patches per patch row
    static_assert(PW == 0 || (B > 0 && B * B == L && PW % (B > 0 ? B : 1) == 0), "square patches must tile the window");
    // warp-local landmark of warp-local token tok
    static __device__ __forceinline__ int of(int tok) {
        if constexpr (PW == 0) return tok / L;
        else return ((tok / PW) / B) * P + (tok % PW) / B;
    }
    // n-tiles of landmarks (8 per tile) met by the 16 tokens tk .. tk+15
    static __device__ __forceinline__ int tile_lo(int tk) {
        if constexpr (PW == 0) return (tk / L) / 8;
        else return (((tk / PW) / B) * P) / 8;
    }
    static __device__ __forceinline__ int tile_hi(int tk) {
        if constexpr (PW == 0) return ((tk + 15) / L) / 8;
        else return ((((tk + 15) / PW) / B) * P + P - 1) / 8;
    }
};

template <typename T, int L, int LPW, int PW = 0, int RS = 1>
__device__ __forceinline__ void landmarks_acc(const T* X, int tok0, float (&c)[2][(LPW + 7) / 8][4], int d, int g,
                                              int t) {
    using O = Opnd<T>;
    using R = typename O::Reg;
    using Pool = Pooling<L, PW>;
    constexpr int NTJ = (LPW + 7) / 8;
    constexpr float inv = 1.f / (float)L;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {  // 16 tokens per k-step: 8-row tiles 2 ks and 2 ks + 1
        // A = X^T, features 16 mf + g (+8); k = 8 b + 2t (+1): token ctok(2 ks + b, 2t (+1))
        R a[2][4];
#pragma unroll
        for (int mf = 0; mf < 2; ++mf)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int f0 = 16 * mf + 8 * (r & 1) + 2 * t;
                const R x = f0 < d ? O::ld(X + ctok<RS>(2 * ks + (r >> 1), g) * d + f0) : O::zero();
                a[mf][r] = O::tr(x);
            }
        // the k-step's tokens lie in [lo, hi] of the chunk
        const int lo = 8 * RS * ((2 * ks) / RS), hi = 8 * RS * ((2 * ks + 1) / RS) + 8 * RS - 1;
        const int jlo = Pool::tile_lo(tok0 + lo), jhi = Pool::tile_hi(tok0 + hi - 15);
#pragma unroll
        for (int j = 0; j < NTJ; ++j) {
            if (j < jlo || j > jhi) continue;  // warp-uniform
            // B = P^T: the tokens of k = 2t (+1) (+8, +9), landmark 8j + g
            auto pv = [&](int tok) -> float { return (Pool::of(tok0 + tok) == 8 * j + g) ? inv : 0.f; };
            const R b0 = O::pk(pv(ctok<RS>(2 * ks, 2 * t)), pv(ctok<RS>(2 * ks, 2 * t + 1)));
            const R b1 = O::pk(pv(ctok<RS>(2 * ks + 1, 2 * t)), pv(ctok<RS>(2 * ks + 1, 2 * t + 1)));
#pragma unroll
            for (int mf = 0; mf < 2; ++mf) O::mma(c[mf][j], a[mf], b0, b1);
        }
    }
}

template <typename T, int LPW>
__device__ __forceinline__ void landmarks_put(const float (&c)[2][(LPW + 7) / 8][4], T* xbar, int j0, int g, int t) {
    constexpr int NTJ = (LPW + 7) / 8, LS = LmS<T>::LS, LO = LmS<T>::LO;
#pragma unroll
    for (int mf = 0; mf < 2; ++mf)
#pragma unroll
        for (int j = 0; j < NTJ; ++j)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int lm = 8 * j + 2 * t + (e & 1), f = 16 * mf + g + 8 * (e >> 1);
                if (lm < LPW) DSt<T>::put(xbar + (j0 + lm) * LS + f, LO, c[mf][j][e]);
            }
}

// Zero landmark rows lo .. hi - 1 of xbar (padding rows when m < 16), all 32
// feature columns of both parts; `idx0`, `step`: this thread's share.
template <typename T>
__device__ __forceinline__ void landmarks_zero(T* xbar, int lo, int hi, int idx0, int step) {
    constexpr int LS = LmS<T>::LS, LO = LmS<T>::LO;
    for (int idx = idx0; idx < (hi - lo) * 32; idx += step) DSt<T>::zero(xbar + (lo + (idx >> 5)) * LS + (idx & 31), LO);
}

// All TPW tokens of the warp (a multiple of 64), then the store.
template <typename T, int TPW, int L, int PW = 0, int RS = 1>
__device__ __forceinline__ void landmarks_mma(const T* X, T* xbar, int j0, int d, int g, int t) {
    constexpr int LPW = TPW / L, NTJ = (LPW + 7) / 8;
    float c[2][NTJ][4];
#pragma unroll
    for (int mf = 0; mf < 2; ++mf)
#pragma unroll
        for (int j = 0; j < NTJ; ++j) c[mf][j][0] = c[mf][j][1] = c[mf][j][2] = c[mf][j][3] = 0.f;
#pragma unroll
    for (int ch = 0; ch < TPW / 64; ++ch) landmarks_acc<T, L, LPW, PW, RS>(X + ch * 64 * d, ch * 64, c, d, g, t);
    landmarks_put<T, LPW>(c, xbar, j0, g, t);
}

// Front, U side, for one warp's NCH chunks of 64 tokens: S_U = Qbar K^T with a
// running row max, G_U^n = exp(S_U - m_U) fed straight from registers as the
// A operand of W_r = G_U^n [V | 1] (B fragments of [V | 1 | 0] by 8x8
// transposes; the ones column yields the denominator), rescaled online when
// the max grows.  W_r (MP x NCOL) is stored at dst with row stride ws after a
// warp sync (so every lane is done reading K and V); the row maxima (log2
// domain) are returned in mU.
// One 64-token chunk of the U side for one 16-landmark m-tile (A operand aq
// = Qbar rows; v0, v1: rows g, g + 8 are real landmarks): S_U = Qbar K^T,
// the running row maxima run0/run1 (log2 domain), w rescaled when they grow,
// G_U^n = exp(S_U - m) fed from registers as the A operand of
// w += G_U^n [V | 1] (B fragments of [V | 1 | 0] by 8x8 transposes; the ones
// column yields the denominator).
// BIAS: bu points at the chunk's first key in row g of the m-tile in the
// M x N block B_U of the score bias (row stride bn).
// RS: token order of the chunk's rows (n-tile nt, row i = token ctok<RS>(nt, i)).
template <typename T, int NCOL, bool BIAS = false, int RS = 1>
__device__ __forceinline__ void su_w_chunk(const typename Opnd<T>::DReg (&aq)[2][4], const T* Kc, const T* Vc, int d,
                                           int g, int t, float sl2, bool v0, bool v1, float (&w)[NCOL / 8][4],
                                           float& run0, float& run1, bool rescale, const float* bu = nullptr,
                                           int bn = 0) {
    using O = Opnd<T>;
    using R = typename O::Reg;
    constexpr int NTO = NCOL / 8;
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
        s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
        const T* kr = Kc + ctok<RS>(nt, g) * d;
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const int c0 = 16 * kk + 2 * t, c1 = c0 + 8;
            const R b0 = c0 < d ? O::ld(kr + c0) : O::zero();
            const R b1 = c1 < d ? O::ld(kr + c1) : O::zero();
            O::mma(s[nt], aq[kk], b0, b1);
        }
    }
    if constexpr (BIAS) {  // scores in the log2 domain, bias included (rows beyond m stay unbiased)
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            // keys of columns 2t, 2t + 1 of n-tile nt
            auto ld2 = [&](const float* p) -> float2 {
                if constexpr (RS == 1) return __ldg(reinterpret_cast<const float2*>(p + 8 * nt + 2 * t));
                else return make_float2(__ldg(p + ctok<RS>(nt, 2 * t)), __ldg(p + ctok<RS>(nt, 2 * t + 1)));
            };
            const float2 b0 = v0 ? ld2(bu) : make_float2(0.f, 0.f);
            const float2 b1 = v1 ? ld2(bu + 8 * bn) : make_float2(0.f, 0.f);
            s[nt][0] = fmaf(s[nt][0], sl2, kLog2e * b0.x);
            s[nt][1] = fmaf(s[nt][1], sl2, kLog2e * b0.y);
            s[nt][2] = fmaf(s[nt][2], sl2, kLog2e * b1.x);
            s[nt][3] = fmaf(s[nt][3], sl2, kLog2e * b1.y);
        }
    }
    const float ssl = BIAS ? 1.f : sl2;
    float mx0 = run0, mx1 = run1;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
        mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]) * ssl);
        mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]) * ssl);
    }
    mx0 = quad_max(mx0);
    mx1 = quad_max(mx1);
    if (rescale) {  // online rescaling of the accumulated rows
        const float f0 = ex2(run0 - mx0), f1 = ex2(run1 - mx1);
#pragma unroll
        for (int j = 0; j < NTO; ++j) {
            w[j][0] *= f0; w[j][1] *= f0; w[j][2] *= f1; w[j][3] *= f1;
        }
    }
    run0 = mx0;
    run1 = mx1;
    auto e0 = [&](float x) { return ex2(fmaf(x, ssl, -mx0)); };
    auto e1 = [&](float x) { return ex2(fmaf(x, ssl, -mx1)); };
#pragma unroll
    for (int kt = 0; kt < 4; ++kt) {
        typename O::DReg a[4];
        a[0] = v0 ? O::dpk(e0(s[2 * kt][0]), e0(s[2 * kt][1])) : O::dzero();
        a[1] = v1 ? O::dpk(e1(s[2 * kt][2]), e1(s[2 * kt][3])) : O::dzero();
        a[2] = v0 ? O::dpk(e0(s[2 * kt + 1][0]), e0(s[2 * kt + 1][1])) : O::dzero();
        a[3] = v1 ? O::dpk(e1(s[2 * kt + 1][2]), e1(s[2 * kt + 1][3])) : O::dzero();
#pragma unroll
        for (int j = 0; j < NTO; ++j) {
            const int c0 = 8 * j + 2 * t;
            const R x0 = c0 < d ? O::ld(Vc + ctok<RS>(2 * kt, g) * d + c0) : (c0 == d ? O::one() : O::zero());
            const R x1 = c0 < d ? O::ld(Vc + ctok<RS>(2 * kt + 1, g) * d + c0) : (c0 == d ? O::one() : O::zero());
            O::mma(w[j], a, O::tr(x0), O::tr(x1));
        }
    }
}

// A operand registers (hi + lo pairs) of Qbar's m-tile mt.
template <typename T>
__device__ __forceinline__ void qbar_afrag(const T* qbar, int mt, int g, int t, typename Opnd<T>::DReg (&aq)[2][4]) {
    constexpr int LS = LmS<T>::LS, LO = LmS<T>::LO;
#pragma unroll
    for (int kk = 0; kk < 2; ++kk) {
        const T* r0 = qbar + (16 * mt + g) * LS + 16 * kk + 2 * t;
        aq[kk][0] = DSt<T>::ld(r0, LO);
        aq[kk][1] = DSt<T>::ld(r0 + 8 * LS, LO);
        aq[kk][2] = DSt<T>::ld(r0 + 8, LO);
        aq[kk][3] = DSt<T>::ld(r0 + 8 * LS + 8, LO);
    }
}

// Front, U side, for one warp's NCH chunks of 64 tokens: su_w_chunk over the
// chunks for every landmark m-tile.  W_r (MP x NCOL) is stored at dst with
// row stride ws after a warp sync (so every lane is done reading K and V);
// the row maxima (log2 domain) are returned in mU.
// BIAS: bu is the unit's M x N block B_U of the score bias, offset to the
// first key of Ks (row stride bn).
template <typename T, int M, int NCOL, int NCH, bool BIAS = false, int RS = 1>
__device__ __forceinline__ void front_su_w(const T* qbar, const T* Ks, const T* Vs, int d, int g, int t, float sl2,
                                           float* dst, int ws, float (&mU)[(M + 15) / 16][2],
                                           const float* bu = nullptr, int bn = 0) {
    using R = typename Opnd<T>::DReg;
    constexpr int MT = (M + 15) / 16, NTO = NCOL / 8;
    float wall[MT][NTO][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
        R aq[2][4];
        qbar_afrag<T>(qbar, mt, g, t, aq);
        const bool v0 = (16 * mt + g) < M, v1 = (16 * mt + g + 8) < M;
        float(&w)[NTO][4] = wall[mt];
#pragma unroll
        for (int j = 0; j < NTO; ++j) w[j][0] = w[j][1] = w[j][2] = w[j][3] = 0.f;
        float run0 = -INFINITY, run1 = -INFINITY;
#pragma unroll 1
        for (int ch = 0; ch < NCH; ++ch)
            su_w_chunk<T, NCOL, BIAS, RS>(aq, Ks + ch * 64 * d, Vs + ch * 64 * d, d, g, t, sl2, v0, v1, w, run0, run1,
                                      NCH > 1, BIAS ? bu + (size_t)(16 * mt + g) * bn + ch * 64 : nullptr, bn);
        mU[mt][0] = run0;
        mU[mt][1] = run1;
    }
    __syncwarp();
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int j = 0; j < NTO; ++j) {
            const int rr = 16 * mt + g, c = 8 * j + 2 * t;
            *reinterpret_cast<float2*>(dst + rr * ws + c) = make_float2(wall[mt][j][0], wall[mt][j][1]);
            *reinterpret_cast<float2*>(dst + (rr + 8) * ws + c) = make_float2(wall[mt][j][2], wall[mt][j][3]);
        }
}

// Combine (several warps per unit): the warps' partial (W_r, m_r), stored in
// their stages at part0 + s * wstride (floats), merge in a fixed order into
// m_U = max_r m_r and W = sum_r 2^(m_r - m_U) W_r, exactly G_U^n [V | 1] with
// the max over all N keys.  Warp r of WPU handles every (WPU*32)-th element.
template <int MP, int NCOL, int WS, int WPU>
__device__ __forceinline__ void combine_partials(const float* part0, size_t wstride, float* mW, float* gmu, int r,
                                                 int lane) {
    for (int e = r * 32 + lane; e < MP * NCOL; e += WPU * 32) {
        const int i = e / NCOL, c = e - (e / NCOL) * NCOL;
        float mu = -INFINITY;
#pragma unroll
        for (int s2 = 0; s2 < WPU; ++s2) mu = fmaxf(mu, part0[(size_t)s2 * wstride + MP * WS + i]);
        float acc = 0.f;
#pragma unroll
        for (int s2 = 0; s2 < WPU; ++s2) {
            const float* ps = part0 + (size_t)s2 * wstride;
            acc = fmaf(ex2(ps[MP * WS + i] - mu), ps[i * WS + c], acc);
        }
        mW[i * WS + c] = acc;
        if (c == 0) gmu[i] = mu;
    }
}

// Core, one warp: G_A^n = exp(Qbar Kbar^T - m_U) (mU: row maxima of this
// warp's rows of S_U in the log2 domain), the iterative pseudo-inverse
// (step 4) and Y = Z W (W = G_U^n [V | 1], fp32 row-major with stride WS at
// mW), stored as Y^T (hi + lo B operand pairs, YtS layout) at yT.
//
// The iteration is run in registers on the symmetric X = A Z_k (Z_0 = a A^T):
// T2 = 15I - 7X + X X, T3 = 13I - X T2, Z <- Z T3/4 and X <- X T3/4 (equal to
// A Z_{k+1}; its factors are polynomials in X and commute).  X is kept exactly
// symmetric (lower triangle mirrored) after every update.  Scalar factors of
// Z (a and the power-of-two range scaling) are dropped: O is a ratio of two
// columns of G_L^n Z W, so they cancel.  Every matrix is split into fp16
// pairs at a power-of-two scale that puts its largest entry in [2^10, 2^11)
// (A once, X, -T2/4, T3/4 and Z every step), and the products are rescaled
// in fp32, so no operand underflows fp16 however small G_A^n's entries are
// (sharp attention: rows of G_A^n far below 1).
//
// DUMP (test-only stage dump): dbg receives G_A^n (M x M), Z (M x M) and
// Y = Z W (M x NCOL), row-major fp32, with the dropped factors restored.
// BIAS: ba is the unit's M x M block B_A of the score bias.
template <typename T, int M, int NCOL, bool DUMP = false, bool BIAS = false>
__device__ __forceinline__ void core_warp(const T* qbar, const T* kbar, const float (&mU)[(M + 15) / 16][2],
                                          const float* mW, T* yT, int iters, float sl2, int g, int t,
                                          float* dbg = nullptr, const float* ba = nullptr) {
    using O = Opnd<T>;
    using D = typename O::DReg;
    constexpr int MT = (M + 15) / 16, LS = LmS<T>::LS, LO = LmS<T>::LO, WS = NCOL + 4, NTO = NCOL / 8;
    constexpr int YS = YtS<T, M>::YS, YLO = YtS<T, M>::LO;
    const uint32_t sel = tril_selector(g, t);
    Frag<MT> Zc;
    HFrag<MT> Xh, Zh;
    int ex = 0;          // Xh holds 2^ex X
    float zscale = 1.f;  // DUMP: Z = zscale 2^-esum Zc
    int esum = 0;
    {
        Frag<MT> Ac;
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            D aq[2][4];
#pragma unroll
            for (int kk = 0; kk < 2; ++kk) {
                const T* r0 = qbar + (16 * mt + g) * LS + 16 * kk + 2 * t;
                aq[kk][0] = DSt<T>::ld(r0, LO);
                aq[kk][1] = DSt<T>::ld(r0 + 8 * LS, LO);
                aq[kk][2] = DSt<T>::ld(r0 + 8, LO);
                aq[kk][3] = DSt<T>::ld(r0 + 8 * LS + 8, LO);
            }
#pragma unroll
            for (int n = 0; n < 2 * MT; ++n) {
                float sa[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
                    const T* kr = kbar + (8 * n + g) * LS + 16 * kk + 2 * t;
                    O::mma(sa, aq[kk], DSt<T>::ld(kr, LO), DSt<T>::ld(kr + 8, LO));
                }
                // log2 of G_A^n (-inf outside the m x m block)
                const int r0 = 16 * mt + g, r1 = r0 + 8, c = 8 * n + 2 * t;
                if constexpr (BIAS) {  // log2(e) B_A joins the shift (c and c + 1 < M together: M is even)
                    const float2 b0 = (r0 < M && c < M) ? __ldg(reinterpret_cast<const float2*>(ba + r0 * M + c))
                                                        : make_float2(0.f, 0.f);
                    const float2 b1 = (r1 < M && c < M) ? __ldg(reinterpret_cast<const float2*>(ba + r1 * M + c))
                                                        : make_float2(0.f, 0.f);
                    Ac[mt][n][0] = (r0 < M && c < M) ? fmaf(sa[0], sl2, fmaf(kLog2e, b0.x, -mU[mt][0])) : -INFINITY;
                    Ac[mt][n][1] = (r0 < M && c + 1 < M) ? fmaf(sa[1], sl2, fmaf(kLog2e, b0.y, -mU[mt][0])) : -INFINITY;
                    Ac[mt][n][2] = (r1 < M && c < M) ? fmaf(sa[2], sl2, fmaf(kLog2e, b1.x, -mU[mt][1])) : -INFINITY;
                    Ac[mt][n][3] = (r1 < M && c + 1 < M) ? fmaf(sa[3], sl2, fmaf(kLog2e, b1.y, -mU[mt][1])) : -INFINITY;
                } else {
                    Ac[mt][n][0] = (r0 < M && c < M) ? fmaf(sa[0], sl2, -mU[mt][0]) : -INFINITY;
                    Ac[mt][n][1] = (r0 < M && c + 1 < M) ? fmaf(sa[1], sl2, -mU[mt][0]) : -INFINITY;
                    Ac[mt][n][2] = (r1 < M && c < M) ? fmaf(sa[2], sl2, -mU[mt][1]) : -INFINITY;
                    Ac[mt][n][3] = (r1 < M && c + 1 < M) ? fmaf(sa[3], sl2, -mU[mt][1]) : -INFINITY;
                }
            }
        }
        // 2^ea G_A^n with its largest entry in [2^10, 2^11): the shift enters
        // the exponent, so no entry underflows for being small in absolute
        // terms (sharp attention can put a whole row of G_A^n far below 1).
        int ea;
        {
            float lmax = -INFINITY;
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                    for (int e = 0; e < 4; ++e) lmax = fmaxf(lmax, Ac[i][n][e]);
            lmax = warp_max_f(lmax);
            ea = (lmax > -INFINITY && lmax < INFINITY) ? 10 - (int)floorf(lmax) : 0;
            const float fa = (float)ea;
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                    for (int e = 0; e < 4; ++e) Ac[i][n][e] = ex2(Ac[i][n][e] + fa);
        }
        // ||A||_inf (max row sum) and ||A||_1 (max column sum) of 2^ea A; A > 0.
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
        // a A A^T = (2^ea A)(2^ea A)^T / (||2^ea A||_1 ||2^ea A||_inf)
        const float x0 = 1.f / (warp_max_nonneg(rmax) * warp_max_nonneg(cmax));
        if constexpr (DUMP) {
            zscale = ldexpf(x0, ea);  // Z_0 = a A^T = x0 2^ea (2^ea A)^T
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int r = 16 * i + g + 8 * (e >> 1), c = 8 * n + 2 * t + (e & 1);
                        if (r < M && c < M) dbg[r * M + c] = ldexpf(Ac[i][n][e], -ea);
                    }
        }
        HFrag<MT> Ah;
        to_hfrag<MT>(Ac, Ah);
        transpose_hfrag<MT>(Ah, Zh);  // Z_0 = (2^ea A)^T (a and 2^ea dropped)
        frag_diag<MT>(Ac, 0.f, g, t);
        mm_hT_acc<MT>(Ah, Ah, Ac);  // X_0 = x0 Ac
        ex = h2_exponent(x0 * frag_absmax<MT>(Ac));
        sym_hfrag<MT>(Ac, Xh, sel, x0 * pow2i(ex));
        if (iters == 0) {
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int kk = 0; kk < MT; ++kk)
#pragma unroll
                    for (int r = 0; r < 4; ++r) {
                        const uint32_t hb = Zh[i][kk][r].hi, lb = Zh[i][kk][r].lo;
                        const float2 h = __half22float2(*reinterpret_cast<const __half2*>(&hb));
                        const float2 l = __half22float2(*reinterpret_cast<const __half2*>(&lb));
                        const int n = 2 * kk + (r >> 1), e = 2 * (r & 1);
                        Zc[i][n][e] = h.x + l.x;
                        Zc[i][n][e + 1] = h.y + l.y;
                    }
        }
    }

    // pseudo-inverse iteration (step 4).  X is split at a scale 2^ex chosen
    // from its largest entry; -T2/4 and T3/4 at the fixed 2^10 (X's
    // eigenvalues lie in [0, 1], so their entries stay within a few units).
    constexpr int kT = 10;
#pragma unroll 1
    for (int it = 0; it < iters; ++it) {
        Frag<MT> F;
        HFrag<MT> Th;
        // 2^(2 ex) T2 = 2^(2 ex) (15 I - 7 X) + (2^ex X)(2^ex X)
        const float sx = pow2i(ex);
        frag_diag<MT>(F, 15.f * sx * sx, g, t);
        frag_add_h<MT>(F, Xh, -7.f * sx);
        mm_hT_acc<MT>(Xh, Xh, F);
        to_hfrag_scaled<MT>(F, Th, -0.25f * pow2i(kT - 2 * ex));  // 2^kT (-T2/4)
        // 2^(ex + kT) T3/4 = 2^(ex + kT) 13/4 I + (2^ex X)(2^kT (-T2/4))
        frag_diag<MT>(F, 3.25f * pow2i(ex + kT), g, t);
        mm_hT_acc<MT>(Xh, Th, F);
        to_hfrag_scaled<MT>(F, Th, pow2i(-ex));  // 2^kT T3/4
        frag_diag<MT>(Zc, 0.f, g, t);
        mm_hT_acc<MT>(Zh, Th, Zc);  // Z 2^kT T3/4
        if constexpr (DUMP) esum += kT;
        if (it + 1 < iters) {
            frag_diag<MT>(F, 0.f, g, t);
            mm_hT_acc<MT>(Xh, Th, F);  // 2^(ex + kT) X T3/4
            const float f = pow2i(-(ex + kT));
            const int en = h2_exponent(f * frag_absmax<MT>(F));
            sym_hfrag<MT>(F, Xh, sel, f * pow2i(en));
            ex = en;
            const int ez = frag_normalise<MT>(Zc);
            if constexpr (DUMP) esum += ez;
            to_hfrag<MT>(Zc, Zh);
        }
    }
    if constexpr (DUMP) {
        const float zs = ldexpf(zscale, -esum);
#pragma unroll
        for (int i = 0; i < MT; ++i)
#pragma unroll
            for (int n = 0; n < 2 * MT; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int r = 16 * i + g + 8 * (e >> 1), c = 8 * n + 2 * t + (e & 1);
                    if (r < M && c < M) dbg[M * M + r * M + c] = zs * Zc[i][n][e];
                }
    }

    // Y = Z W (split-tf32), stored as Y^T (hi + lo B operand pairs)
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
        if constexpr (DUMP) {
            const float zs = ldexpf(zscale, -esum);
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int j = 0; j < NTO; ++j)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int r = 16 * i + g + 8 * (e >> 1), c = 8 * j + 2 * t + (e & 1);
                        if (r < M) dbg[2 * M * M + r * NCOL + c] = zs * y[i][j][e];
                    }
        }
        // fp16 has a narrow range: Y is scaled by a power of two.  Numerator
        // and denominator columns share the factor, so it cancels in step 7.
        float scale = 1.f;
        if (O::kNarrowRange) {
            float ymax = 0.f;
#pragma unroll
            for (int i = 0; i < MT; ++i)
#pragma unroll
                for (int j = 0; j < NTO; ++j)
#pragma unroll
                    for (int e = 0; e < 4; ++e) ymax = fmaxf(ymax, fabsf(y[i][j][e]));
            ymax = warp_max_nonneg(ymax);
            if (ymax > 0.f && ymax < INFINITY) scale = pow2i(14 - ilogbf(ymax));
        }
        __syncwarp();  // Y^T may overlay the landmarks and W: every lane has read them
#pragma unroll
        for (int i = 0; i < MT; ++i)
#pragma unroll
            for (int j = 0; j < NTO; ++j) {
                const int rr = 16 * i + g, c = 8 * j + 2 * t;
                DSt<T>::put(yT + c * YS + rr, YLO, y[i][j][0] * scale);
                DSt<T>::put(yT + (c + 1) * YS + rr, YLO, y[i][j][1] * scale);
                DSt<T>::put(yT + c * YS + rr + 8, YLO, y[i][j][2] * scale);
                DSt<T>::put(yT + (c + 1) * YS + rr + 8, YLO, y[i][j][3] * scale);
            }
    }
}

// ---- distributed core for m = 32, 64: CW = m/16 warps, warp c owns rows 16c..16c+15 ----
// The m x m operands no longer fit one warp's registers.  Each warp keeps the
// A operands of its own rows (X and Z, fp16 pairs) and reads right-hand
// factors from two shared-memory matrices (hi and lo planes, rows padded to
// m + 8 halves so ldmatrix is conflict-free) that alternate roles: X in one,
// -T2/4 in the other, T3/4 over X once every warp has used X, the next X over
// -T2/4 once every warp has used it; three barriers per step.

template <int M>
__device__ __forceinline__ void dist_store(unsigned char* mat, int row, int col, const H2Pair& p) {
    constexpr int SS = DistScratch<M>::SS;
    *reinterpret_cast<uint32_t*>(mat + ((size_t)row * SS + col) * 2) = p.hi;
    *reinterpret_cast<uint32_t*>(mat + DistScratch<M>::PLANE + ((size_t)row * SS + col) * 2) = p.lo;
}

// Own rows of s*acc into a scratch matrix.
template <int M>
__device__ __forceinline__ void dist_put(unsigned char* mat, const float (&acc)[M / 8][4], float s, int c, int g,
                                         int t) {
#pragma unroll
    for (int n = 0; n < M / 8; ++n) {
        dist_store<M>(mat, 16 * c + g, 8 * n + 2 * t, split_h2(s * acc[n][0], s * acc[n][1]));
        dist_store<M>(mat, 16 * c + g + 8, 8 * n + 2 * t, split_h2(s * acc[n][2], s * acc[n][3]));
    }
}

// The symmetric matrix defined by the lower triangle of s*acc: own blocks on
// and below the diagonal (diagonal blocks mirrored) and their transposes.
template <int M>
__device__ __forceinline__ void dist_put_sym(unsigned char* mat, const float (&acc)[M / 8][4], float s, int c,
                                             int g, int t, uint32_t sel) {
#pragma unroll
    for (int n = 0; n < M / 8; ++n)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int R = 2 * c + h;
            if (R < n) continue;  // warp-uniform
            H2Pair p = split_h2(s * acc[n][2 * h], s * acc[n][2 * h + 1]);
            if (R == n) {
                p.hi = prmt(p.hi, movmatrix_trans(p.hi), sel);
                p.lo = prmt(p.lo, movmatrix_trans(p.lo), sel);
                dist_store<M>(mat, 8 * R + g, 8 * n + 2 * t, p);
            } else {
                dist_store<M>(mat, 8 * R + g, 8 * n + 2 * t, p);
                dist_store<M>(mat, 8 * n + g, 8 * R + 2 * t,
                              H2Pair{movmatrix_trans(p.hi), movmatrix_trans(p.lo)});
            }
        }
}

// A operand of the own rows (tr: of the transpose's own rows) from a scratch matrix.
template <int M, bool TR>
__device__ __forceinline__ void dist_load_a(const unsigned char* mat, H2Pair (&a)[M / 16][4], int c, int lane) {
    constexpr int SS = DistScratch<M>::SS;
    const int blk = lane >> 3, rr = lane & 7;
#pragma unroll
    for (int kk = 0; kk < M / 16; ++kk) {
        int row, col;
        if (TR) {
            row = 16 * kk + 8 * (blk >> 1) + rr;
            col = 16 * c + 8 * (blk & 1);
        } else {
            row = 16 * c + 8 * (blk & 1) + rr;
            col = 16 * kk + 8 * (blk >> 1);
        }
        uint32_t h[4], l[4];
        const unsigned char* ph = mat + ((size_t)row * SS + col) * 2;
        if (TR) {
            ldsm_x4_t(h, ph);
            ldsm_x4_t(l, ph + DistScratch<M>::PLANE);
        } else {
            ldsm_x4(h, ph);
            ldsm_x4(l, ph + DistScratch<M>::PLANE);
        }
#pragma unroll
        for (int r = 0; r < 4; ++r) a[kk][r] = H2Pair{h[r], l[r]};
    }
}

// acc[a] = s I + A_a P^T over the own rows for NA left operands sharing the
// right factor P (all m rows, from scratch); with CI also adds (-7I) P^T,
// whose own-row block lies in k-step c (i7: its diagonal A register).
template <int M, int NA, bool CI>
__device__ __forceinline__ void dist_mm(const H2Pair (*const (&A)[NA])[4], const unsigned char* mat,
                                        float (*const (&acc)[NA])[4], float s, uint32_t i7, int c, int g, int t,
                                        int lane) {
    using H = Mma16<__half>;
    constexpr int SS = DistScratch<M>::SS, NT = M / 8;
#pragma unroll
    for (int a = 0; a < NA; ++a)
#pragma unroll
        for (int n = 0; n < NT; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e)
                acc[a][n][e] = ((16 * c + 8 * (e >> 1) + g) == (8 * n + (e & 1) + 2 * t)) ? s : 0.f;
    const int blk = lane >> 3, rr = lane & 7;
#pragma unroll
    for (int kk = 0; kk < M / 16; ++kk)
#pragma unroll
        for (int jp = 0; jp < NT / 2; ++jp) {
            uint32_t bh[4], bl[4];
            const unsigned char* ph = mat + ((size_t)(16 * jp + 8 * (blk >> 1) + rr) * SS + 16 * kk + 8 * (blk & 1)) * 2;
            ldsm_x4(bh, ph);
            ldsm_x4(bl, ph + DistScratch<M>::PLANE);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int n = 2 * jp + h;
#pragma unroll
                for (int a = 0; a < NA; ++a) {
                    const H2Pair* Ak = A[a][kk];
                    const uint32_t ahi[4] = {Ak[0].hi, Ak[1].hi, Ak[2].hi, Ak[3].hi};
                    const uint32_t alo[4] = {Ak[0].lo, Ak[1].lo, Ak[2].lo, Ak[3].lo};
                    H::k16(acc[a][n], alo, bh[2 * h], bh[2 * h + 1]);
                    H::k16(acc[a][n], ahi, bl[2 * h], bl[2 * h + 1]);
                    H::k16(acc[a][n], ahi, bh[2 * h], bh[2 * h + 1]);
                }
                if (CI && kk == c) {
                    const uint32_t ci[4] = {i7, 0u, 0u, i7};
                    H::k16(acc[0][n], ci, bl[2 * h], bl[2 * h + 1]);
                    H::k16(acc[0][n], ci, bh[2 * h], bh[2 * h + 1]);
                }
            }
        }
}

// Core on CW = M/16 warps (warp c of them calls with its index; bar_id is a
// named barrier reserved for these warps; mat0, mat1, aux: DistScratch
// areas): G_A^n from the landmarks and m_U (gmu, log2 domain), the iteration
// of step 4, Y = Z W (W: fp32, row stride NCOL + 4 at mW) stored as Y^T at
// yT.  Same arithmetic as core_warp, except that X, -T2/4 and T3/4 are split
// at the fixed scale 2^10 (their entries stay within a few units, since X's
// eigenvalues lie in [0, 1]), which saves a barrier per scale; A is split at
// 2^ea with its largest entry in [2^10, 2^11), Z renormalised every step.
template <typename T, int M, int NCOL>
__device__ __forceinline__ void dist_core(const T* qbar, const T* kbar, const float* gmu, const float* mW, T* yT,
                                          unsigned char* mat0, unsigned char* mat1, float* aux, int iters, float sl2,
                                          int c, int lane, int bar_id) {
    using S = DistScratch<M>;
    using O = Opnd<T>;
    using D = typename O::DReg;
    constexpr int CW = S::CW, KT = M / 16, NT = M / 8, LS = LmS<T>::LS, LO = LmS<T>::LO, WS = NCOL + 4,
                  NTO = NCOL / 8, YS = YtS<T, M>::YS, YLO = YtS<T, M>::LO;
    const int g = lane >> 2, t = lane & 3;
    unsigned char* cur = mat0;
    unsigned char* oth = mat1;
    float* cols = aux;                // [CW][M] column-sum partials
    float* slots = aux + CW * M;      // [4][CW] maxima
    auto csync = [&]() { named_barrier(bar_id, CW * 32); };
    const uint32_t sel = tril_selector(g, t);
    constexpr float kS = 1024.f, kS2 = 1048576.f;  // fixed scale 2^10 of X, -T2/4, T3/4 (and its square)
    uint32_t i7;  // A operand register of -7 kS I's diagonal blocks
    {
        const __half2 h = __floats2half2_rn(g == 2 * t ? -7.f * kS : 0.f, g == 2 * t + 1 ? -7.f * kS : 0.f);
        i7 = *reinterpret_cast<const uint32_t*>(&h);
    }
    H2Pair Xa[KT][4], Za[KT][4];
    float acc[NT][4], zc[NT][4];
    // ---- G_A^n, own rows ----
    {
        D aq[2][4];
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const T* r0 = qbar + (16 * c + g) * LS + 16 * kk + 2 * t;
            aq[kk][0] = DSt<T>::ld(r0, LO);
            aq[kk][1] = DSt<T>::ld(r0 + 8 * LS, LO);
            aq[kk][2] = DSt<T>::ld(r0 + 8, LO);
            aq[kk][3] = DSt<T>::ld(r0 + 8 * LS + 8, LO);
        }
        const float mu0 = gmu[16 * c + g], mu1 = gmu[16 * c + g + 8];
#pragma unroll
        for (int n = 0; n < NT; ++n) {
            float sa[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int kk = 0; kk < 2; ++kk) {
                const T* kr = kbar + (8 * n + g) * LS + 16 * kk + 2 * t;
                O::mma(sa, aq[kk], DSt<T>::ld(kr, LO), DSt<T>::ld(kr + 8, LO));
            }
            acc[n][0] = fmaf(sa[0], sl2, -mu0);  // log2 of G_A^n
            acc[n][1] = fmaf(sa[1], sl2, -mu0);
            acc[n][2] = fmaf(sa[2], sl2, -mu1);
            acc[n][3] = fmaf(sa[3], sl2, -mu1);
        }
    }
    // 2^ea G_A^n with its largest entry in [2^10, 2^11) (the shift enters the
    // exponent, as in core_warp)
    {
        float lm = -INFINITY;
#pragma unroll
        for (int n = 0; n < NT; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) lm = fmaxf(lm, acc[n][e]);
        lm = warp_max_f(lm);
        if (lane == 0) slots[3 * CW + c] = lm;
        csync();
        float lmax = -INFINITY;
#pragma unroll
        for (int w = 0; w < CW; ++w) lmax = fmaxf(lmax, slots[3 * CW + w]);
        const float fa = (lmax > -INFINITY && lmax < INFINITY) ? (float)(10 - (int)floorf(lmax)) : 0.f;
#pragma unroll
        for (int n = 0; n < NT; ++n)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[n][e] = ex2(acc[n][e] + fa);
    }
    // ---- ||A||_inf, ||A||_1 (A > 0) and A into scratch ----
    {
        float r0 = 0.f, r1 = 0.f;
#pragma unroll
        for (int n = 0; n < NT; ++n) {
            r0 += acc[n][0] + acc[n][1];
            r1 += acc[n][2] + acc[n][3];
        }
        r0 += __shfl_xor_sync(0xffffffffu, r0, 1);
        r0 += __shfl_xor_sync(0xffffffffu, r0, 2);
        r1 += __shfl_xor_sync(0xffffffffu, r1, 1);
        r1 += __shfl_xor_sync(0xffffffffu, r1, 2);
        const float rm = warp_max_nonneg(fmaxf(r0, r1));
        if (lane == 0) slots[c] = rm;
#pragma unroll
        for (int n = 0; n < NT; ++n)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                float cs = acc[n][e] + acc[n][e + 2];
                cs += __shfl_xor_sync(0xffffffffu, cs, 4);
                cs += __shfl_xor_sync(0xffffffffu, cs, 8);
                cs += __shfl_xor_sync(0xffffffffu, cs, 16);
                if (g == 0) cols[c * M + 8 * n + 2 * t + e] = cs;
            }
    }
    dist_put<M>(cur, acc, 1.f, c, g, t);  // 2^ea A
    csync();
    float alpha;  // a A A^T = alpha (2^ea A)(2^ea A)^T
    {
        float rmax = 0.f, cmax = 0.f;
#pragma unroll
        for (int w = 0; w < CW; ++w) rmax = fmaxf(rmax, slots[w]);
        for (int col = lane; col < M; col += 32) {
            float cs = 0.f;
#pragma unroll
            for (int w = 0; w < CW; ++w) cs += cols[w * M + col];
            cmax = fmaxf(cmax, cs);
        }
        alpha = 1.f / (rmax * warp_max_nonneg(cmax));
    }
    {
        H2Pair Aa[KT][4];
#pragma unroll
        for (int kk = 0; kk < KT; ++kk)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const int n = 2 * kk + (r >> 1), e = 2 * (r & 1);
                Aa[kk][r] = split_h2(acc[n][e], acc[n][e + 1]);
            }
        const H2Pair(*const As[1])[4] = {Aa};
        float(*const Ds[1])[4] = {acc};
        dist_mm<M, 1, false>(As, cur, Ds, 0.f, 0u, c, g, t, lane);  // (2^ea A)(2^ea A)^T
    }
    dist_load_a<M, true>(cur, Za, c, lane);  // Z_0 = (2^ea A)^T (a and 2^ea dropped)
    dist_put_sym<M>(oth, acc, kS * alpha, c, g, t, sel);  // kS X_0
    csync();
    dist_load_a<M, false>(oth, Xa, c, lane);
    {
        unsigned char* tmp = cur;
        cur = oth;
        oth = tmp;
    }
    if (iters == 0) {
#pragma unroll
        for (int kk = 0; kk < KT; ++kk)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                const uint32_t hb = Za[kk][r].hi, lb = Za[kk][r].lo;
                const float2 h = __half22float2(*reinterpret_cast<const __half2*>(&hb));
                const float2 l = __half22float2(*reinterpret_cast<const __half2*>(&lb));
                const int n = 2 * kk + (r >> 1), e = 2 * (r & 1);
                zc[n][e] = h.x + l.x;
                zc[n][e + 1] = h.y + l.y;
            }
    }
    // ---- iteration (step 4): X in cur ----
#pragma unroll 1
    for (int it = 0; it < iters; ++it) {
        {
            const H2Pair(*const As[1])[4] = {Xa};
            float(*const Ds[1])[4] = {acc};
            dist_mm<M, 1, true>(As, cur, Ds, 15.f * kS2, i7, c, g, t, lane);  // kS^2 T2 = kS^2 (15I - 7X + X X)
        }
        dist_put<M>(oth, acc, -0.25f / kS, c, g, t);  // kS (-T2/4)
        csync();
        {
            const H2Pair(*const As[1])[4] = {Xa};
            float(*const Ds[1])[4] = {acc};
            dist_mm<M, 1, false>(As, oth, Ds, 3.25f * kS2, 0u, c, g, t, lane);  // kS^2 T3/4
        }
        dist_put<M>(cur, acc, 1.f / kS, c, g, t);  // kS T3/4 (every warp is done with X)
        csync();
        if (it + 1 < iters) {
            const H2Pair(*const As[2])[4] = {Za, Xa};
            float(*const Ds[2])[4] = {zc, acc};
            dist_mm<M, 2, false>(As, cur, Ds, 0.f, 0u, c, g, t, lane);  // Z kS T3/4, kS^2 X T3/4
            dist_put_sym<M>(oth, acc, 1.f / kS, c, g, t, sel);       // every warp is done with -T2/4
            float zm = 0.f;
#pragma unroll
            for (int n = 0; n < NT; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) zm = fmaxf(zm, fabsf(zc[n][e]));
            zm = warp_max_nonneg(zm);
            if (lane == 0) slots[CW + c] = zm;
            csync();
            dist_load_a<M, false>(oth, Xa, c, lane);
            unsigned char* tmp = cur;
            cur = oth;
            oth = tmp;
            float zmax = 0.f;
#pragma unroll
            for (int w = 0; w < CW; ++w) zmax = fmaxf(zmax, slots[CW + w]);
            const float sc = (zmax > 0.f && zmax < INFINITY) ? pow2i(10 - ilogbf(zmax)) : 1.f;
#pragma unroll
            for (int kk = 0; kk < KT; ++kk)
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const int n = 2 * kk + (r >> 1), e = 2 * (r & 1);
                    Za[kk][r] = split_h2(sc * zc[n][e], sc * zc[n][e + 1]);
                }
        } else {
            const H2Pair(*const As[1])[4] = {Za};
            float(*const Ds[1])[4] = {zc};
            dist_mm<M, 1, false>(As, cur, Ds, 0.f, 0u, c, g, t, lane);  // Z T3/4
        }
    }
    // ---- Y = Z W, own rows (split-tf32), stored as Y^T ----
    {
        float y[NTO][4];
#pragma unroll
        for (int j = 0; j < NTO; ++j) y[j][0] = y[j][1] = y[j][2] = y[j][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < NT; ++kk) {
            const uint32_t ah[4] = {__float_as_uint(zc[kk][0]), __float_as_uint(zc[kk][2]), __float_as_uint(zc[kk][1]),
                                    __float_as_uint(zc[kk][3])};
            const uint32_t al[4] = {tf32_lo(zc[kk][0]), tf32_lo(zc[kk][2]), tf32_lo(zc[kk][1]), tf32_lo(zc[kk][3])};
#pragma unroll
            for (int j = 0; j < NTO; ++j) {
                const float y0 = mW[(8 * kk + 2 * t) * WS + 8 * j + g];
                const float y1 = mW[(8 * kk + 2 * t + 1) * WS + 8 * j + g];
                const uint32_t bh0 = __float_as_uint(y0), bh1 = __float_as_uint(y1);
                const uint32_t bl0 = tf32_lo(y0), bl1 = tf32_lo(y1);
                mma_tf32(y[j], al[0], al[1], al[2], al[3], bh0, bh1);
                mma_tf32(y[j], ah[0], ah[1], ah[2], ah[3], bl0, bl1);
                mma_tf32(y[j], ah[0], ah[1], ah[2], ah[3], bh0, bh1);
            }
        }
        float scale = 1.f;
        if (O::kNarrowRange) {
            float ym = 0.f;
#pragma unroll
            for (int j = 0; j < NTO; ++j)
#pragma unroll
                for (int e = 0; e < 4; ++e) ym = fmaxf(ym, fabsf(y[j][e]));
            ym = warp_max_nonneg(ym);
            if (lane == 0) slots[2 * CW + c] = ym;
            csync();
            float ymax = 0.f;
#pragma unroll
            for (int w = 0; w < CW; ++w) ymax = fmaxf(ymax, slots[2 * CW + w]);
            if (ymax > 0.f && ymax < INFINITY) scale = pow2i(14 - ilogbf(ymax));
        }
        csync();  // Y^T may overlay W, which every core warp reads in full
#pragma unroll
        for (int j = 0; j < NTO; ++j) {
            const int rr = 16 * c + g, cc = 8 * j + 2 * t;
            DSt<T>::put(yT + cc * YS + rr, YLO, y[j][0] * scale);
            DSt<T>::put(yT + (cc + 1) * YS + rr, YLO, y[j][1] * scale);
            DSt<T>::put(yT + cc * YS + rr + 8, YLO, y[j][2] * scale);
            DSt<T>::put(yT + (cc + 1) * YS + rr + 8, YLO, y[j][3] * scale);
        }
    }
}

// Output for one warp's NCH chunks: O = (G_L^n Y_:d) / (G_L^n Y_d) (steps
// 5-7); G_L^n fragments come from glf (parked) or are recomputed from Qs and
// Kbar; rows are written row-major to obase (N_w x d), each to its own token
// (tiles in the RS token order of the chunks).
// BIAS (recomputed G_L^n only): bl is B_L of the score bias at the warp's
// first token (row stride M).
template <typename T, int M, int NCOL, int NCH, bool GLS, bool BIAS = false, int RS = 1>
__device__ __forceinline__ void output_rows(const uint32_t* glf, const T* Qs, const T* kbar, const T* yT,
                                            T* obase, int d, int g, int t, int lane, float sl2,
                                            const float* bl = nullptr) {
    using O = Opnd<T>;
    using R = typename O::DReg;
    constexpr int KTL = (M >= 16) ? M / 16 : 1, NTO = NCOL / 8, YS = YtS<T, M>::YS, YLO = YtS<T, M>::LO;
    R by[KTL][NTO][2];
#pragma unroll
    for (int kk = 0; kk < KTL; ++kk)
#pragma unroll
        for (int j = 0; j < NTO; ++j) {
            const T* yr = yT + (8 * j + g) * YS + 16 * kk + 2 * t;
            by[kk][j][0] = DSt<T>::ld(yr, YLO);
            by[kk][j][1] = (M >= 16) ? DSt<T>::ld(yr + 8, YLO) : O::dzero();
        }
    const int jd = d >> 3, tdn = (d & 7) >> 1;
    const int src = (lane & ~3) | tdn;
#pragma unroll 1
    for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
        for (int tm = 0; tm < 4; ++tm) {
            R f[KTL][4];
            if constexpr (GLS) {
#pragma unroll
                for (int kk = 0; kk < KTL; ++kk) GlPark<T, M>::get(glf, ((ch * 4 + tm) * KTL + kk) * 32 + lane, f[kk]);
            } else {
                gl_tile<T, M, KTL, BIAS, RS>(Qs + (ch * 64 + mtok<RS>(tm, g)) * d, kbar, d, g, t, sl2, f,
                                             BIAS ? bl + (size_t)(ch * 64 + mtok<RS>(tm, g)) * M : nullptr);
            }
            float o[NTO][4];
#pragma unroll
            for (int j = 0; j < NTO; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
            if constexpr (M >= 16) {
#pragma unroll
                for (int kk = 0; kk < KTL; ++kk)
#pragma unroll
                    for (int j = 0; j < NTO; ++j) O::mma(o[j], f[kk], by[kk][j][0], by[kk][j][1]);
            } else {
#pragma unroll
                for (int j = 0; j < NTO; ++j) O::mma8(o[j], f[0][0], f[0][1], by[0][j][0]);
            }
            float d0 = 0.f, d1 = 0.f;
#pragma unroll
            for (int j = 0; j < NTO; ++j)
                if (j == jd) {
                    d0 = o[j][0];
                    d1 = o[j][2];
                }
            const float i0 = __fdividef(1.f, __shfl_sync(0xffffffffu, d0, src));
            const float i1 = __fdividef(1.f, __shfl_sync(0xffffffffu, d1, src));
            T* o0 = obase + (ch * 64 + mtok<RS>(tm, g)) * d;
            T* o1 = o0 + mrow<RS>() * d;
#pragma unroll
            for (int j = 0; j < NTO; ++j) {
                const int c = 8 * j + 2 * t;
                if (c < d) {
                    O::st2(o0 + c, o[j][0] * i0, o[j][1] * i0);
                    O::st2(o1 + c, o[j][2] * i1, o[j][3] * i1);
                }
            }
        }
}

template <typename T, int M, int NCOL, int TPW, int WPU, int GROUPS, bool GLS, int CW>
__global__ void __launch_bounds__(GROUPS * Layout<T, M, NCOL, TPW, WPU, GLS, CW>::GW * 32, 1)
nystra_tc_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                 T* __restrict__ out, long long n_units, int d, int iters, float sl2,
                 unsigned int* fault, int active) {
    using Lay = Layout<T, M, NCOL, TPW, WPU, GLS, CW>;
    constexpr int N = Lay::N, NCH = Lay::NCH, MT = Lay::MT, MP = Lay::MP, WS = Lay::WS, KTL = Lay::KTL,
                  GW = Lay::GW;
    constexpr int L = N / M;      // tokens per landmark segment (<= TPW)
    constexpr int LPW = TPW / L;  // landmarks owned by one warp
    static_assert(sizeof(T) == 2, "the grouped kernel takes 16-bit I/O (its layout assumes it)");
    static_assert(L <= TPW && TPW % L == 0, "segments must not straddle warps");
    static_assert(CW == 1 || CW == M / 16, "the distributed core has one warp per 16 landmarks");

    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = warp / GW, r = warp - grp * GW;
    const bool tok = (GW == WPU) || r < WPU;  // token warp (owns TPW tokens); others only help the core
    const int g = lane >> 2, t = lane & 3;
    unsigned char* gb = smem_raw + (size_t)grp * Lay::GROUP_BYTES;
    unsigned char* wb = smem_raw + (size_t)GROUPS * Lay::GROUP_BYTES +
                        (size_t)(grp * WPU + (r < WPU ? r : WPU - 1)) * Lay::WARP_BYTES;
    const int td = TPW * d;  // elements per staged tensor
    T* Qs = reinterpret_cast<T*>(wb);
    T* Ks = Qs + td;
    T* Vs = Qs + 2 * td;
    uint32_t* glf = reinterpret_cast<uint32_t*>(wb + Lay::GLF);
    float* wpart = reinterpret_cast<float*>(wb + Lay::WPART);
    T* qbar = reinterpret_cast<T*>(gb + Lay::G_QBAR);
    T* kbar = reinterpret_cast<T*>(gb + Lay::G_KBAR);
    float* gmu = reinterpret_cast<float*>(gb + Lay::G_MU);
    float* mW = reinterpret_cast<float*>(gb + Lay::G_W);
    T* yT = reinterpret_cast<T*>(gb + Lay::G_YT);
    uint64_t* barQK = reinterpret_cast<uint64_t*>(gb + Lay::G_BAR) + 2 * r;  // Q and K rows
    uint64_t* barV = barQK + 1;                                                // V rows

    auto gsync = [&]() {
        if constexpr (GW == 1) __syncwarp();
        else named_barrier(1 + grp, GW * 32);
    };
    // group barrier that also tells every warp whether any warp's wait gave up
    auto gsync_or = [&](bool f) -> bool {
        if constexpr (GW == 1) {
            __syncwarp();
            return f;
        } else {
            return named_barrier_or(1 + grp, GW * 32, f);
        }
    };
    // distributed-core scratch
    unsigned char* mat0 = nullptr;
    unsigned char* mat1 = nullptr;
    float* aux = nullptr;
    if constexpr (CW > 1) {
        using DSc = DistScratch<(M > 16 ? M : 32)>;
        if constexpr (Lay::SCR_IN_STAGE) {
            unsigned char* w0 = smem_raw + (size_t)GROUPS * Lay::GROUP_BYTES + (size_t)(grp * WPU) * Lay::WARP_BYTES;
            mat0 = w0 + Lay::WPART;
            aux = reinterpret_cast<float*>(mat0 + DSc::MAT);
            mat1 = w0 + Lay::WARP_BYTES + Lay::WPART;
        } else {
            mat0 = gb + Lay::G_SCR;
            mat1 = mat0 + DSc::MAT;
            aux = reinterpret_cast<float*>(mat1 + DSc::MAT);
        }
    }

    // Only the first `active` groups of a CTA take units (see launch_cfg).
    const long long stride = (long long)gridDim.x * active;
    long long u = grp < active ? (long long)blockIdx.x * active + grp : n_units;
    const uint32_t tile_bytes = (uint32_t)(td * sizeof(T));
    // This warp's rows of a unit are contiguous in HBM: one bulk copy per tensor.
    auto unit_off = [&](long long unit) { return (size_t)unit * N * d + (size_t)r * td; };
    auto arm_qk = [&]() { mbar_arrive_expect_tx(barQK, 2u * tile_bytes); };
    auto issue_q = [&](long long unit) { bulk_g2s(Qs, q + unit_off(unit), tile_bytes, barQK); };
    auto issue_k = [&](long long unit) { bulk_g2s(Ks, k + unit_off(unit), tile_bytes, barQK); };
    auto issue_v = [&](long long unit) {
        mbar_arrive_expect_tx(barV, tile_bytes);
        bulk_g2s(Vs, v + unit_off(unit), tile_bytes, barV);
    };

    if (tok && lane == 0) {
        mbar_init(barQK, 1);
        mbar_init(barV, 1);
        fence_mbar_init();
    }
    gsync();
    if (tok && u < n_units && lane == 0) {
        arm_qk();
        issue_q(u);
        issue_k(u);
        issue_v(u);
    }
    uint32_t phase_qk = 0, phase_v = 0;
    bool pend_qk = tok && u < n_units, pend_v = pend_qk;  // copies issued and not yet seen complete
    bool failed = false;  // a bounded wait of this warp gave up (warp-uniform)

    for (; u < n_units; u += stride) {
        // ---------------- stage: bounded wait for Q and K ----------------
        if (tok && !failed) {
            if (__all_sync(0xffffffffu, mbar_wait_bounded(barQK, phase_qk, kWaitNs))) {
                phase_qk ^= 1u;
                pend_qk = false;
            } else {
                failed = true;  // the whole group stops at the next barrier
                if (lane == 0) atomicOr(fault, 1u);
            }
        }

        // ---------------- front: landmarks (Algorithm 1 step 1) ----------------
        if (tok) {
            landmarks_mma<T, TPW, L>(Qs, qbar, r * LPW, d, g, t);
            landmarks_mma<T, TPW, L>(Ks, kbar, r * LPW, d, g, t);
            if (M < MP && r == 0) {  // zero the padding landmark rows
                landmarks_zero<T>(qbar, M, MP, lane, 32);
                landmarks_zero<T>(kbar, M, MP, lane, 32);
            }
        }
        if (gsync_or(failed)) break;

        // ---------------- front [P1]: S_L, G_L^n fragments ----------------
        if (GLS && tok) {
#pragma unroll 1
            for (int ch = 0; ch < NCH; ++ch)
#pragma unroll
                for (int tm = 0; tm < 4; ++tm) {
                    typename Opnd<T>::DReg f[KTL][4];
                    gl_tile<T, M, KTL>(Qs + (ch * 64 + 16 * tm + g) * d, kbar, d, g, t, sl2, f);
#pragma unroll
                    for (int kk = 0; kk < KTL; ++kk)
                        GlPark<T, M>::put(glf, ((ch * 4 + tm) * KTL + kk) * 32 + lane, f[kk]);
                }
        }

        // ---------------- stage: bounded wait for V ----------------
        if (tok && !failed) {
            if (__all_sync(0xffffffffu, mbar_wait_bounded(barV, phase_v, kWaitNs))) {
                phase_v ^= 1u;
                pend_v = false;
            } else {
                failed = true;
                if (lane == 0) atomicOr(fault, 1u);
            }
        }
        if (GW == 1 && failed) break;

        // ------- front: S_U, running m_U, G_U^n, W_r = G_U^n [V | 1] -------
        float mU[MT][2];  // this warp's row maxima of S_U, log2 domain
        if (tok) {
            front_su_w<T, M, NCOL, NCH>(qbar, Ks, Vs, d, g, t, sl2, WPU == 1 ? mW : wpart, WS, mU);
            if ((WPU > 1 || CW > 1) && t == 0) {
                float* mdst = WPU > 1 ? wpart + MP * WS : gmu;
#pragma unroll
                for (int mt = 0; mt < MT; ++mt) {
                    mdst[16 * mt + g] = mU[mt][0];
                    mdst[16 * mt + g + 8] = mU[mt][1];
                }
            }
        }

        // ---------------- combine (WPU > 1) ----------------
        if constexpr (WPU > 1) {
            gsync();
            if (tok)
                combine_partials<MP, NCOL, WS, WPU>(
                    reinterpret_cast<const float*>(smem_raw + (size_t)GROUPS * Lay::GROUP_BYTES +
                                                   (size_t)(grp * WPU) * Lay::WARP_BYTES + Lay::WPART),
                    Lay::WARP_BYTES / 4, mW, gmu, r, lane);
        }
        if (gsync_or(failed)) break;

        // Q and K of this unit are consumed (in P2 Q stays for the output):
        // prefetch the next unit's rows.  V's region holds the output first.
        // With the core's scratch in the K/V rows, K waits for the core.
        const long long un = u + stride;
        auto prefetch_qk = [&]() {
            fence_proxy_async_smem();  // this lane's reads of Q/K precede the async refill
            __syncwarp();
            if (tok && un < n_units && !failed) {
                if (lane == 0) {
                    arm_qk();
                    if constexpr (GLS) issue_q(un);
                    issue_k(un);
                }
                pend_qk = true;
            }
        };
        if constexpr (!Lay::SCR_IN_STAGE) prefetch_qk();

        // ---------------- core: G_A^n, Z_0, iteration, Y ----------------
        if constexpr (CW == 1) {
            if (r == 0) {
                if constexpr (WPU > 1) {
#pragma unroll
                    for (int mt = 0; mt < MT; ++mt) {
                        mU[mt][0] = gmu[16 * mt + g];
                        mU[mt][1] = gmu[16 * mt + g + 8];
                    }
                }
                core_warp<T, M, NCOL>(qbar, kbar, mU, mW, yT, iters, sl2, g, t);
            }
        } else {
            if (r < CW)
                dist_core<T, (M > 16 ? M : 32), NCOL>(qbar, kbar, gmu, mW, yT, mat0, mat1, aux, iters, sl2, r, lane,
                                                      1 + GROUPS + grp);
        }
        gsync();
        if constexpr (Lay::SCR_IN_STAGE) prefetch_qk();

        if (tok) {
            // ---------------- output: O = (G_L^n Y_:d) / (G_L^n Y_d) ----------------
            output_rows<T, M, NCOL, NCH, GLS>(glf, Qs, kbar, yT, Vs, d, g, t, lane, sl2);

            // The output rows are staged in V's region: one bulk store, and once it
            // has read shared memory, the next unit's V can land there.
            fence_proxy_async_smem();  // this lane's staging writes precede the bulk store
            __syncwarp();
            if (lane == 0) {
                bulk_s2g(out + unit_off(u), Vs, tile_bytes);
                bulk_commit();
                bulk_wait_read_all();
            }
        }
        // [P2] Q was needed until now: every warp of the group is done reading
        // the landmarks before anyone overwrites them.
        if constexpr (!GLS) {
            fence_proxy_async_smem();  // reads of Q precede its refill
            gsync();
        }
        if (tok && un < n_units && !failed) {
            if (lane == 0) {
                if constexpr (!GLS) issue_q(un);
                issue_v(un);
            }
            pend_v = true;
        }
        __syncwarp();
    }
    if (tok && lane == 0) bulk_wait_all();  // outstanding output stores complete before exit
    // Fault path only: copies still in flight land before the CTA's memory is released.
    if (tok && pend_qk) (void)__all_sync(0xffffffffu, mbar_wait_bounded(barQK, phase_qk, kWaitNs));
    if (tok && pend_v) (void)__all_sync(0xffffffffu, mbar_wait_bounded(barV, phase_v, kWaitNs));
}

// Largest number of groups per CTA that fits the shared-memory and register
// budgets (M <= 16 needs about 160 registers per thread, M = 32 about 255).
template <typename T, int M, int NCOL, int TPW, int WPU, bool GLS, int CW>
constexpr int groups_that_fit() {
    using Lay = Layout<T, M, NCOL, TPW, WPU, GLS, CW>;
    const int by_smem = (int)(kSmemLimit / Lay::PER_GROUP);
    const int by_regs = ((M <= 16) ? 12 : 8) / Lay::GW;
    const int n = by_smem < by_regs ? by_smem : by_regs;
    const int cap = (CW > 1) ? 7 : 15;  // named barriers: 1 + group barriers + core barriers <= 16
    return n > cap ? cap : n;
}

template <typename T, int M, int NCOL, int TPW, int WPU, int CW = 1>
cudaError_t launch_cfg(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                       int iters, cudaStream_t stream, unsigned int* fault) {
    // G_L^n parked (P1) unless recomputing it (P2) fits more groups.
    constexpr int kG1 = groups_that_fit<T, M, NCOL, TPW, WPU, true, CW>();
    constexpr int kG2 = groups_that_fit<T, M, NCOL, TPW, WPU, false, CW>();
    constexpr bool kGls = kG1 >= 1 && kG1 >= kG2;
    constexpr int kGroups = kGls ? kG1 : kG2;
    static_assert(kGroups >= 1, "configuration does not fit on one SM");
    using Lay = Layout<T, M, NCOL, TPW, WPU, kGls, CW>;
    auto kern = nystra_tc_kernel<T, M, NCOL, TPW, WPU, kGroups, kGls, CW>;
    const size_t smem = (size_t)kGroups * Lay::PER_GROUP;
    static std::atomic<int> s_blocks[kMaxDevices];  // persistent grid size per device
    int blocks = 0;
    if (cudaError_t e = persistent_grid(kern, kGroups * Lay::GW * 32, smem, s_blocks, &blocks); e != cudaSuccess)
        return e;
    // Wave quantisation: every group processes ceil(units / groups) units, so
    // use the fewest groups per CTA that still reach the minimal number of
    // rounds (fewer co-resident groups contend less for the SM).
    const long long rounds = (n_units + blocks * kGroups - 1) / (blocks * kGroups);
    int active = (int)((n_units + blocks * rounds - 1) / (blocks * rounds));
    active = active < 1 ? 1 : (active > kGroups ? kGroups : active);
    const long long want = (n_units + active - 1) / active;
    const long long grid = want < blocks ? want : blocks;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<(unsigned)grid, kGroups * Lay::GW * 32, smem, stream>>>((const T*)q, (const T*)k, (const T*)v,
                                                                  (T*)out, n_units, d, iters, sl2, fault, active);
    return cudaGetLastError();
}

// Stage-pool kernel for 8x8 windows (nystra_pool.cuh, N = 64 translation unit
// only).  PW: 0 = segment landmarks, else square patches of a PW-wide window.
template <typename T, int M, int NCOL, int PW = 0>
cudaError_t launch_pool(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                        int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias = nullptr);

// Team kernel for 16x16 windows (nystra_team.cuh, N = 256 translation unit only).
template <typename T, int M, int NCOL, int PW = 0>
cudaError_t launch_team(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                        int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias = nullptr);

// fp32 I/O: 8x8 windows with m <= 16 only (the stage-pool kernel).
template <int TPW, int WPU>
cudaError_t launch_f32(const void* q, const void* k, const void* v, void* out, long long n_units, int d, int m,
                       int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias = nullptr) {
    if constexpr (TPW == 64 && WPU == 1) {
        const bool wide = d > 30;
        if (m == 8)
            return wide ? launch_pool<float, 8, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_pool<float, 8, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
        if (m == 16)
            return wide ? launch_pool<float, 16, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_pool<float, 16, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
    }
    return cudaErrorInvalidValue;
}

// fp32 I/O only in the translation units that take it (F32).
template <bool F32, int TPW, int WPU>
cudaError_t launch_f32_if(const void* q, const void* k, const void* v, void* out, long long n_units, int d, int m,
                          int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias) {
    if constexpr (F32)
        return launch_f32<TPW, WPU>(q, k, v, out, n_units, d, m, iters, stream, fault, bias);
    else
        return cudaErrorInvalidValue;  // not reached: the caller routes fp32 I/O elsewhere
}

// Streaming team kernel for 32x32 windows (nystra_stream.cuh, N = 1024 translation unit only).
template <typename T, int M, int NCOL, int PW = 0>
cudaError_t launch_stream(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                          int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias = nullptr);

// Dispatch on m and the output-column padding for one window size.
// bias (m <= 16 only: the one-warp core) selects the kernels with a score bias.
template <typename T, int TPW, int WPU>
cudaError_t launch_n(const void* q, const void* k, const void* v, void* out, long long n_units, int d, int m,
                     int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias = nullptr) {
    const bool wide = d > 30;  // the ones column needs a fifth n-tile when d_h = 32
    if (bias && m > 16) return cudaErrorInvalidValue;  // not reached: the caller sends these to the SIMT path
    if constexpr (TPW == 64 && WPU == 1) {
        if (m == 8)
            return wide ? launch_pool<T, 8, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_pool<T, 8, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
        if (m == 16)
            return wide ? launch_pool<T, 16, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_pool<T, 16, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
    }
    if constexpr (TPW == 64 && WPU == 4) {
        if (m == 8)
            return wide ? launch_team<T, 8, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_team<T, 8, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
        if (m == 16)
            return wide ? launch_team<T, 16, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_team<T, 16, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
        // m = 32 with d_h <= 30 fits two teams per SM; d_h = 32 only one, so it
        // stays on the grouped kernel
        if (m == 32 && !wide) return launch_team<T, 32, 32>(q, k, v, out, n_units, d, iters, stream, fault);
    }
    if constexpr (TPW == 128 && WPU == 8) {
        if (m == 8)
            return wide ? launch_stream<T, 8, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_stream<T, 8, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
        if (m == 16)
            return wide ? launch_stream<T, 16, 40>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                        : launch_stream<T, 16, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
        if (m == 32)
            return wide ? launch_stream<T, 32, 40>(q, k, v, out, n_units, d, iters, stream, fault)
                        : launch_stream<T, 32, 32>(q, k, v, out, n_units, d, iters, stream, fault);
    }
    // The grouped kernel: m = 32 at 8x8 windows (core in one warp's registers)
    // and at 16x16 windows with d_h = 32 (core on two warps); every m = 64.
    if (m == 32) {
        if constexpr (TPW == 64 && WPU == 1)
            return wide ? launch_cfg<T, 32, 40, 64, 1, 1>(q, k, v, out, n_units, d, iters, stream, fault)
                        : launch_cfg<T, 32, 32, 64, 1, 1>(q, k, v, out, n_units, d, iters, stream, fault);
        if constexpr (TPW == 64 && WPU == 4)
            return launch_cfg<T, 32, 40, 64, 4, 2>(q, k, v, out, n_units, d, iters, stream, fault);
        return cudaErrorInvalidValue;  // not reached: the stream kernel takes 32x32 windows
    }
    if (m == 64) {
        // the core on four warps; W partials of 64 rows need K/V rows of at
        // least 128 tokens per token warp
        constexpr int TP = (TPW * WPU == 64) ? 64 : (TPW * WPU == 256) ? 128 : 256;
        constexpr int WP = TPW * WPU / TP;
        return wide ? launch_cfg<T, 64, 40, TP, WP, 4>(q, k, v, out, n_units, d, iters, stream, fault)
                    : launch_cfg<T, 64, 32, TP, WP, 4>(q, k, v, out, n_units, d, iters, stream, fault);
    }
    return cudaErrorInvalidValue;  // not reached: m is checked by the caller
}

// Square-patch landmarks on the tensor cores: 16-bit I/O, m = 16 (4 x 4
// patches of 2x2, 4x4 or 8x8 tokens), one window size per translation unit.
template <typename T, int TPW, int WPU>
cudaError_t launch_patches(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                           int m, int iters, cudaStream_t stream, unsigned int* fault,
                           const NystraBias* bias = nullptr) {
    const bool wide = d > 30;
    if (m != 16) return cudaErrorInvalidValue;  // not reached: checked by the caller
    if constexpr (TPW == 64 && WPU == 1)
        return wide ? launch_pool<T, 16, 40, 8>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                    : launch_pool<T, 16, 32, 8>(q, k, v, out, n_units, d, iters, stream, fault, bias);
    if constexpr (TPW == 64 && WPU == 4)
        return wide ? launch_team<T, 16, 40, 16>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                    : launch_team<T, 16, 32, 16>(q, k, v, out, n_units, d, iters, stream, fault, bias);
    if constexpr (TPW == 128 && WPU == 8)
        return wide ? launch_stream<T, 16, 40, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias)
                    : launch_stream<T, 16, 32, 32>(q, k, v, out, n_units, d, iters, stream, fault, bias);
    return cudaErrorInvalidValue;
}

}  // namespace tc
}  // namespace nystra

// One translation unit per window size and factor precision defines its fault
// word and entry points: BF and HF are the kernels' element types for bf16 and
// fp16 I/O (the plain types carry the derived factors as hi + lo pairs,
// Single16<...> rounds them to 16 bits); F32 says whether this unit also
// takes fp32 I/O (the 8x8 stage-pool kernel).
#define NYSTRA_TC_DEFINE(NAME, TPW, WPU, BF, HF, F32)                                                        \
    namespace nystra {                                                                                       \
    __device__ unsigned int g_fault_tc_##NAME;                                                               \
    }                                                                                                        \
    namespace nystra_host {                                                                                  \
    cudaError_t launch_nystra_tc_##NAME(const void* q, const void* k, const void* v, void* out,              \
                                        long long n_units, int d, int m, int iters, int pool, int dtype,     \
                                        cudaStream_t stream, const nystra::NystraBias* bias) {               \
        static unsigned int* s_fault[64] = {};  /* device address of the fault word, per device */      \
        int dev = 0;                                                                                         \
        cudaError_t e = cudaGetDevice(&dev);                                                                 \
        if (e != cudaSuccess) return e;                                                                      \
        if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;                                             \
        if (!s_fault[dev]) {                                                                                 \
            e = cudaGetSymbolAddress((void**)&s_fault[dev], nystra::g_fault_tc_##NAME);                      \
            if (e != cudaSuccess) return e;                                                                  \
        }                                                                                                    \
        unsigned int* fault = s_fault[dev];                                                                  \
        if (pool != 0) {                                                                                     \
            if (dtype == 1)                                                                                  \
                return nystra::tc::launch_patches<BF, TPW, WPU>(q, k, v, out, n_units, d, m, iters, stream,  \
                                                                fault, bias);                                \
            if (dtype == 2)                                                                                  \
                return nystra::tc::launch_patches<HF, TPW, WPU>(q, k, v, out, n_units, d, m, iters, stream,  \
                                                                fault, bias);                                \
            return cudaErrorInvalidValue; /* not reached: fp32 patches take the SIMT path */                 \
        }                                                                                                    \
        if (dtype == 0)                                                                                      \
            return nystra::tc::launch_f32_if<F32, TPW, WPU>(q, k, v, out, n_units, d, m, iters, stream, fault, \
                                                            bias);                                           \
        if (dtype == 1)                                                                                      \
            return nystra::tc::launch_n<BF, TPW, WPU>(q, k, v, out, n_units, d, m, iters, stream, fault, bias); \
        return nystra::tc::launch_n<HF, TPW, WPU>(q, k, v, out, n_units, d, m, iters, stream, fault, bias);  \
    }                                                                                                        \
    unsigned int take_fault_word_tc_##NAME(cudaError_t* err) {                                               \
        unsigned int w = 0, zero = 0;                                                                        \
        *err = cudaMemcpyFromSymbol(&w, nystra::g_fault_tc_##NAME, sizeof(w));                               \
        if (*err == cudaSuccess && w != 0)                                                                   \
            *err = cudaMemcpyToSymbol(nystra::g_fault_tc_##NAME, &zero, sizeof(zero));                       \
        return w;                                                                                            \
    }                                                                                                        \
    }
