// Fused Q/K/V projection + PnP-Nystra for 16x16 and 32x32 windows (N = 256
// or 1024 tokens), m <= 16 (and m = 32 at 32x32 windows), even d_h <= 32,
// 16-bit I/O.  The projections of Eq. (1) (Q = X W_Q, K = X W_K, V = X W_V
// per head, plus the optional projection bias) are computed on the tensor
// cores chunk by chunk and handed straight to the streaming kernel's phases
// (nystra_stream.cuh), so Q, K and V never reach HBM.
//
// The structure is the streaming kernel's: a team of four token warps (N / 4
// tokens each) and a core warp per (window, head) unit, per-unit state
// double-buffered, each token warp walking the same chunk tasks (Q(k), KV(k),
// OUT(k - 1): landmark sums, S_U and partial W, output) over 64-token chunks.
// Where the streaming kernel bulk-copies a chunk of Q, K or V into the token
// warp's slot, this one projects it there: A fragments are the window's
// token rows, read from global memory two k-steps ahead of their MMAs, the B
// fragments the head's weights staged in shared memory once per CTA
// (head-stationary CTAs, as in nystra_qkv.cuh: the CTAs serving one window's
// heads run side by side, so its tokens come from L2 after the first).  The
// output pass projects its chunk of Q once more instead of re-reading it.
// The token warp makes its own chunks, so there is no copy ring: one slot
// per token warp, its only waits the bounded hand-offs with the core warp.
#pragma once

#include "nystra_qkv.cuh"

namespace nystra {
namespace tc {

// Projection of one 64-token chunk of a window into NB of the three blocks:
// for b < NB, dst[b] (64 x d, row stride d) = X W_mat[b] of head h (+ bias),
// rounded to T.  xr: the chunk's first token row (C contiguous values per
// token) in global memory; wf: the head's staged weight fragments
// (stage_weights).  Passes of 16 RM tokens (RM m-tiles: the accumulators of
// NB blocks x RM m-tiles stay within the registers the warp's other state
// leaves), A fragments two k-steps ahead of their MMAs.
template <typename T, int NB, int RM>
__device__ __forceinline__ void project_chunk(const T* __restrict__ xr, const uint2* wf,
                                              const float* __restrict__ bqkv, int C, int h, int d, int ks,
                                              const int (&mat)[NB], T* const (&dst)[NB], int g, int t, int lane) {
    using Op = Mma16<T>;
#pragma unroll 1
    for (int pass = 0; pass < 4 / RM; ++pass) {
        float acc[NB][4][RM][4];
#pragma unroll
        for (int b = 0; b < NB; ++b)
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
#pragma unroll
                for (int mt = 0; mt < RM; ++mt)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[b][nt][mt][e] = 0.f;
        // lane's token rows 16 (RM pass + mt) + g (+8), inputs 2t (+1) and 2t + 8 (+1) of each k-step
        const T* r0 = xr + (size_t)(16 * RM * pass + g) * C + 2 * t;
        auto lda = [&](int kk, uint32_t (&a)[RM][4]) {
            const int k = 16 * kk;
            const bool v0 = k + 2 * t < C, v1 = k + 8 + 2 * t < C;  // C even: pairs are whole
#pragma unroll
            for (int mt = 0; mt < RM; ++mt) {
                const T* p = r0 + (size_t)(16 * mt) * C + k;
                a[mt][0] = v0 ? ldg_u32(p) : 0u;
                a[mt][1] = v0 ? ldg_u32(p + 8 * C) : 0u;
                a[mt][2] = v1 ? ldg_u32(p + 8) : 0u;
                a[mt][3] = v1 ? ldg_u32(p + 8 * C + 8) : 0u;
            }
        };
        auto mma_step = [&](int kk, const uint32_t (&a)[RM][4]) {
            const uint2* wk = wf + (size_t)kk * (3 * 4 * 32) + lane;
#pragma unroll
            for (int b = 0; b < NB; ++b)
#pragma unroll
                for (int nt = 0; nt < 4; ++nt) {
                    const uint2 w = wk[(mat[b] * 4 + nt) * 32];
#pragma unroll
                    for (int mt = 0; mt < RM; ++mt) Op::k16(acc[b][nt][mt], a[mt], w.x, w.y);
                }
        };
        // k-steps at or beyond ks load nothing (v0 = v1 = false)
        uint32_t a0[RM][4], a1[RM][4];
        lda(0, a0);
        lda(1, a1);
#pragma unroll 1
        for (int kk = 0; kk < ks; kk += 2) {
            mma_step(kk, a0);
            lda(kk + 2, a0);
            if (kk + 1 < ks) mma_step(kk + 1, a1);
            lda(kk + 3, a1);
        }
        // + bias, rounded to the I/O type
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            const float* bm = bqkv ? bqkv + mat[b] * C + h * d : nullptr;
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
                const int col = 8 * nt + 2 * t;
                if (col < d) {
                    const float b0 = bm ? __ldg(bm + col) : 0.f, b1 = bm ? __ldg(bm + col + 1) : 0.f;
#pragma unroll
                    for (int mt = 0; mt < RM; ++mt) {
                        const int row = 16 * (RM * pass + mt) + g;
                        const float* c = acc[b][nt][mt];
                        *reinterpret_cast<uint32_t*>(dst[b] + row * d + col) = Op::pack(c[0] + b0, c[1] + b1);
                        *reinterpret_cast<uint32_t*>(dst[b] + (row + 8) * d + col) = Op::pack(c[2] + b0, c[3] + b1);
                    }
                }
            }
        }
    }
}

template <typename T, int M, int NCOL, int TPW>
struct QsLayout {
    static constexpr int NT = 4, N = NT * TPW, CH = 64, NCHK = TPW / CH;  // token warps, chunks per warp
    static constexpr int CWN = M > 16 ? M / 16 : 1;  // core warps (m = 32: distributed core)
    static constexpr int MT = (M + 15) / 16, MP = MT * 16, WS = NCOL + 4;
    static constexpr int DS = (NCOL == 32) ? 30 : 32;
    static constexpr int L = N / M, LPW = TPW / L;  // tokens per segment, segments per token warp
    static constexpr size_t XB = (size_t)CH * DS * 2;  // one tensor's chunk
    static constexpr size_t SLOT = 2 * XB;             // K and V (Q uses the first half)
    static constexpr size_t WPB = (size_t)MP * WS * 4 + MP * 4;  // W partial, row maxima
    static_assert(WPB <= SLOT, "the W partial lives in the slot of the last K/V chunk");
    // per-unit state, as in StreamLayout (Y^T over Qbar, W and m_U)
    static constexpr size_t B_QB = 0;
    static constexpr size_t B_W = B_QB + LmS<T>::bytes(MP);
    static constexpr size_t B_MU = B_W + MP * WS * 4;
    static constexpr size_t B_KB = ((B_MU + MP * 4 + 15) / 16) * 16;
    static constexpr size_t B_YT = B_QB;
    static constexpr size_t BUF = ((B_KB + LmS<T>::bytes(MP) + 127) / 128) * 128;
    static_assert(YtS<T, M>::bytes(NCOL) <= B_KB, "Y^T must fit over Qbar, W and m_U");
    static constexpr size_t SCR = CWN > 1 ? DistScratch<(M > 16 ? M : 32)>::BYTES : 0;
    static constexpr size_t T_BUF = NT * SLOT;
    static constexpr size_t T_BAR = T_BUF + 2 * BUF;  // F[2], C[2]
    static constexpr size_t T_SCR = ((T_BAR + 4 * 8 + 127) / 128) * 128;
    static constexpr size_t TEAM = ((T_SCR + SCR + 127) / 128) * 128;
    static constexpr int WARPS = NT + CWN;  // per team
    // weights: 3 blocks x 4 n-tiles x 32 lanes x 8 bytes per k-step of 16 inputs
    static constexpr size_t FRAG = 3 * 4 * 32 * 8;
    static constexpr size_t HDR = 128;
    static constexpr size_t teams_at(int ks) { return (kSmemLimit - HDR - (size_t)ks * FRAG) / TEAM; }
    // teams per CTA: as many as fit beside the widest projection (C = 352), at most 3
    static constexpr int TEAMS = teams_at(22) < 3 ? (int)teams_at(22) : 3;
    static constexpr size_t bytes(int ks) { return HDR + (size_t)ks * FRAG + TEAMS * TEAM; }
    static_assert(TEAMS >= 1, "a team must fit beside the weights");
    static_assert(M <= 32 && L >= 16 && LPW <= 8 && TPW % CH == 0, "segments per token warp fit one n-tile");
    static_assert(XB % 16 == 0 && SLOT % 16 == 0 && BUF % 16 == 0 && FRAG % 128 == 0, "alignment");
};

// Block bi of a team's task sequence for `count` units: (unit, type), type
// 0 = Q, 1 = KV, 2 = OUT.  SHORT (the one-warp core, m <= 16): Q(0), KV(0),
// then Q(k), OUT(k - 1), KV(k) for k >= 1, finally OUT(count - 1).
// Otherwise Q(k), KV(k), OUT(k - 1), finally OUT(count - 1).  The streaming
// kernel's orders, one block of NCHK chunk tasks each.
template <bool SHORT>
__device__ __forceinline__ int2 qs_block(int bi, int count) {
    if constexpr (SHORT) {
        if (bi < 2) return make_int2(0, bi);
        const int k = (bi - 2) / 3 + 1, r = (bi - 2) % 3;
        if (k == count) return make_int2(count - 1, 2);
        return r == 0 ? make_int2(k, 0) : (r == 1 ? make_int2(k - 1, 2) : make_int2(k, 1));
    } else {
        const int vi = bi < 2 ? bi : (bi < 3 * count - 1 ? bi + 1 : bi + 3);
        const int k = vi / 3, r = vi % 3;
        return r < 2 ? make_int2(k, r) : make_int2(k - 1, 2);
    }
}

template <typename T, int M, int NCOL, int TPW, int PW, bool BIAS>
__global__ void __launch_bounds__(QsLayout<T, M, NCOL, TPW>::TEAMS * QsLayout<T, M, NCOL, TPW>::WARPS * 32, 1)
nystra_qkv_stream_kernel(const T* __restrict__ x, const T* __restrict__ wqkv, const float* __restrict__ bqkv,
                         T* __restrict__ out, long long n_windows, int heads, int d, int ks, int iters, float sl2,
                         unsigned int* fault, NystraBias bias) {
    static_assert(!BIAS || M <= 16, "a score bias runs with the one-warp core");
    using Lay = QsLayout<T, M, NCOL, TPW>;
    using R = typename Opnd<T>::DReg;
    constexpr int NT = Lay::NT, N = Lay::N, MP = Lay::MP, WS = Lay::WS, L = Lay::L, LPW = Lay::LPW,
                  NTO = NCOL / 8, MT = Lay::MT, NCHK = Lay::NCHK, TEAMS = Lay::TEAMS;
    constexpr bool SHORT = M <= 16;

    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int team = warp / Lay::WARPS, r = warp - team * Lay::WARPS;  // r >= NT: core warps
    const int g = lane >> 2, t = lane & 3;
    const int C = heads * d;
    const int h = (int)(blockIdx.x % heads);
    const long long Gh = gridDim.x / heads;  // CTAs serving head h
    uint2* wf = reinterpret_cast<uint2*>(smem_raw + Lay::HDR);
    unsigned char* tb = smem_raw + Lay::HDR + (size_t)ks * Lay::FRAG + (size_t)team * Lay::TEAM;
    auto buf = [&](int b) { return tb + Lay::T_BUF + (size_t)b * Lay::BUF; };
    uint64_t* barF = reinterpret_cast<uint64_t*>(tb + Lay::T_BAR);  // F[b]: the state for the core is ready
    uint64_t* barC = barF + 2;                                       // C[b]: the core's Y^T is ready

    // windows of this team: w0, w0 + stride, ...
    const long long stride = Gh * TEAMS;
    const long long w0 = (long long)(blockIdx.x / heads) * TEAMS + team;
    const int count = w0 < n_windows ? (int)((n_windows - w0 + stride - 1) / stride) : 0;
    auto unit_of = [&](int kk) { return (w0 + (long long)kk * stride) * heads + h; };
    auto bias_slice = [&](int kk) -> long long { return bias.per_window ? unit_of(kk) : h; };

    if (threadIdx.x == 0) {
        for (int tm = 0; tm < TEAMS; ++tm) {
            uint64_t* bb = reinterpret_cast<uint64_t*>(smem_raw + Lay::HDR + (size_t)ks * Lay::FRAG +
                                                       (size_t)tm * Lay::TEAM + Lay::T_BAR);
            mbar_init(bb, NT);
            mbar_init(bb + 1, NT);
            mbar_init(bb + 2, Lay::CWN);
            mbar_init(bb + 3, Lay::CWN);
        }
        fence_mbar_init();
    }
    // padding landmark rows (m < 16) stay zero: nothing else writes them
    if constexpr (M < MP) {
        for (int idx = threadIdx.x; idx < TEAMS * 2 * (MP - M) * 32; idx += blockDim.x) {
            const int tm = idx / (2 * (MP - M) * 32), rem = idx - tm * 2 * (MP - M) * 32;
            const int b = rem / ((MP - M) * 32), e = rem - b * (MP - M) * 32;
            unsigned char* bb = smem_raw + Lay::HDR + (size_t)ks * Lay::FRAG + (size_t)tm * Lay::TEAM + Lay::T_BUF +
                                (size_t)b * Lay::BUF;
            landmarks_zero<T>(reinterpret_cast<T*>(bb + Lay::B_QB), M + (e >> 5), M + (e >> 5) + 1, e & 31, 32);
            landmarks_zero<T>(reinterpret_cast<T*>(bb + Lay::B_KB), M + (e >> 5), M + (e >> 5) + 1, e & 31, 32);
        }
    }
    stage_weights<T>(wqkv, C, h, d, ks, wf);
    __syncthreads();

    if (r >= NT) {
        // ======================= core warp(s) =======================
        const int c = r - NT;
        for (int kk = 0; kk < count; ++kk) {
            const int b = kk & 1;
            bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(barF + b, (uint32_t)((kk >> 1) & 1), kWaitNs));
            if constexpr (Lay::CWN > 1)  // the core warps decide together
                ok = !named_barrier_or(1 + TEAMS + team, Lay::CWN * 32, !ok);
            if (!ok) {  // the token warps stopped (or stalled): stop too
                if (lane == 0) atomicOr(fault, 1u);
                break;
            }
            unsigned char* bb = buf(b);
            const float* gmu = reinterpret_cast<const float*>(bb + Lay::B_MU);
            if constexpr (Lay::CWN == 1) {
                float mU[1][2] = {{gmu[g], gmu[g + 8]}};
                const float* bAu = BIAS ? bias.A + (size_t)bias_slice(kk) * M * M : nullptr;
                core_warp<T, M, NCOL, false, BIAS>(reinterpret_cast<const T*>(bb + Lay::B_QB),
                                                   reinterpret_cast<const T*>(bb + Lay::B_KB), mU,
                                                   reinterpret_cast<const float*>(bb + Lay::B_W),
                                                   reinterpret_cast<T*>(bb + Lay::B_YT), iters, sl2, g, t, nullptr,
                                                   bAu);
            } else {
                using DSc = DistScratch<(M > 16 ? M : 32)>;
                unsigned char* scr = tb + Lay::T_SCR;
                dist_core<T, (M > 16 ? M : 32), NCOL>(
                    reinterpret_cast<const T*>(bb + Lay::B_QB), reinterpret_cast<const T*>(bb + Lay::B_KB), gmu,
                    reinterpret_cast<const float*>(bb + Lay::B_W), reinterpret_cast<T*>(bb + Lay::B_YT), scr,
                    scr + DSc::MAT, reinterpret_cast<float*>(scr + 2 * DSc::MAT), iters, sl2, c, lane,
                    1 + TEAMS + team);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(barC + b);
        }
        return;
    }

    // ======================= token warp r =======================
    T* X0 = reinterpret_cast<T*>(tb + (size_t)r * Lay::SLOT);  // Q, or K (then V at X1)
    T* X1 = reinterpret_cast<T*>(tb + (size_t)r * Lay::SLOT + Lay::XB);
    const uint32_t xbytes = (uint32_t)(Lay::CH * d * sizeof(T));
    auto tok0 = [&](int c) { return r * TPW + c * Lay::CH; };  // the chunk's first token in the window
    auto xrows = [&](int kk, int c) { return x + ((w0 + (long long)kk * stride) * N + tok0(c)) * (size_t)C; };
    auto tsync = [&]() { named_barrier(1 + team, NT * 32); };
    auto tsync_or = [&](bool f) { return named_barrier_or(1 + team, NT * 32, f); };

    bool failed = false;  // a bounded wait of this warp gave up (warp-uniform)
    float cq[2][1][4], ck[2][1][4], w[MT][NTO][4], run[MT][2];
    R aq[MT][2][4];
    const int total = 3 * count * NCHK;
    for (int vv = 0; vv < total; ++vv) {
        const int2 blk = qs_block<SHORT>(vv / NCHK, count);
        const int kk = blk.x, type = blk.y, c = vv % NCHK;
        const int b = kk & 1;
        unsigned char* bb = buf(b);
        const long long bsl = BIAS ? bias_slice(kk) : 0;
        if (type == 0) {
            // ---------------- Q(k): projection, landmark sums of Qbar ----------------
            {
                const int mat[1] = {0};
                T* const dst[1] = {X0};
                project_chunk<T, 1, 2>(xrows(kk, c), wf, bqkv, C, h, d, ks, mat, dst, g, t, lane);
            }
            __syncwarp();
            if (c == 0)
#pragma unroll
                for (int mf = 0; mf < 2; ++mf) cq[mf][0][0] = cq[mf][0][1] = cq[mf][0][2] = cq[mf][0][3] = 0.f;
            landmarks_acc<T, L, LPW, PW>(X0, c * Lay::CH, cq, d, g, t);
            if (c == NCHK - 1) {
                // Qbar overlays the Y^T of unit k - 2: with the long core's
                // task order (m = 32) a warp's OUT(k - 2) precedes this task
                // without a barrier in between, so wait for every warp's.
                if constexpr (!SHORT)
                    if (tsync_or(failed)) break;
                landmarks_put<T, LPW>(cq, reinterpret_cast<T*>(bb + Lay::B_QB), r * LPW, g, t);
                if (tsync_or(failed)) break;
                if constexpr (!SHORT)  // KV(k) follows directly
#pragma unroll
                    for (int mt = 0; mt < MT; ++mt)
                        qbar_afrag<T>(reinterpret_cast<const T*>(bb + Lay::B_QB), mt, g, t, aq[mt]);
            }
        } else if (type == 1) {
            // ---------------- KV(k): projections, Kbar sums, S_U, partial W ----------------
            {
                const int mat[2] = {1, 2};
                T* const dst[2] = {X0, X1};
                project_chunk<T, 2, 1>(xrows(kk, c), wf, bqkv, C, h, d, ks, mat, dst, g, t, lane);
            }
            __syncwarp();
            if (c == 0) {
                if constexpr (SHORT)  // OUT(k - 1) ran since Q(k): reload Qbar's operands
#pragma unroll
                    for (int mt = 0; mt < MT; ++mt)
                        qbar_afrag<T>(reinterpret_cast<const T*>(bb + Lay::B_QB), mt, g, t, aq[mt]);
#pragma unroll
                for (int mf = 0; mf < 2; ++mf) ck[mf][0][0] = ck[mf][0][1] = ck[mf][0][2] = ck[mf][0][3] = 0.f;
#pragma unroll
                for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
                    for (int j = 0; j < NTO; ++j) w[mt][j][0] = w[mt][j][1] = w[mt][j][2] = w[mt][j][3] = 0.f;
                    run[mt][0] = run[mt][1] = -INFINITY;
                }
            }
            landmarks_acc<T, L, LPW, PW>(X0, c * Lay::CH, ck, d, g, t);
#pragma unroll
            for (int mt = 0; mt < MT; ++mt)
                su_w_chunk<T, NCOL, BIAS>(aq[mt], X0, X1, d, g, t, sl2, 16 * mt + g < M, 16 * mt + g + 8 < M, w[mt],
                                          run[mt][0], run[mt][1], true,
                                          BIAS ? bias.U + (size_t)bsl * M * N + (size_t)(16 * mt + g) * N + tok0(c)
                                               : nullptr,
                                          N);
            if (c == NCHK - 1) {
                landmarks_put<T, LPW>(ck, reinterpret_cast<T*>(bb + Lay::B_KB), r * LPW, g, t);
                // the partial goes over this slot's K and V rows, consumed above
                float* wpart = reinterpret_cast<float*>(X0);
                __syncwarp();
#pragma unroll
                for (int mt = 0; mt < MT; ++mt)
#pragma unroll
                    for (int j = 0; j < NTO; ++j) {
                        const int cc = 8 * j + 2 * t, rr = 16 * mt + g;
                        *reinterpret_cast<float2*>(wpart + rr * WS + cc) = make_float2(w[mt][j][0], w[mt][j][1]);
                        *reinterpret_cast<float2*>(wpart + (rr + 8) * WS + cc) = make_float2(w[mt][j][2], w[mt][j][3]);
                    }
                if (t == 0) {
#pragma unroll
                    for (int mt = 0; mt < MT; ++mt) {
                        wpart[MP * WS + 16 * mt + g] = run[mt][0];
                        wpart[MP * WS + 16 * mt + g + 8] = run[mt][1];
                    }
                }
                tsync();
                combine_partials<MP, NCOL, WS, NT>(reinterpret_cast<const float*>(tb), Lay::SLOT / 4,
                                                    reinterpret_cast<float*>(bb + Lay::B_W),
                                                    reinterpret_cast<float*>(bb + Lay::B_MU), r, lane);
                if (tsync_or(failed)) break;
                __syncwarp();
                if (lane == 0) mbar_arrive(barF + b);
            }
        } else {
            // ---------------- OUT(k): Q projected again, output rows of this chunk ----------------
            if (c == 0 && !failed) {
                if (!__all_sync(0xffffffffu, mbar_wait_bounded(barC + b, (uint32_t)((kk >> 1) & 1), kWaitNs))) {
                    failed = true;
                    if (lane == 0) atomicOr(fault, 1u);
                }
            }
            if (!failed) {
                {
                    const int mat[1] = {0};
                    T* const dst[1] = {X0};
                    project_chunk<T, 1, 2>(xrows(kk, c), wf, bqkv, C, h, d, ks, mat, dst, g, t, lane);
                }
                __syncwarp();
                output_rows<T, M, NCOL, 1, false, BIAS>(
                    nullptr, X0, reinterpret_cast<const T*>(bb + Lay::B_KB), reinterpret_cast<const T*>(bb + Lay::B_YT),
                    X0, d, g, t, lane, sl2, BIAS ? bias.L + (size_t)bsl * N * M + (size_t)tok0(c) * M : nullptr);
                fence_proxy_async_smem();  // this lane's writes precede the bulk store
                __syncwarp();
                if (lane == 0) {
                    bulk_s2g(out + ((size_t)unit_of(kk) * N + tok0(c)) * d, X0, xbytes);
                    bulk_commit();
                    bulk_wait_read_all();  // the slot is rewritten by the next task
                }
                __syncwarp();
            }
        }
    }
    if (lane == 0) bulk_wait_all();  // output stores complete before exit
}

template <typename T, int M, int NCOL, int TPW, int PW, bool BIAS>
cudaError_t launch_qkv_stream_cfg(const void* x, const void* wqkv, const float* bqkv, void* out, long long n_windows,
                                  int heads, int d, int iters, cudaStream_t stream, unsigned int* fault,
                                  const NystraBias& bias) {
    using Lay = QsLayout<T, M, NCOL, TPW>;
    auto kern = nystra_qkv_stream_kernel<T, M, NCOL, TPW, PW, BIAS>;
    const int C = heads * d, ks = (C + 15) / 16;
    const size_t smem = Lay::bytes(ks);
    if (smem > kSmemLimit) return cudaErrorInvalidValue;  // not reached: the caller bounds C
    static std::atomic<int> s_blocks[kMaxDevices];  // persistent grid size per device
    int blocks = 0;
    if (cudaError_t e = persistent_grid(kern, Lay::TEAMS * Lay::WARPS * 32, Lay::bytes(22), s_blocks, &blocks);
        e != cudaSuccess)
        return e;
    // CTAs per head: enough to fill the device, no more than the head's windows need
    long long per_head = blocks / heads;
    if (per_head < 1) per_head = 1;
    const long long need = (n_windows + Lay::TEAMS - 1) / Lay::TEAMS;
    if (per_head > need) per_head = need;
    const long long grid = per_head * heads;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<(unsigned)grid, Lay::TEAMS * Lay::WARPS * 32, smem, stream>>>((const T*)x, (const T*)wqkv, bqkv, (T*)out,
                                                                         n_windows, heads, d, ks, iters, sl2, fault,
                                                                         bias);
    return cudaGetLastError();
}

// 16x16 (TPW = 64) and 32x32 (TPW = 256) windows: m in {8, 16} (also m = 32
// at 32x32 windows; square patches: m = 16); d_h read at run time.
template <typename T, int TPW>
cudaError_t launch_qkv_stream(const void* x, const void* wqkv, const float* bqkv, void* out, long long n_windows,
                              int heads, int d, int m, int iters, int pool, cudaStream_t stream, unsigned int* fault,
                              const NystraBias* bias) {
    const bool wide = d > 30;  // the ones column needs a fifth n-tile when d_h = 32
    const NystraBias b = bias ? *bias : NystraBias{};
    constexpr int PWQ = TPW == 64 ? 16 : 32;  // window width for square patches
    const bool bi = bias != nullptr;
#define NYSTRA_QS(M_, NC_, PW_, B_) \
    launch_qkv_stream_cfg<T, M_, NC_, TPW, PW_, B_>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream, fault, b)
    if (pool != 0) {
        if (m != 16) return cudaErrorInvalidValue;  // not reached: checked by the caller
        if (bi) return wide ? NYSTRA_QS(16, 40, PWQ, true) : NYSTRA_QS(16, 32, PWQ, true);
        return wide ? NYSTRA_QS(16, 40, PWQ, false) : NYSTRA_QS(16, 32, PWQ, false);
    }
    if (m == 8) {
        if (bi) return wide ? NYSTRA_QS(8, 40, 0, true) : NYSTRA_QS(8, 32, 0, true);
        return wide ? NYSTRA_QS(8, 40, 0, false) : NYSTRA_QS(8, 32, 0, false);
    }
    if (m == 16) {
        if (bi) return wide ? NYSTRA_QS(16, 40, 0, true) : NYSTRA_QS(16, 32, 0, true);
        return wide ? NYSTRA_QS(16, 40, 0, false) : NYSTRA_QS(16, 32, 0, false);
    }
    if constexpr (TPW == 256)
        if (m == 32 && !bi) return wide ? NYSTRA_QS(32, 40, 0, false) : NYSTRA_QS(32, 32, 0, false);
#undef NYSTRA_QS
    return cudaErrorInvalidValue;  // not reached: checked by the caller
}

}  // namespace tc
}  // namespace nystra

// One translation unit per element type defines its fault word and entry
// point: N = 256 or 1024.
#define NYSTRA_QKVS_DEFINE(NAME, T)                                                                         \
    namespace nystra {                                                                                      \
    __device__ unsigned int g_fault_qkvs_##NAME;                                                            \
    }                                                                                                       \
    namespace nystra_host {                                                                                 \
    cudaError_t launch_nystra_qkvs_##NAME(const void* x, const void* wqkv, const float* bqkv, void* out,    \
                                          long long n_windows, int heads, int N, int d, int m, int iters,   \
                                          int pool, cudaStream_t stream, const nystra::NystraBias* bias) {  \
        static unsigned int* s_fault[nystra::kMaxDevices] = {}; /* fault word's address, per device */     \
        int dev = 0;                                                                                        \
        cudaError_t e = cudaGetDevice(&dev);                                                                \
        if (e != cudaSuccess) return e;                                                                     \
        if (dev < 0 || dev >= nystra::kMaxDevices) return cudaErrorInvalidDevice;                          \
        if (!s_fault[dev]) {                                                                                \
            e = cudaGetSymbolAddress((void**)&s_fault[dev], nystra::g_fault_qkvs_##NAME);                   \
            if (e != cudaSuccess) return e;                                                                 \
        }                                                                                                   \
        if (N == 256)                                                                                       \
            return nystra::tc::launch_qkv_stream<T, 64>(x, wqkv, bqkv, out, n_windows, heads, d, m, iters,  \
                                                        pool, stream, s_fault[dev], bias);                  \
        if (N == 1024)                                                                                      \
            return nystra::tc::launch_qkv_stream<T, 256>(x, wqkv, bqkv, out, n_windows, heads, d, m, iters, \
                                                         pool, stream, s_fault[dev], bias);                 \
        return cudaErrorInvalidValue; /* not reached: checked by the caller */                              \
    }                                                                                                       \
    unsigned int take_fault_word_qkvs_##NAME(cudaError_t* err) {                                            \
        unsigned int w = 0, zero = 0;                                                                       \
        *err = cudaMemcpyFromSymbol(&w, nystra::g_fault_qkvs_##NAME, sizeof(w));                            \
        if (*err == cudaSuccess && w != 0)                                                                  \
            *err = cudaMemcpyToSymbol(nystra::g_fault_qkvs_##NAME, &zero, sizeof(zero));                    \
        return w;                                                                                           \
    }                                                                                                       \
    }
