// Team PnP-Nystra kernel for 16x16 windows (N = 256 tokens), m <= 32, even
// d_h <= 32, 16-bit I/O (m = 32: the core runs on two warps, dist_core).  Included by the N = 256 translation unit after
// nystra_tc.cuh, whose per-phase device functions it reuses.
//
// In the grouped kernel the m x m core runs on one warp of a unit's group
// while the group's other warps wait, so the core (a latency-bound chain of
// small products) is exposed once per unit.  Here a team is four token warps
// (64 tokens each, as in the grouped kernel) plus a dedicated core warp, and
// the per-unit state handed between them is double-buffered: while the core
// warp runs the iteration of unit k, the token warps run the front phase of
// unit k + 1 and then the output of unit k.
//
// Token warp r, unit k (buffer b = k mod 2):
//   wait Q, K rows -> landmarks -> [sync] -> wait V -> S_U, partial W_r ->
//   copy the Q rows of unit k - 1 again (into the V rows, now consumed) ->
//   [sync] -> combine into W, m_U -> [sync] -> signal the core (mbarrier
//   F_b) -> copy Q, K of unit k + 1 -> wait for the core of unit k - 1
//   (mbarrier C_{1-b}) and for its Q rows -> output of unit k - 1 (S_L and
//   G_L^n from those rows and Kbar, then O) written in place over them and
//   bulk-stored -> copy V of unit k + 1.
// Core warp, unit k: wait F_b -> G_A^n, iteration, Y^T into buffer b ->
//   signal C_b.
// G_L^n is recomputed in the output pass rather than parked: its hi + lo
// pairs would take 16 KB per unit, which costs a team per SM, while reading a
// unit's Q rows a second time (3.75 KB per token warp, usually from L2: they
// were read about one unit earlier) costs no shared memory.
// [sync] is a named barrier over the four token warps.  Every wait on an
// mbarrier is bounded; a warp whose wait gives up keeps to the barrier
// sequence, and the token warps leave the loop together after the next
// barrier, whose OR-reduction gives every warp the same verdict.
#pragma once

#include "nystra_tc.cuh"

namespace nystra {
namespace tc {

template <typename T, int M, int NCOL>
struct TeamLayout {
    static constexpr int NT = 4, TPW = 64, N = NT * TPW;  // token warps, tokens per token warp
    static constexpr int CWN = M > 16 ? M / 16 : 1;        // core warps (m = 32: distributed core)
    static constexpr int DS = (NCOL == 32) ? 30 : 32;
    static constexpr int MP = M > 16 ? M : 16, LS = LmS<T>::LS, WS = NCOL + 4;
    static constexpr int KTL = (M >= 16) ? M / 16 : 1;
    static constexpr size_t STAGE = 3 * (size_t)TPW * DS * 2;  // a token warp's Q, K, V rows
    static constexpr size_t WPART = (size_t)TPW * DS * 2;      // partial W_r after Q (K, V consumed)
    static_assert((size_t)MP * WS * 4 + MP * 4 <= 2 * (size_t)TPW * DS * 2, "W partial must fit in K+V");
    // one buffer of per-unit state
    static constexpr size_t B_QB = 0;
    static constexpr size_t B_KB = B_QB + LmS<T>::bytes(MP);
    static constexpr size_t B_W = B_KB + LmS<T>::bytes(MP);
    static constexpr size_t B_MU = B_W + MP * WS * 4;
    static constexpr size_t B_YT = ((B_MU + MP * 4 + 15) / 16) * 16;
    static constexpr size_t BUF = ((B_YT + YtS<T, M>::bytes(NCOL) + 127) / 128) * 128;
    // team memory: stages, two buffers, mbarriers
    static constexpr size_t T_BUF = NT * STAGE;
    static constexpr size_t T_BAR = T_BUF + 2 * BUF;  // barQK[4], barV[4], F[2], C[2]
    static constexpr size_t T_SCR = ((T_BAR + 12 * 8 + 127) / 128) * 128;  // distributed core's scratch
    static constexpr size_t TEAM =
        ((T_SCR + (CWN > 1 ? DistScratch<(M > 16 ? M : 32)>::BYTES : 0) + 127) / 128) * 128;
    static constexpr int TEAMS = (int)(kSmemLimit / TEAM) < 3 ? (int)(kSmemLimit / TEAM) : 3;
    static constexpr int WARPS = NT + CWN;  // per team
    static_assert(TEAMS >= 1, "team does not fit in shared memory");
    static_assert(STAGE % 16 == 0 && BUF % 16 == 0, "16-byte alignment");
};

template <typename T, int M, int NCOL, int DC, int PW, bool BIAS>
__global__ void __launch_bounds__(TeamLayout<T, M, NCOL>::TEAMS * TeamLayout<T, M, NCOL>::WARPS * 32, 1)
nystra_team_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                   T* __restrict__ out, long long n_units, int d_in, int iters, float sl2, unsigned int* fault,
                   NystraBias bias) {
    static_assert(!BIAS || M <= 16, "a score bias runs with the one-warp core");
    const int d = DC ? DC : d_in;  // d_h, a compile-time constant for the common head widths
    using Lay = TeamLayout<T, M, NCOL>;
    constexpr int NT = Lay::NT, TPW = Lay::TPW, N = Lay::N, MP = Lay::MP, WS = Lay::WS, NCOLC = NCOL;
    constexpr int L = N / M, LPW = TPW / L;
    constexpr int RS = row_step(DC);  // token order of the staged rows (bank-conflict-free fragment loads)
    static_assert(L <= TPW && TPW % L == 0, "segments must not straddle warps");

    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int team = warp / Lay::WARPS, r = warp - team * Lay::WARPS;  // r >= NT: core warps
    const int g = lane >> 2, t = lane & 3;
    unsigned char* tb = smem_raw + (size_t)team * Lay::TEAM;
    auto buf = [&](int b) { return tb + Lay::T_BUF + (size_t)b * Lay::BUF; };
    uint64_t* bars = reinterpret_cast<uint64_t*>(tb + Lay::T_BAR);
    uint64_t* barF = bars + 8;  // F[b]: the token warps' state for the core is ready
    uint64_t* barC = bars + 10; // C[b]: the core's Y^T is ready

    const long long stride = (long long)gridDim.x * Lay::TEAMS;
    const long long u0 = (long long)blockIdx.x * Lay::TEAMS + team;

    if (threadIdx.x == 0) {
        for (int tm = 0; tm < Lay::TEAMS; ++tm) {
            uint64_t* bb = reinterpret_cast<uint64_t*>(smem_raw + (size_t)tm * Lay::TEAM + Lay::T_BAR);
            for (int i = 0; i < 8; ++i) mbar_init(bb + i, 1);
            mbar_init(bb + 8, NT);
            mbar_init(bb + 9, NT);
            mbar_init(bb + 10, Lay::CWN);
            mbar_init(bb + 11, Lay::CWN);
        }
        fence_mbar_init();
    }
    // padding landmark rows (m < 16) stay zero: nothing else writes them
    if constexpr (M < MP) {
        for (int idx = threadIdx.x; idx < Lay::TEAMS * 2 * (MP - M) * 16; idx += blockDim.x) {
            const int tm = idx / (2 * (MP - M) * 16), rem = idx - tm * 2 * (MP - M) * 16;
            const int b = rem / ((MP - M) * 16), e = rem - b * (MP - M) * 16;
            unsigned char* bb = smem_raw + (size_t)tm * Lay::TEAM + Lay::T_BUF + (size_t)b * Lay::BUF;
            const int jr = M + (e >> 4), p = e & 15;
            landmarks_zero<T>(reinterpret_cast<T*>(bb + Lay::B_QB), jr, jr + 1, 2 * p, 64);
            landmarks_zero<T>(reinterpret_cast<T*>(bb + Lay::B_QB), jr, jr + 1, 2 * p + 1, 64);
            landmarks_zero<T>(reinterpret_cast<T*>(bb + Lay::B_KB), jr, jr + 1, 2 * p, 64);
            landmarks_zero<T>(reinterpret_cast<T*>(bb + Lay::B_KB), jr, jr + 1, 2 * p + 1, 64);
        }
    }
    __syncthreads();

    if (r >= NT) {
        // ======================= core warp(s) =======================
        const int c = r - NT;
        for (long long kk = 0;; ++kk) {
            const long long u = u0 + kk * stride;
            if (u >= n_units) break;
            const int b = (int)(kk & 1);
            const uint32_t par = (uint32_t)((kk >> 1) & 1);
            bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(barF + b, par, kWaitNs));
            if constexpr (Lay::CWN > 1)  // the core warps decide together
                ok = !named_barrier_or(1 + Lay::TEAMS + team, Lay::CWN * 32, !ok);
            if (!ok) {  // the token warps stopped (or stalled): stop too
                if (lane == 0) atomicOr(fault, 1u);
                break;
            }
            unsigned char* bb = buf(b);
            const float* gmu = reinterpret_cast<const float*>(bb + Lay::B_MU);
            if constexpr (Lay::CWN == 1) {
                float mU[1][2] = {{gmu[g], gmu[g + 8]}};
                const float* bAu =
                    BIAS ? bias.A + (size_t)(bias.per_window ? u : u % bias.heads) * M * M : nullptr;
                core_warp<T, M, NCOLC, false, BIAS>(reinterpret_cast<const T*>(bb + Lay::B_QB),
                                                    reinterpret_cast<const T*>(bb + Lay::B_KB), mU,
                                                    reinterpret_cast<const float*>(bb + Lay::B_W),
                                                    reinterpret_cast<T*>(bb + Lay::B_YT), iters, sl2, g, t,
                                                    nullptr, bAu);
            } else {
                using DSc = DistScratch<(M > 16 ? M : 32)>;
                unsigned char* scr = tb + Lay::T_SCR;
                dist_core<T, (M > 16 ? M : 32), NCOLC>(
                    reinterpret_cast<const T*>(bb + Lay::B_QB), reinterpret_cast<const T*>(bb + Lay::B_KB), gmu,
                    reinterpret_cast<const float*>(bb + Lay::B_W), reinterpret_cast<T*>(bb + Lay::B_YT), scr,
                    scr + DSc::MAT, reinterpret_cast<float*>(scr + 2 * DSc::MAT), iters, sl2, c, lane,
                    1 + Lay::TEAMS + team);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(barC + b);
        }
        return;
    }

    // ======================= token warp r =======================
    T* Qs = reinterpret_cast<T*>(tb + (size_t)r * Lay::STAGE);
    const int td = TPW * d;
    T* Ks = Qs + td;
    T* Vs = Qs + 2 * td;
    float* wpart = reinterpret_cast<float*>(tb + (size_t)r * Lay::STAGE + Lay::WPART);
    uint64_t* barQK = bars + r;
    uint64_t* barV = bars + 4 + r;  // V rows, and the Q rows read again for the output (alternately)
    const uint32_t tile_bytes = (uint32_t)(td * sizeof(T));
    auto unit_off = [&](long long unit) { return (size_t)unit * N * d + (size_t)r * td; };
    // L2 policies: the first read of Q is kept for its second read (the
    // output pass, about one unit later); every other read is its last.
    const uint64_t keep = l2_evict_last(), drop = l2_evict_first();
    auto issue_qk = [&](long long unit) {
        mbar_arrive_expect_tx(barQK, 2u * tile_bytes);
        bulk_g2s_hint(Qs, q + unit_off(unit), tile_bytes, barQK, keep);
        bulk_g2s_hint(Ks, k + unit_off(unit), tile_bytes, barQK, drop);
    };
    auto issue_v = [&](long long unit) {
        mbar_arrive_expect_tx(barV, tile_bytes);
        bulk_g2s_hint(Vs, v + unit_off(unit), tile_bytes, barV, drop);
    };
    auto issue_q_again = [&](long long unit) {  // the output pass's Q rows, into the V rows
        mbar_arrive_expect_tx(barV, tile_bytes);
        bulk_g2s_hint(Vs, q + unit_off(unit), tile_bytes, barV, drop);
    };
    auto tsync = [&]() { named_barrier(1 + team, NT * 32); };
    // barrier that also tells every token warp whether any of them failed
    auto tsync_or = [&](bool f) { return named_barrier_or(1 + team, NT * 32, f); };
    uint32_t phase_qk = 0, phase_v = 0;
    bool pend_qk = false, pend_v = false;  // copies issued and not yet seen complete
    bool failed = false;                   // a bounded wait of this warp gave up (warp-uniform)
    auto wait_v = [&]() {  // bounded wait for the copy on barV (V rows or Q rows again)
        if (failed) return;
        if (__all_sync(0xffffffffu, mbar_wait_bounded(barV, phase_v, kWaitNs))) {
            phase_v ^= 1u;
            pend_v = false;
        } else {
            failed = true;
            if (lane == 0) atomicOr(fault, 1u);
        }
    };

    // Output of unit kk (its core has run on buffer kk mod 2, its Q rows have
    // been copied again into the V rows): S_L, G_L^n and O tile by tile,
    // written in place over those Q rows; returns once the bulk store has
    // read them.
    auto output_unit = [&](long long kk) {
        const int b = (int)(kk & 1);
        if (failed) return;
        const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(barC + b, (uint32_t)((kk >> 1) & 1), kWaitNs));
        if (!ok) {
            failed = true;
            if (lane == 0) atomicOr(fault, 1u);
            return;
        }
        wait_v();
        if (failed) return;
        unsigned char* bb = buf(b);
        const long long uk = u0 + kk * stride;
        const float* bLu =
            BIAS ? bias.L + (size_t)(bias.per_window ? uk : uk % bias.heads) * N * M + (size_t)r * TPW * M : nullptr;
        output_rows<T, M, NCOLC, 1, false, BIAS, RS>(nullptr, Vs, reinterpret_cast<const T*>(bb + Lay::B_KB),
                                                 reinterpret_cast<const T*>(bb + Lay::B_YT), Vs, d, g, t, lane, sl2,
                                                 bLu);
        fence_proxy_async_smem();  // this lane's writes precede the bulk store
        __syncwarp();
        if (lane == 0) {
            // O is not read again: evict it first, keeping L2 for the Q rows read twice
            bulk_s2g_hint(out + unit_off(uk), Vs, tile_bytes, drop);
            bulk_commit();
            bulk_wait_read_all();
        }
        __syncwarp();
    };

    if (u0 < n_units && lane == 0) {
        issue_qk(u0);
        issue_v(u0);
    }
    pend_qk = pend_v = u0 < n_units;
    long long kk = 0;
    bool broke = false;  // the token warps left the loop together after a failed wait
    for (;; ++kk) {
        const long long u = u0 + kk * stride;
        if (u >= n_units) break;
        const long long bs = BIAS ? (bias.per_window ? u : u % bias.heads) : 0;
        const float* bUu = BIAS ? bias.U + (size_t)bs * M * N : nullptr;
        const int b = (int)(kk & 1);
        unsigned char* bb = buf(b);
        T* qbar = reinterpret_cast<T*>(bb + Lay::B_QB);
        T* kbar = reinterpret_cast<T*>(bb + Lay::B_KB);
        // ---------------- bounded wait for Q and K ----------------
        if (!failed) {
            const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(barQK, phase_qk, kWaitNs));
            if (ok) {
                phase_qk ^= 1u;
                pend_qk = false;
            } else {
                failed = true;
                if (lane == 0) atomicOr(fault, 1u);
            }
        }
        // ---------------- landmarks (Algorithm 1 step 1) ----------------
        // Buffer b's Kbar was last read by the output of unit kk - 2, which
        // every token warp ran in the previous iteration after that
        // iteration's last barrier: the sums go to registers first, and a
        // barrier separates those outputs from the stores.
        {
            constexpr int NTJ = (LPW + 7) / 8;
            float cq[2][NTJ][4], ck[2][NTJ][4];
#pragma unroll
            for (int mf = 0; mf < 2; ++mf)
#pragma unroll
                for (int j = 0; j < NTJ; ++j)
#pragma unroll
                    for (int e = 0; e < 4; ++e) cq[mf][j][e] = ck[mf][j][e] = 0.f;
            landmarks_acc<T, L, LPW, PW, RS>(Qs, 0, cq, d, g, t);
            landmarks_acc<T, L, LPW, PW, RS>(Ks, 0, ck, d, g, t);
            tsync();
            landmarks_put<T, LPW>(cq, qbar, r * LPW, g, t);
            landmarks_put<T, LPW>(ck, kbar, r * LPW, g, t);
        }
        if (tsync_or(failed)) {
            broke = true;
            break;
        }
        // ---------------- bounded wait for V ----------------
        wait_v();
        // ---------------- S_U, partial W_r and row maxima ----------------
        constexpr int MT = (M + 15) / 16;
        float mU[MT][2];
        front_su_w<T, M, NCOLC, 1, BIAS, RS>(qbar, Ks, Vs, d, g, t, sl2, wpart, WS, mU,
                                         BIAS ? bUu + r * TPW : nullptr, N);
        if (t == 0) {
#pragma unroll
            for (int mt = 0; mt < MT; ++mt) {
                wpart[MP * WS + 16 * mt + g] = mU[mt][0];
                wpart[MP * WS + 16 * mt + g + 8] = mU[mt][1];
            }
        }
        tsync();
        combine_partials<MP, NCOLC, WS, NT>(reinterpret_cast<const float*>(tb + Lay::WPART), Lay::STAGE / 4,
                                             reinterpret_cast<float*>(bb + Lay::B_W),
                                             reinterpret_cast<float*>(bb + Lay::B_MU), r, lane);
        if (tsync_or(failed)) {
            broke = true;
            break;
        }
        // ---------------- hand buffer b to the core warp ----------------
        __syncwarp();
        if (lane == 0) mbar_arrive(barF + b);
        // Q, K, V and the partials are consumed: copy the next unit's Q and K
        // rows, and the previous unit's Q rows again (into the V rows) for its output.
        const long long un = u + stride;
        fence_proxy_async_smem();
        __syncwarp();
        if (un < n_units && !failed) {
            if (lane == 0) issue_qk(un);
            pend_qk = true;
        }
        if (kk >= 1 && !failed) {
            if (lane == 0) issue_q_again(u - stride);
            pend_v = true;
        }
        // ---------------- output of the previous unit ----------------
        if (kk >= 1) output_unit(kk - 1);
        // The V rows are free (the output's staging has been read).
        if (un < n_units && !failed) {
            if (lane == 0) issue_v(un);
            pend_v = true;
        }
    }
    if (kk >= 1 && !broke && !failed) {  // the last unit's output: its Q rows again, then the output
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) issue_q_again(u0 + (kk - 1) * stride);
        pend_v = true;
        output_unit(kk - 1);
    }
    if (lane == 0) bulk_wait_all();  // output stores complete before exit
    // Fault path only: copies still in flight land before the CTA's memory is released.
    if (pend_qk) (void)__all_sync(0xffffffffu, mbar_wait_bounded(barQK, phase_qk, kWaitNs));
    if (pend_v) (void)__all_sync(0xffffffffu, mbar_wait_bounded(barV, phase_v, kWaitNs));
}

template <typename T, int M, int NCOL, int DC, int PW, bool BIAS = false>
cudaError_t launch_team_dc(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                        int iters, cudaStream_t stream, unsigned int* fault, NystraBias bias = {}) {
    using Lay = TeamLayout<T, M, NCOL>;
    auto kern = nystra_team_kernel<T, M, NCOL, DC, PW, BIAS>;
    const size_t smem = (size_t)Lay::TEAMS * Lay::TEAM;
    static std::atomic<int> s_blocks[kMaxDevices];  // persistent grid size per device
    int blocks = 0;
    if (cudaError_t e = persistent_grid(kern, Lay::TEAMS * Lay::WARPS * 32, smem, s_blocks, &blocks); e != cudaSuccess)
        return e;
    const long long want = (n_units + Lay::TEAMS - 1) / Lay::TEAMS;
    const long long grid = want < blocks ? want : blocks;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<(unsigned)grid, Lay::TEAMS * Lay::WARPS * 32, smem, stream>>>((const T*)q, (const T*)k, (const T*)v, (T*)out,
                                                                 n_units, d, iters, sl2, fault, bias);
    return cudaGetLastError();
}

// The common head widths get kernels with d_h as a compile-time constant
// (constant strides and column bounds); others read it at run time.
template <typename T, int M, int NCOL, int PW>
cudaError_t launch_team(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                     int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias) {
    if constexpr (M <= 16)
        if (bias) {  // a score bias: the common head widths compiled in for m = 16 with segment
                     // landmarks (the common case), d_h read at run time otherwise
            if constexpr (M != 16 || PW != 0) {
            } else if constexpr (NCOL == 32) {
                if (d == 30)
                    return launch_team_dc<T, M, NCOL, 30, PW, true>(q, k, v, out, n_units, d, iters, stream, fault,
                                                                      *bias);
            } else {
                if (d == 32)
                    return launch_team_dc<T, M, NCOL, 32, PW, true>(q, k, v, out, n_units, d, iters, stream, fault,
                                                                      *bias);
            }
            return launch_team_dc<T, M, NCOL, 0, PW, true>(q, k, v, out, n_units, d, iters, stream, fault, *bias);
        }
    if constexpr (NCOL == 32) {
        if (d == 30) return launch_team_dc<T, M, NCOL, 30, PW>(q, k, v, out, n_units, d, iters, stream, fault);
    } else {
        if (d == 32) return launch_team_dc<T, M, NCOL, 32, PW>(q, k, v, out, n_units, d, iters, stream, fault);
    }
    return launch_team_dc<T, M, NCOL, 0, PW>(q, k, v, out, n_units, d, iters, stream, fault);
}

}  // namespace tc
}  // namespace nystra
