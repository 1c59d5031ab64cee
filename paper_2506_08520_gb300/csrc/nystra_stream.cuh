// Streaming team kernel for 32x32 windows (N = 1024 tokens), m <= 32, even
// d_h <= 32, 16-bit I/O (m = 32: the core runs on two warps, dist_core).  Included by the N = 1024 translation unit after
// nystra_tc.cuh, whose per-phase device functions it reuses.
//
// A whole 32x32 unit (Q, K, V: 184 KB at d_h = 30) fills an SM, so staging
// units whole leaves HBM idle while the front phase runs and serialises the
// m x m core with everything else.  This kernel streams 64-token chunks
// instead.  A team is four token warps (256 tokens each) plus a dedicated core
// warp; per-unit state (landmarks, W, m_U, Y^T) is double-buffered, so the
// core warp runs the iteration of unit k while the token warps work on unit
// k + 1 and the output of unit k.  Each token warp walks a fixed sequence of
// chunk tasks through a private ring of NSLOT chunk buffers, copying task
// v + NSLOT into a buffer as soon as task v has released it:
//
//   Q(k)   Q chunk -> landmark sums of Qbar          (after the 4th: [sync])
//   KV(k)  K and V chunks -> landmark sums of Kbar, S_U with running maxima,
//          partial W_r = G_U^n [V | 1]               (after the 4th: [sync],
//          combine into W and m_U, [sync], signal the core: mbarrier F_b)
//   OUT(k-1) Q chunk of the previous unit, read again -> S_L, G_L^n (from the
//          resident Kbar), O = (G_L^n Y_:d) / (G_L^n Y_d) once the core of
//          that unit is done (mbarrier C_b), written in place over the Q rows
//          and bulk-stored.
//
// Q is read twice (the second time usually from L2: it was read about one
// unit earlier); K, V once; O written once.  [sync] is a named barrier over
// the four token warps.  Every mbarrier wait is bounded; a warp whose wait
// gives up keeps to the barrier sequence and the token warps leave together
// after the next barrier, whose OR-reduction gives every warp the same verdict.
#pragma once

#include "nystra_tc.cuh"

namespace nystra {
namespace tc {

template <typename T, int M, int NCOL>
struct StreamLayout {
    static constexpr int NT = 4, TPW = 256, N = NT * TPW, CH = 64, NCHK = TPW / CH;
    static constexpr int CWN = M > 16 ? M / 16 : 1;  // core warps (m = 32: distributed core)
    static constexpr int MT = (M + 15) / 16;         // landmark m-tiles
    static constexpr int DS = (NCOL == 32) ? 30 : 32;
    static constexpr int MP = MT * 16, LS = LmS<T>::LS, WS = NCOL + 4;
    static constexpr int L = N / M, LPW = TPW / L;  // tokens per segment, segments per token warp
    static constexpr size_t XB = (size_t)CH * DS * 2;  // one tensor's chunk
    static constexpr size_t SLOT = 2 * XB;             // K and V (Q uses the first half)
    static constexpr size_t WPB = (size_t)MP * WS * 4 + MP * 4;  // W partial, row maxima
    static_assert(WPB <= SLOT, "the W partial lives in the slot of the last K/V chunk");
    // per-unit state.  Y^T is written by the core once it has read Qbar, W
    // and m_U for the last time, so it overlays them; a unit's Qbar is next
    // written two units later, after a token-warp barrier that follows every
    // warp's output pass of the unit (see the task order).
    static constexpr size_t B_QB = 0;
    static constexpr size_t B_W = B_QB + LmS<T>::bytes(MP);
    static constexpr size_t B_MU = B_W + MP * WS * 4;
    static constexpr size_t B_KB = ((B_MU + MP * 4 + 15) / 16) * 16;
    static constexpr size_t B_YT = B_QB;
    static constexpr size_t BUF = ((B_KB + LmS<T>::bytes(MP) + 127) / 128) * 128;
    static_assert(YtS<T, M>::bytes(NCOL) <= B_KB, "Y^T must fit over Qbar, W and m_U");
    static constexpr size_t SCR = CWN > 1 ? DistScratch<(M > 16 ? M : 32)>::BYTES : 0;
    template <int S>
    struct Team {
        static constexpr size_t WARP = S * SLOT;  // a token warp's ring of chunk buffers
        static constexpr size_t T_BUF = NT * WARP;
        static constexpr size_t T_BAR = T_BUF + 2 * BUF;  // slot bars [NT][S], F[2], C[2]
        static constexpr size_t T_SCR = ((T_BAR + (NT * S + 4) * 8 + 127) / 128) * 128;
        static constexpr size_t BYTES = ((T_SCR + SCR + 127) / 128) * 128;
    };
    static constexpr int WARPS = NT + CWN;  // per team
    // three teams with two-deep rings when they fit, else two with three-deep,
    // else two with two-deep
    static constexpr bool kThree = 3 * Team<2>::BYTES <= kSmemLimit;
    static constexpr bool kDeep = 2 * Team<3>::BYTES <= kSmemLimit;
    static constexpr int TEAMS = kThree ? 3 : (2 * Team<2>::BYTES <= kSmemLimit ? 2 : 1);
    static constexpr int NSLOT = kThree ? 2 : (kDeep ? 3 : 2);
    using TL = Team<NSLOT>;
    static constexpr size_t TEAM = TL::BYTES;
    static_assert(TEAMS * TEAM <= kSmemLimit, "teams must fit");
    static_assert(M <= 32 && L >= 16 && LPW <= 8, "segments per token warp fit one n-tile");
    static_assert(XB % 16 == 0 && SLOT % 16 == 0 && TL::WARP % 16 == 0 && BUF % 16 == 0, "16-byte alignment");
};

// Chunk task v of a team that processes `count` units (12 * count tasks, in
// blocks of four chunks).  SHORT (the one-warp core of m <= 16): Q(0), KV(0),
// then for k >= 1 Q(k), OUT(k - 1), KV(k), finally OUT(count - 1): a unit's Q
// rows are read again two blocks after their first read, while they are
// still in L2, and the core of unit k runs during Q(k + 1).  Otherwise (the
// slower distributed core of m = 32): Q(k), KV(k), OUT(k - 1) for each k,
// finally OUT(count - 1), so the core has two blocks to finish.
struct StreamTask {
    int k, type, c;  // unit (team-local), 0 = Q, 1 = KV, 2 = OUT, chunk
};
template <bool SHORT>
__device__ __forceinline__ StreamTask stream_task(int v, int count) {
    if constexpr (SHORT) {
        const int blk = v >> 2, c = v & 3;
        if (blk < 2) return {0, blk, c};
        const int k = (blk - 2) / 3 + 1, r = blk - 2 - 3 * (k - 1);
        if (k == count) return {count - 1, 2, c};
        return r == 0 ? StreamTask{k, 0, c} : (r == 1 ? StreamTask{k - 1, 2, c} : StreamTask{k, 1, c});
    } else {
        int i;  // position in the sequence Q(k) KV(k) OUT(k - 1), k = 0 .. count (without OUT(-1), Q/KV(count))
        if (v < 8) i = v;
        else if (v < 12 * count - 4) i = v + 4;
        else i = v + 12;
        const int k = i / 12, r = i - 12 * k;
        if (r < 8) return {k, r >> 2, r & 3};
        return {k - 1, 2, r & 3};
    }
}

template <typename T, int M, int NCOL, int DC, int PW, bool BIAS>
__global__ void __launch_bounds__(StreamLayout<T, M, NCOL>::TEAMS * StreamLayout<T, M, NCOL>::WARPS * 32, 1)
nystra_stream_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                     T* __restrict__ out, long long n_units, int d_in, int iters, float sl2, unsigned int* fault,
                     NystraBias bias) {
    static_assert(!BIAS || M <= 16, "a score bias runs with the one-warp core");
    const int d = DC ? DC : d_in;  // d_h, a compile-time constant for the common head widths
    using Lay = StreamLayout<T, M, NCOL>;
    using TL = typename Lay::TL;
    using R = typename Opnd<T>::DReg;
    constexpr int RS = row_step(DC);  // token order of the chunk rows (bank-conflict-free fragment loads)
    constexpr int NT = Lay::NT, TPW = Lay::TPW, N = Lay::N, MP = Lay::MP, WS = Lay::WS,
                  NSLOT = Lay::NSLOT, L = Lay::L, LPW = Lay::LPW, NTO = NCOL / 8, MT = Lay::MT;

    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int team = warp / Lay::WARPS, r = warp - team * Lay::WARPS;  // r >= NT: core warps
    const int g = lane >> 2, t = lane & 3;
    unsigned char* tb = smem_raw + (size_t)team * Lay::TEAM;
    auto buf = [&](int b) { return tb + TL::T_BUF + (size_t)b * Lay::BUF; };
    uint64_t* bars = reinterpret_cast<uint64_t*>(tb + TL::T_BAR);
    uint64_t* barF = bars + NT * NSLOT;  // F[b]: the token warps' state for the core is ready
    uint64_t* barC = barF + 2;           // C[b]: the core's Y^T is ready

    const long long stride = (long long)gridDim.x * Lay::TEAMS;
    // team-major numbering: when the units do not divide evenly, the teams with one unit more
    // sit on different SMs (one per SM) instead of filling the first SMs' every team
    const long long u0 = (long long)team * gridDim.x + blockIdx.x;
    const int count = u0 < n_units ? (int)((n_units - u0 + stride - 1) / stride) : 0;  // units of this team

    if (threadIdx.x == 0) {
        for (int tm = 0; tm < Lay::TEAMS; ++tm) {
            uint64_t* bb = reinterpret_cast<uint64_t*>(smem_raw + (size_t)tm * Lay::TEAM + TL::T_BAR);
            for (int i = 0; i < NT * NSLOT; ++i) mbar_init(bb + i, 1);
            mbar_init(bb + NT * NSLOT, NT);
            mbar_init(bb + NT * NSLOT + 1, NT);
            mbar_init(bb + NT * NSLOT + 2, Lay::CWN);
            mbar_init(bb + NT * NSLOT + 3, Lay::CWN);
        }
        fence_mbar_init();
    }
    // padding landmark rows (m < 16) stay zero: nothing else writes them
    if constexpr (M < MP) {
        for (int idx = threadIdx.x; idx < Lay::TEAMS * 2 * (MP - M) * 32; idx += blockDim.x) {
            const int tm = idx / (2 * (MP - M) * 32), rem = idx - tm * 2 * (MP - M) * 32;
            const int b = rem / ((MP - M) * 32), e = rem - b * (MP - M) * 32;
            T* qb = reinterpret_cast<T*>(smem_raw + (size_t)tm * Lay::TEAM + TL::T_BUF + (size_t)b * Lay::BUF +
                                         Lay::B_QB);
            T* kb = reinterpret_cast<T*>(smem_raw + (size_t)tm * Lay::TEAM + TL::T_BUF + (size_t)b * Lay::BUF +
                                         Lay::B_KB);
            landmarks_zero<T>(qb, M + (e >> 5), M + (e >> 5) + 1, e & 31, 32);
            landmarks_zero<T>(kb, M + (e >> 5), M + (e >> 5) + 1, e & 31, 32);
        }
    }
    __syncthreads();

    if (r >= NT) {
        // ======================= core warp(s) =======================
        const int c = r - NT;
        for (int kk = 0; kk < count; ++kk) {
            const int b = kk & 1;
            bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(barF + b, (uint32_t)((kk >> 1) & 1), kWaitNs));
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
                const long long uk = u0 + kk * stride;
                const float* bAu =
                    BIAS ? bias.A + (size_t)(bias.per_window ? uk : uk % bias.heads) * M * M : nullptr;
                core_warp<T, M, NCOL, false, BIAS>(reinterpret_cast<const T*>(bb + Lay::B_QB),
                                                   reinterpret_cast<const T*>(bb + Lay::B_KB), mU,
                                                   reinterpret_cast<const float*>(bb + Lay::B_W),
                                                   reinterpret_cast<T*>(bb + Lay::B_YT), iters, sl2, g, t, nullptr,
                                                   bAu);
            } else {
                using DSc = DistScratch<(M > 16 ? M : 32)>;
                unsigned char* scr = tb + TL::T_SCR;
                dist_core<T, (M > 16 ? M : 32), NCOL>(
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
    unsigned char* wr = tb + (size_t)r * TL::WARP;
    uint64_t* sbar = bars + r * NSLOT;
    const uint32_t xbytes = (uint32_t)(Lay::CH * d * sizeof(T));
    auto slot_x = [&](int s, int h) { return reinterpret_cast<T*>(wr + (size_t)s * Lay::SLOT + h * Lay::XB); };
    auto chunk_off = [&](long long unit, int c) {
        return ((size_t)unit * N + (size_t)r * TPW + (size_t)c * Lay::CH) * d;
    };
    const int total = 12 * count;
    // L2 policies: the first read of Q is kept for its second read (OUT);
    // every other read is its last.
    const uint64_t keep = l2_evict_last(), drop = l2_evict_first();
    // lane 0: copies of task vv into its slot
    auto issue = [&](int vv) {
        const StreamTask tk = stream_task<(M <= 16)>(vv, count);
        const int s = vv % NSLOT;
        const size_t off = chunk_off(u0 + tk.k * stride, tk.c);
        if (tk.type == 1) {
            mbar_arrive_expect_tx(sbar + s, 2u * xbytes);
            bulk_g2s_hint(slot_x(s, 0), k + off, xbytes, sbar + s, drop);
            bulk_g2s_hint(slot_x(s, 1), v + off, xbytes, sbar + s, drop);
        } else {
            mbar_arrive_expect_tx(sbar + s, xbytes);
            bulk_g2s_hint(slot_x(s, 0), q + off, xbytes, sbar + s, tk.type == 0 ? keep : drop);
        }
    };
    auto tsync = [&]() { named_barrier(1 + team, NT * 32); };
    // barrier that also tells every token warp whether any of them failed
    auto tsync_or = [&](bool f) { return named_barrier_or(1 + team, NT * 32, f); };

    int issued = 0, consumed = 0;
    if (lane == 0)
        for (; issued < NSLOT && issued < total; ++issued) issue(issued);
    issued = __shfl_sync(0xffffffffu, issued, 0);

    bool failed = false;  // a bounded wait of this warp gave up (warp-uniform)
    float cq[2][1][4], ck[2][1][4], w[MT][NTO][4], run[MT][2];
    R aq[MT][2][4];
    for (int vv = 0; vv < total; ++vv) {
        const StreamTask tk = stream_task<(M <= 16)>(vv, count);
        const int s = vv % NSLOT;
        const int b = tk.k & 1;
        unsigned char* bb = buf(b);
        // BIAS: the unit's score-bias slice (N = 1024 tokens, M landmarks)
        const long long bsl = BIAS ? (bias.per_window ? u0 + tk.k * stride : (u0 + tk.k * stride) % bias.heads) : 0;
        // ---------------- bounded wait for this task's chunk ----------------
        if (!failed) {
            if (__all_sync(0xffffffffu, mbar_wait_bounded(sbar + s, (uint32_t)((vv / NSLOT) & 1), kWaitNs))) {
                ++consumed;
            } else {
                failed = true;
                if (lane == 0) atomicOr(fault, 1u);
            }
        }
        T* X0 = slot_x(s, 0);
        if (tk.type == 0) {
            // ---------------- Q(k): landmark sums of Qbar ----------------
            if (tk.c == 0)
#pragma unroll
                for (int mf = 0; mf < 2; ++mf) cq[mf][0][0] = cq[mf][0][1] = cq[mf][0][2] = cq[mf][0][3] = 0.f;
            landmarks_acc<T, L, LPW, PW, RS>(X0, tk.c * Lay::CH, cq, d, g, t);
            if (tk.c == Lay::NCHK - 1) {
                // Qbar overlays the Y^T of unit k - 2: with the long core's
                // task order (m = 32) a warp's OUT(k - 2) precedes this task
                // without a barrier in between, so wait for every warp's.
                if constexpr (M > 16)
                    if (tsync_or(failed)) break;
                landmarks_put<T, LPW>(cq, reinterpret_cast<T*>(bb + Lay::B_QB), r * LPW, g, t);
                if (tsync_or(failed)) break;
                if constexpr (M > 16)  // KV(k) follows directly
#pragma unroll
                    for (int mt = 0; mt < MT; ++mt)
                        qbar_afrag<T>(reinterpret_cast<const T*>(bb + Lay::B_QB), mt, g, t, aq[mt]);
            }
        } else if (tk.type == 1) {
            // ---------------- KV(k): Kbar sums, S_U, partial W ----------------
            if (tk.c == 0) {
                if constexpr (M <= 16)  // OUT(k - 1) ran since Q(k): reload Qbar's operands
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
            landmarks_acc<T, L, LPW, PW, RS>(X0, tk.c * Lay::CH, ck, d, g, t);
#pragma unroll
            for (int mt = 0; mt < MT; ++mt)
                su_w_chunk<T, NCOL, BIAS, RS>(aq[mt], X0, slot_x(s, 1), d, g, t, sl2, 16 * mt + g < M,
                                          16 * mt + g + 8 < M, w[mt], run[mt][0], run[mt][1], true,
                                          BIAS ? bias.U + (size_t)bsl * M * N + (size_t)(16 * mt + g) * N +
                                                     r * TPW + tk.c * Lay::CH
                                               : nullptr,
                                          N);
            if (tk.c == Lay::NCHK - 1) {
                landmarks_put<T, LPW>(ck, reinterpret_cast<T*>(bb + Lay::B_KB), r * LPW, g, t);
                // the partial goes over this slot's K and V rows, consumed above
                float* wpart = reinterpret_cast<float*>(slot_x(s, 0));
                __syncwarp();
#pragma unroll
                for (int mt = 0; mt < MT; ++mt)
#pragma unroll
                    for (int j = 0; j < NTO; ++j) {
                        const int c = 8 * j + 2 * t, rr = 16 * mt + g;
                        *reinterpret_cast<float2*>(wpart + rr * WS + c) = make_float2(w[mt][j][0], w[mt][j][1]);
                        *reinterpret_cast<float2*>(wpart + (rr + 8) * WS + c) = make_float2(w[mt][j][2], w[mt][j][3]);
                    }
                if (t == 0) {
#pragma unroll
                    for (int mt = 0; mt < MT; ++mt) {
                        wpart[MP * WS + 16 * mt + g] = run[mt][0];
                        wpart[MP * WS + 16 * mt + g + 8] = run[mt][1];
                    }
                }
                tsync();
                combine_partials<MP, NCOL, WS, NT>(reinterpret_cast<const float*>(tb + (size_t)s * Lay::SLOT),
                                                    TL::WARP / 4, reinterpret_cast<float*>(bb + Lay::B_W),
                                                    reinterpret_cast<float*>(bb + Lay::B_MU), r, lane);
                if (tsync_or(failed)) break;
                __syncwarp();
                if (lane == 0) mbar_arrive(barF + b);
            }
        } else {
            // ---------------- OUT(k): output rows of this chunk ----------------
            if (tk.c == 0 && !failed) {
                if (!__all_sync(0xffffffffu, mbar_wait_bounded(barC + b, (uint32_t)((tk.k >> 1) & 1), kWaitNs))) {
                    failed = true;
                    if (lane == 0) atomicOr(fault, 1u);
                }
            }
            if (!failed) {
                output_rows<T, M, NCOL, 1, false, BIAS, RS>(
                    nullptr, X0, reinterpret_cast<const T*>(bb + Lay::B_KB), reinterpret_cast<const T*>(bb + Lay::B_YT),
                    X0, d, g, t, lane, sl2,
                    BIAS ? bias.L + (size_t)bsl * N * M + (size_t)(r * TPW + tk.c * Lay::CH) * M : nullptr);
                fence_proxy_async_smem();  // this lane's writes precede the bulk store
                __syncwarp();
                if (lane == 0) {
                    // O is not read again: evict it first, keeping L2 for the Q rows the
                    // output pass reads a second time
                    bulk_s2g_hint(out + chunk_off(u0 + tk.k * stride, tk.c), X0, xbytes, drop);
                    bulk_commit();
                    bulk_wait_read_all();
                }
            }
        }
        // The slot is released: copy the task NSLOT ahead into it.
        fence_proxy_async_smem();
        __syncwarp();
        if (issued < total && !failed) {
            if (lane == 0) issue(issued);
            ++issued;
        }
    }
    if (lane == 0) bulk_wait_all();  // output stores complete before exit
    // Fault path only: copies issued and not yet seen complete land before
    // the CTA's shared memory is released.
    for (int i = consumed; i < issued; ++i)
        (void)__all_sync(0xffffffffu, mbar_wait_bounded(sbar + i % NSLOT, (uint32_t)((i / NSLOT) & 1), kWaitNs));
}

template <typename T, int M, int NCOL, int DC, int PW, bool BIAS = false>
cudaError_t launch_stream_dc(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                          int iters, cudaStream_t stream, unsigned int* fault, NystraBias bias = {}) {
    using Lay = StreamLayout<T, M, NCOL>;
    auto kern = nystra_stream_kernel<T, M, NCOL, DC, PW, BIAS>;
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
cudaError_t launch_stream(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                     int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias) {
    if constexpr (M <= 16)
        if (bias) {  // a score bias: the common head widths compiled in for m = 16 with segment
                     // landmarks (the common case), d_h read at run time otherwise
            if constexpr (M != 16 || PW != 0) {
            } else if constexpr (NCOL == 32) {
                if (d == 30)
                    return launch_stream_dc<T, M, NCOL, 30, PW, true>(q, k, v, out, n_units, d, iters, stream, fault,
                                                                      *bias);
            } else {
                if (d == 32)
                    return launch_stream_dc<T, M, NCOL, 32, PW, true>(q, k, v, out, n_units, d, iters, stream, fault,
                                                                      *bias);
            }
            return launch_stream_dc<T, M, NCOL, 0, PW, true>(q, k, v, out, n_units, d, iters, stream, fault, *bias);
        }
    if constexpr (NCOL == 32) {
        if (d == 30) return launch_stream_dc<T, M, NCOL, 30, PW>(q, k, v, out, n_units, d, iters, stream, fault);
    } else {
        if (d == 32) return launch_stream_dc<T, M, NCOL, 32, PW>(q, k, v, out, n_units, d, iters, stream, fault);
    }
    return launch_stream_dc<T, M, NCOL, 0, PW>(q, k, v, out, n_units, d, iters, stream, fault);
}

}  // namespace tc
}  // namespace nystra
