// Stage-pool PnP-Nystra kernel for 8x8 windows (N = 64 tokens), m <= 16,
// even d_h <= 32, 16-bit or fp32 I/O (fp32: split bf16 operands, see Opnd).
// Included by the N = 64 translation unit after nystra_tc.cuh, whose
// per-phase device functions it reuses.
//
// One warp processes one (window, head) unit at a time, as the grouped
// kernel does with one warp per unit, but a warp's Q, K and V rows are only
// needed by its front phase (landmarks, S_L and G_L^n, S_U and W), while the
// core (m x m iteration) and the output phase run on warp-private state.  A
// CTA therefore keeps NW warps on NS = NW / 2 shared staging buffers (as many
// as fit: 12 on 6) instead of one buffer per warp: warp w always uses stage w mod NS, alternating with
// its partner warp (w + NS) mod NW.  When a warp's front phase has consumed
// the stage it issues the bulk copies of the partner's next unit into it, so
// the copy overlaps the warp's own core and output.  Each warp waits on its
// own mbarrier, whose k-th phase is its k-th unit: a warp's next copy is only
// issued after it consumed the previous one, so phase parities never alias.
//
// Warp-private memory holds the landmarks, the parked G_L^n fragments, W,
// Y^T (over the landmarks, dead after G_A^n) and the output tile (over the
// rest, dead after the core), written with one bulk store per unit.
//
// Units: CTA b takes units b, b + G, b + 2G, ... (G = grid size); warp w
// takes the CTA's j-th unit for j = w (mod NW).
#pragma once

#include "nystra_tc.cuh"

namespace nystra {
namespace tc {

template <typename T, int M, int NCOL>
struct PoolLayout {
    static constexpr int ES = (int)sizeof(T);          // bytes per I/O element
    static constexpr int DS = (NCOL == 32) ? 30 : 32;  // staged row width bound (d_h <= DS)
    static constexpr int MP = 16, LS = LmS<T>::LS, WS = NCOL + 4, YS = YtS<T, M>::YS;
    static constexpr int KTL = (M >= 16) ? M / 16 : 1;  // k-steps of O = G_L^n Y
    static constexpr size_t STAGE = 3 * 64 * DS * ES;   // Q, K, V rows of one unit
    // warp-private layout
    static constexpr size_t GLF = 0;
    static constexpr size_t QB = GLF + 4 * KTL * 32 * GlPark<T, M>::BYTES;
    static constexpr size_t KB = QB + LmS<T>::bytes(MP);
    static constexpr size_t W = KB + LmS<T>::bytes(MP);  // fp32 MP x NCOL, row stride WS
    static constexpr size_t YT = QB;                     // Y^T: written after the core's last landmark read
    static constexpr size_t YT_BYTES = YtS<T, M>::bytes(NCOL);
    static constexpr size_t OUT = YT + YT_BYTES;  // output tile: Kbar's tail and W are dead by then
    static constexpr size_t END_A = W + MP * WS * 4;
    static constexpr size_t END_B = OUT + 64 * DS * ES;
    static constexpr size_t BAR = (((END_A > END_B) ? END_A : END_B) + 15) / 16 * 16;
    static constexpr size_t CNT = BAR + 8;  // copies issued to this warp (fault path)
    static constexpr size_t PRIV = ((BAR + 16 + 127) / 128) * 128;
    // warps: the most (up to 16 for 16-bit I/O, 8 for fp32), in pairs sharing a stage, that fit
    static constexpr int fit_warps() {
        int n = ES == 2 ? 16 : 8;
        while (n > 2 && (size_t)(n / 2) * STAGE + (size_t)n * PRIV > kSmemLimit) n -= 2;
        return n;
    }
    static constexpr int NW = fit_warps();
    static constexpr int NS = NW / 2;  // shared stages
    static constexpr size_t BYTES = NS * STAGE + NW * PRIV;
    static_assert(NW == 2 * NS, "each stage alternates between two warps");
    static_assert(YT + YT_BYTES <= W, "Y^T must not overlap W (read while Y^T is produced)");
    static_assert(OUT % 16 == 0 && STAGE % 16 == 0 && PRIV % 16 == 0, "bulk copies need 16-byte alignment");
    static_assert(BYTES <= kSmemLimit, "pool does not fit in shared memory");
};

template <typename T, int M, int NCOL, int DC, int PW, bool BIAS>
__global__ void __launch_bounds__(PoolLayout<T, M, NCOL>::NW * 32, 1)
nystra_pool_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v, T* __restrict__ out,
                   long long n_units, int d_in, int iters, float sl2, unsigned int* fault, NystraBias bias) {
    const int d = DC ? DC : d_in;  // d_h, a compile-time constant for the common head widths
    using P = PoolLayout<T, M, NCOL>;
    constexpr int L = 64 / M;  // tokens per landmark segment
    constexpr int RS = row_step(DC);  // token order of the staged rows (bank-conflict-free fragment loads)
    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int g = lane >> 2, t = lane & 3;
    const int partner = (w + P::NS) % P::NW;

    T* Qs = reinterpret_cast<T*>(smem_raw + (size_t)(w % P::NS) * P::STAGE);
    T* Ks = Qs + 64 * d;
    T* Vs = Qs + 128 * d;
    unsigned char* pv = smem_raw + (size_t)P::NS * P::STAGE + (size_t)w * P::PRIV;
    unsigned char* pp = smem_raw + (size_t)P::NS * P::STAGE + (size_t)partner * P::PRIV;
    uint32_t* glf = reinterpret_cast<uint32_t*>(pv + P::GLF);
    T* qbar = reinterpret_cast<T*>(pv + P::QB);
    T* kbar = reinterpret_cast<T*>(pv + P::KB);
    float* mW = reinterpret_cast<float*>(pv + P::W);
    T* yT = reinterpret_cast<T*>(pv + P::YT);
    T* ob = reinterpret_cast<T*>(pv + P::OUT);
    uint64_t* bar = reinterpret_cast<uint64_t*>(pv + P::BAR);
    uint32_t* cnt = reinterpret_cast<uint32_t*>(pv + P::CNT);

    const uint32_t tile_bytes = (uint32_t)(64 * d * sizeof(T));
    const long long G = gridDim.x;
    auto unit_of = [&](long long j) { return (long long)blockIdx.x + j * G; };
    // lane 0: copies of unit u into this warp's stage, completing on `b`
    auto issue = [&](long long u, uint64_t* b, uint32_t* c) {
        atomicAdd(c, 1u);
        mbar_arrive_expect_tx(b, 3u * tile_bytes);
        const size_t off = (size_t)u * 64 * d;
        bulk_g2s(Qs, q + off, tile_bytes, b);
        bulk_g2s(Ks, k + off, tile_bytes, b);
        bulk_g2s(Vs, v + off, tile_bytes, b);
    };

    if (lane == 0) {
        mbar_init(bar, 1);
        *cnt = 0u;
        fence_mbar_init();
    }
    __syncthreads();
    if (w < P::NS && lane == 0 && unit_of(w) < n_units) issue(unit_of(w), bar, cnt);

    uint32_t phase = 0, consumed = 0;
    for (long long j = w;; j += P::NW) {
        const long long u = unit_of(j);
        if (u >= n_units) break;
        // BIAS: this unit's blocks of the score bias (N = 64)
        const long long bs = BIAS ? (bias.per_window ? u : u % bias.heads) : 0;
        const float* bLu = BIAS ? bias.L + (size_t)bs * 64 * M : nullptr;
        const float* bUu = BIAS ? bias.U + (size_t)bs * M * 64 : nullptr;
        const float* bAu = BIAS ? bias.A + (size_t)bs * M * M : nullptr;
        const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(bar, phase, kWaitNs));
        if (!ok) {
            if (lane == 0) atomicOr(fault, 1u);
            break;
        }
        phase ^= 1u;
        ++consumed;
        // the previous unit's output store has read its staging (which
        // overlaps the landmarks and W written below)
        if (lane == 0) bulk_wait_read_all();
        __syncwarp();
        // ---------------- front: landmarks (Algorithm 1 step 1) ----------------
        landmarks_mma<T, 64, L, PW, RS>(Qs, qbar, 0, d, g, t);
        landmarks_mma<T, 64, L, PW, RS>(Ks, kbar, 0, d, g, t);
        if constexpr (M < P::MP) {  // zero the padding landmark rows
            landmarks_zero<T>(qbar, M, P::MP, lane, 32);
            landmarks_zero<T>(kbar, M, P::MP, lane, 32);
        }
        __syncwarp();
        // ---------------- front: S_L, G_L^n fragments (parked) ----------------
#pragma unroll
        for (int tm = 0; tm < 4; ++tm) {
            typename Opnd<T>::DReg f[P::KTL][4];
            gl_tile<T, M, P::KTL, BIAS, RS>(Qs + mtok<RS>(tm, g) * d, kbar, d, g, t, sl2, f,
                                            BIAS ? bLu + mtok<RS>(tm, g) * M : nullptr);
#pragma unroll
            for (int kk = 0; kk < P::KTL; ++kk) GlPark<T, M>::put(glf, (tm * P::KTL + kk) * 32 + lane, f[kk]);
        }
        // ---------------- front: S_U, m_U, W = G_U^n [V | 1] ----------------
        float mU[1][2];
        front_su_w<T, M, NCOL, 1, BIAS, RS>(qbar, Ks, Vs, d, g, t, sl2, mW, P::WS, mU, bUu, 64);
        // The stage is consumed: hand it to the partner's next unit.
        fence_proxy_async_smem();
        __syncwarp();
        const long long un = unit_of(j + P::NS);
        if (lane == 0 && un < n_units)
            issue(un, reinterpret_cast<uint64_t*>(pp + P::BAR), reinterpret_cast<uint32_t*>(pp + P::CNT));
        // ---------------- core: G_A^n, Z_0, iteration, Y ----------------
        core_warp<T, M, NCOL, false, BIAS>(qbar, kbar, mU, mW, yT, iters, sl2, g, t, nullptr, bAu);
        __syncwarp();
        // ---------------- output: O = (G_L^n Y_:d) / (G_L^n Y_d) ----------------
        output_rows<T, M, NCOL, 1, true, false, RS>(glf, Qs, kbar, yT, ob, d, g, t, lane, sl2);
        fence_proxy_async_smem();  // this lane's staging writes precede the bulk store
        __syncwarp();
        if (lane == 0) {
            bulk_s2g(out + (size_t)u * 64 * d, ob, tile_bytes);
            bulk_commit();
        }
    }
    if (lane == 0) bulk_wait_all();  // output stores complete before exit
    // Fault path only: a copy issued to this warp that it did not consume
    // (its wait gave up) still lands before the CTA's memory is released.
    __syncthreads();
    if (*cnt > consumed) (void)__all_sync(0xffffffffu, mbar_wait_bounded(bar, phase, kWaitNs));
}

template <typename T, int M, int NCOL, int DC, int PW, bool BIAS = false>
cudaError_t launch_pool_dc(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                        int iters, cudaStream_t stream, unsigned int* fault, NystraBias bias = {}) {
    using P = PoolLayout<T, M, NCOL>;
    auto kern = nystra_pool_kernel<T, M, NCOL, DC, PW, BIAS>;
    static std::atomic<int> s_blocks[kMaxDevices];  // persistent grid size per device
    int blocks = 0;
    if (cudaError_t e = persistent_grid(kern, P::NW * 32, P::BYTES, s_blocks, &blocks); e != cudaSuccess)
        return e;
    const long long grid = n_units < blocks ? n_units : blocks;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<(unsigned)grid, P::NW * 32, P::BYTES, stream>>>((const T*)q, (const T*)k, (const T*)v, (T*)out,
                                                             n_units, d, iters, sl2, fault, bias);
    return cudaGetLastError();
}

// The common head widths get kernels with d_h as a compile-time constant
// (constant strides and column bounds); others read it at run time.
template <typename T, int M, int NCOL, int PW>
cudaError_t launch_pool(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                     int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias) {
    if (bias)  // a score bias: d_h read at run time (one kernel per shape, not per width)
        return launch_pool_dc<T, M, NCOL, 0, PW, true>(q, k, v, out, n_units, d, iters, stream, fault, *bias);
    if constexpr (NCOL == 32) {
        if (d == 30) return launch_pool_dc<T, M, NCOL, 30, PW>(q, k, v, out, n_units, d, iters, stream, fault);
    } else {
        if (d == 32) return launch_pool_dc<T, M, NCOL, 32, PW>(q, k, v, out, n_units, d, iters, stream, fault);
    }
    return launch_pool_dc<T, M, NCOL, 0, PW>(q, k, v, out, n_units, d, iters, stream, fault);
}

}  // namespace tc
}  // namespace nystra
