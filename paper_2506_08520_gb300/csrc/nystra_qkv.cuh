// Fused Q/K/V projection front end for 8x8 windows (N = 64 tokens), m <= 16,
// even d_h <= 32, 16-bit I/O.  The projections of Eq. (1) (Q = X W_Q,
// K = X W_K, V = X W_V, split into heads, plus the optional projection bias
// of the restoration models' layers) are computed on the tensor cores from the
// window's tokens and handed straight to the stage-pool kernel's phases
// (nystra_pool.cuh: landmarks, S_L / G_L^n, S_U / W, the core, the output),
// so Q, K and V never reach HBM: per unit the launch reads the window's
// tokens (from HBM once per window, from L2 for its other heads) instead of
// Q, K and V.
//
// Head-stationary CTAs.  CTA c serves head h = c mod heads and the windows
// c / heads + i G_h (G_h = grid / heads CTAs per head, i = 0, 1, ...), so the
// head's weights (three d_h x C blocks) are staged in shared memory once per
// CTA, as m16n8k16 B fragments in lane order (one conflict-free 8-byte load
// per fragment), and the CTAs of one window's heads work on the same windows
// at about the same time, so the window's tokens come from L2 after the first.
//
// Warps.  Each of the NW warps takes one unit at a time (window i = w,
// w + NW, ... of its CTA).  It projects in two halves of 32 tokens: A
// fragments (token rows, C contiguous 16-bit values) straight from global
// memory, loaded three k-steps ahead of their MMAs (two with shared stages,
// whose 12 warps leave fewer registers), against the three weight
// blocks at once (96 fp32 accumulators); the results plus bias, rounded to
// the I/O type as an unfused projection would store them, go to a Q, K, V
// stage.  The core and the output run on warp-private state; the output tile
// leaves with one bulk store.
//
// Stages.  A stage is dead once the front phase has read it (G_L^n is
// parked, so the output does not read Q again).  With a short projection
// (C <= 64) two warps share each stage (PAIR: 12 warps on 6 stages, as the
// pool kernel shares its stages): warp w and warp w + NS take turns in the
// order of their windows (stage w mod NS serves windows i = w mod NS, + NS,
// + 2 NS, ...), the k-th user waiting, on the stage's mbarrier (bounded), for
// the (k-1)-th to arrive after its front phase; the extra warps hide the
// core's latency.  A longer projection keeps the stage busy for most of a
// unit, so sharing would serialise the two warps' projections: 8 warps with a
// stage each, and no waits (measured: 12 shared-stage warps are 16% faster at
// C = 32, 2-12% slower at C = 180).
#pragma once

#include "nystra_pool.cuh"

namespace nystra {
namespace tc {

template <typename T, int M, int NCOL, bool PAIR>
struct QkvLayout {
    using PL = PoolLayout<T, M, NCOL>;
    static constexpr size_t HDR = 128;               // the shared stages' mbarriers
    static constexpr size_t FRAG = 3 * 4 * 32 * 8;   // weight fragments per k-step: 3 blocks x 4 n-tiles x 32 lanes x 8 B
    // warps per CTA: 12 on 6 shared stages (C <= 64), else as many with a
    // stage each as fit beside the widest projection's weights (C = 352)
    static constexpr int NW = PAIR ? 12 : (int)((kSmemLimit - HDR - 22 * FRAG) / (PL::STAGE + PL::PRIV));
    static constexpr int NS = PAIR ? NW / 2 : NW;    // Q/K/V stages
    // k-steps ks = ceil(C / 16): header, weights, stages, warp-private state
    static constexpr size_t stages_at(int ks) { return HDR + (size_t)ks * FRAG; }
    static constexpr size_t priv_at(int ks) { return stages_at(ks) + NS * PL::STAGE; }
    static constexpr size_t bytes(int ks) { return priv_at(ks) + NW * PL::PRIV; }
    static_assert(NS * 8 <= HDR, "one mbarrier per stage");
    static_assert(PL::STAGE % 128 == 0 && PL::PRIV % 128 == 0 && FRAG % 128 == 0, "regions stay 128-byte aligned");
};

__device__ __forceinline__ uint32_t ldg_u32(const void* p) { return __ldg(reinterpret_cast<const unsigned int*>(p)); }

// Stages head h's weight fragments: entry ((kk * 3 + mat) * 4 + nt) * 32 + lane
// holds the two B registers of lane `lane` for k-step kk, block mat (Q, K, V)
// and n-tile nt: features n = 8 nt + lane / 4 of the head, inputs
// k = 16 kk + 2 (lane % 4) (+1) and k + 8 (+1); zero beyond d_h or C.
template <typename T>
__device__ __forceinline__ void stage_weights(const T* __restrict__ wqkv, int C, int h, int d, int ks, uint2* wf) {
    const int total = ks * 3 * 4 * 32;
    for (int i = threadIdx.x; i < total; i += blockDim.x) {
        const int ln = i & 31, nt = (i >> 5) & 3, rest = i >> 7;
        const int mat = rest % 3, kk = rest / 3;
        const int n = 8 * nt + (ln >> 2), k = 16 * kk + 2 * (ln & 3);
        uint2 f = make_uint2(0u, 0u);
        if (n < d) {
            const T* row = wqkv + (size_t)(mat * C + h * d + n) * C;
            if (k < C) f.x = ldg_u32(row + k);
            if (k + 8 < C) f.y = ldg_u32(row + k + 8);
        }
        wf[i] = f;
    }
}

// Q, K, V of one unit ([64, d] each, row-major, consecutive in `qkv`) from the
// window's tokens xw ([64, C] in global memory) and the staged fragments; the
// A fragments are loaded DEPTH k-steps ahead of their MMAs.
template <typename T, int DEPTH>
__device__ __forceinline__ void project_unit(const T* __restrict__ xw, const uint2* wf,
                                             const float* __restrict__ bqkv, int C, int h, int d, int ks, T* qkv,
                                             int g, int t, int lane) {
    using Op = Mma16<T>;
#pragma unroll 1
    for (int half = 0; half < 2; ++half) {
        float acc[3][4][2][4];
#pragma unroll
        for (int a = 0; a < 3; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b)
#pragma unroll
                for (int c = 0; c < 2; ++c)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[a][b][c][e] = 0.f;
        // lane's token rows 32 half + 16 mt + g (+8), inputs 2t (+1) and 2t + 8 (+1) of each k-step
        const T* r0 = xw + (size_t)(32 * half + g) * C + 2 * t;
        auto lda = [&](int kk, uint32_t (&a)[2][4]) {
            const int k = 16 * kk;
            const bool v0 = k + 2 * t < C, v1 = k + 8 + 2 * t < C;  // C even: pairs are whole
#pragma unroll
            for (int mt = 0; mt < 2; ++mt) {
                const T* p = r0 + (size_t)(16 * mt) * C + k;
                a[mt][0] = v0 ? ldg_u32(p) : 0u;
                a[mt][1] = v0 ? ldg_u32(p + 8 * C) : 0u;
                a[mt][2] = v1 ? ldg_u32(p + 8) : 0u;
                a[mt][3] = v1 ? ldg_u32(p + 8 * C + 8) : 0u;
            }
        };
        auto mma_step = [&](int kk, const uint32_t (&a)[2][4]) {
            const uint2* wk = wf + (size_t)kk * (3 * 4 * 32) + lane;
#pragma unroll
            for (int mat = 0; mat < 3; ++mat)
#pragma unroll
                for (int nt = 0; nt < 4; ++nt) {
                    const uint2 b = wk[(mat * 4 + nt) * 32];
                    Op::k16(acc[mat][nt][0], a[0], b.x, b.y);
                    Op::k16(acc[mat][nt][1], a[1], b.x, b.y);
                }
        };
        // k-steps at or beyond ks load nothing (v0 = v1 = false)
        if constexpr (DEPTH == 3) {
            uint32_t a0[2][4], a1[2][4], a2[2][4];
            lda(0, a0);
            lda(1, a1);
            lda(2, a2);
#pragma unroll 1
            for (int kk = 0; kk < ks; kk += 3) {
                mma_step(kk, a0);
                lda(kk + 3, a0);
                if (kk + 1 < ks) mma_step(kk + 1, a1);
                lda(kk + 4, a1);
                if (kk + 2 < ks) mma_step(kk + 2, a2);
                lda(kk + 5, a2);
            }
        } else {
            uint32_t a0[2][4], a1[2][4];
            lda(0, a0);
            lda(1, a1);
#pragma unroll 1
            for (int kk = 0; kk < ks; kk += 2) {
                mma_step(kk, a0);
                lda(kk + 2, a0);
                if (kk + 1 < ks) mma_step(kk + 1, a1);
                lda(kk + 3, a1);
            }
        }
        // + bias, rounded to the I/O type, into the stage
#pragma unroll
        for (int mat = 0; mat < 3; ++mat) {
            T* dst = qkv + (size_t)mat * 64 * d;
            const float* bm = bqkv ? bqkv + mat * C + h * d : nullptr;
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
                const int col = 8 * nt + 2 * t;
                if (col < d) {
                    const float b0 = bm ? __ldg(bm + col) : 0.f, b1 = bm ? __ldg(bm + col + 1) : 0.f;
#pragma unroll
                    for (int mt = 0; mt < 2; ++mt) {
                        const int row = 32 * half + 16 * mt + g;
                        const float* c = acc[mat][nt][mt];
                        *reinterpret_cast<uint32_t*>(dst + row * d + col) = Op::pack(c[0] + b0, c[1] + b1);
                        *reinterpret_cast<uint32_t*>(dst + (row + 8) * d + col) = Op::pack(c[2] + b0, c[3] + b1);
                    }
                }
            }
        }
    }
}

template <typename T, int M, int NCOL, int PW, bool BIAS, bool PAIR>
__global__ void __launch_bounds__(QkvLayout<T, M, NCOL, PAIR>::NW * 32, 1)
nystra_qkv_kernel(const T* __restrict__ x, const T* __restrict__ wqkv, const float* __restrict__ bqkv,
                  T* __restrict__ out, long long n_windows, int heads, int d, int ks, int iters, float sl2,
                  unsigned int* fault, NystraBias bias) {
    using P = QkvLayout<T, M, NCOL, PAIR>;
    using PL = typename P::PL;
    constexpr int L = 64 / M;  // tokens per landmark segment
    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int g = lane >> 2, t = lane & 3;
    const int C = heads * d;
    const int h = (int)(blockIdx.x % heads);
    const long long Gh = gridDim.x / heads, w0 = blockIdx.x / heads;

    const int st = w % P::NS;  // this warp's stage (PAIR: shared with warp (w + NS) mod NW)
    uint64_t* sbar = reinterpret_cast<uint64_t*>(smem_raw) + st;
    uint2* wf = reinterpret_cast<uint2*>(smem_raw + P::HDR);
    T* Qs = reinterpret_cast<T*>(smem_raw + P::stages_at(ks) + (size_t)st * PL::STAGE);
    T* Ks = Qs + 64 * d;
    T* Vs = Qs + 128 * d;
    unsigned char* pv = smem_raw + P::priv_at(ks) + (size_t)w * PL::PRIV;
    uint32_t* glf = reinterpret_cast<uint32_t*>(pv + PL::GLF);
    T* qbar = reinterpret_cast<T*>(pv + PL::QB);
    T* kbar = reinterpret_cast<T*>(pv + PL::KB);
    float* mW = reinterpret_cast<float*>(pv + PL::W);
    T* yT = reinterpret_cast<T*>(pv + PL::YT);
    T* ob = reinterpret_cast<T*>(pv + PL::OUT);
    const uint32_t tile_bytes = (uint32_t)(64 * d * sizeof(T));

    if (threadIdx.x == 0) {
        for (int j = 0; j < P::NS; ++j) mbar_init(reinterpret_cast<uint64_t*>(smem_raw) + j, 1);
        fence_mbar_init();
    }
    stage_weights<T>(wqkv, C, h, d, ks, wf);
    __syncthreads();

    for (long long i = w;; i += P::NW) {
        const long long win = w0 + i * Gh;
        if (win >= n_windows) break;
        const long long u = win * heads + h;
        // the stage's k-th use (windows st, st + NS, ... alternate between the
        // two warps): wait until use k - 1 has finished its front phase
        const long long k = (i - st) / P::NS;
        if (PAIR && k > 0 && !__all_sync(0xffffffffu, mbar_wait_bounded(sbar, (uint32_t)((k - 1) & 1), kWaitNs))) {
            if (lane == 0) atomicOr(fault, 1u);
            break;
        }
        const long long bs = BIAS ? (bias.per_window ? u : h) : 0;
        const float* bLu = BIAS ? bias.L + (size_t)bs * 64 * M : nullptr;
        const float* bUu = BIAS ? bias.U + (size_t)bs * M * 64 : nullptr;
        const float* bAu = BIAS ? bias.A + (size_t)bs * M * M : nullptr;
        // ---------------- projection (Eq. 1) into the stage ----------------
        project_unit<T, PAIR ? 2 : 3>(x + (size_t)win * 64 * C, wf, bqkv, C, h, d, ks, Qs, g, t, lane);
        // the previous unit's output store has read its staging (which
        // overlaps the landmarks and W written below)
        if (lane == 0) bulk_wait_read_all();
        __syncwarp();
        // ---------------- front: landmarks (Algorithm 1 step 1) ----------------
        landmarks_mma<T, 64, L, PW>(Qs, qbar, 0, d, g, t);
        landmarks_mma<T, 64, L, PW>(Ks, kbar, 0, d, g, t);
        if constexpr (M < PL::MP) {  // zero the padding landmark rows
            landmarks_zero<T>(qbar, M, PL::MP, lane, 32);
            landmarks_zero<T>(kbar, M, PL::MP, lane, 32);
        }
        __syncwarp();
        // ---------------- front: S_L, G_L^n fragments (parked) ----------------
#pragma unroll
        for (int tm = 0; tm < 4; ++tm) {
            typename Opnd<T>::DReg f[PL::KTL][4];
            gl_tile<T, M, PL::KTL, BIAS>(Qs + (16 * tm + g) * d, kbar, d, g, t, sl2, f,
                                         BIAS ? bLu + (16 * tm + g) * M : nullptr);
#pragma unroll
            for (int kk = 0; kk < PL::KTL; ++kk) GlPark<T, M>::put(glf, (tm * PL::KTL + kk) * 32 + lane, f[kk]);
        }
        // ---------------- front: S_U, m_U, W = G_U^n [V | 1] ----------------
        float mU[1][2];
        front_su_w<T, M, NCOL, 1, BIAS>(qbar, Ks, Vs, d, g, t, sl2, mW, PL::WS, mU, bUu, 64);
        // the stage has been read: hand it to the other warp's next window
        if constexpr (PAIR) {
            __syncwarp();
            if (lane == 0) mbar_arrive(sbar);
        }
        // ---------------- core: G_A^n, Z_0, iteration, Y ----------------
        core_warp<T, M, NCOL, false, BIAS>(qbar, kbar, mU, mW, yT, iters, sl2, g, t, nullptr, bAu);
        __syncwarp();
        // ---------------- output: O = (G_L^n Y_:d) / (G_L^n Y_d) ----------------
        output_rows<T, M, NCOL, 1, true>(glf, Qs, kbar, yT, ob, d, g, t, lane, sl2);
        fence_proxy_async_smem();  // this lane's staging writes precede the bulk store
        __syncwarp();
        if (lane == 0) {
            bulk_s2g(out + (size_t)u * 64 * d, ob, tile_bytes);
            bulk_commit();
        }
    }
    if (lane == 0) bulk_wait_all();  // output stores complete before exit
}

template <typename T, int M, int NCOL, int PW, bool BIAS, bool PAIR>
cudaError_t launch_qkv_cfg(const void* x, const void* wqkv, const float* bqkv, void* out, long long n_windows,
                           int heads, int d, int iters, cudaStream_t stream, unsigned int* fault,
                           const NystraBias& bias) {
    using P = QkvLayout<T, M, NCOL, PAIR>;
    auto kern = nystra_qkv_kernel<T, M, NCOL, PW, BIAS, PAIR>;
    const int C = heads * d, ks = (C + 15) / 16;
    const size_t smem = P::bytes(ks);
    if (smem > kSmemLimit) return cudaErrorInvalidValue;  // not reached: the caller bounds C
    static std::atomic<int> s_blocks[kMaxDevices];  // persistent grid size per device
    int blocks = 0;
    if (cudaError_t e = persistent_grid(kern, P::NW * 32, kSmemLimit, s_blocks, &blocks); e != cudaSuccess)
        return e;
    // CTAs per head: enough to fill the device, no more than there are windows
    long long per_head = blocks / heads;
    if (per_head < 1) per_head = 1;
    if (per_head > n_windows) per_head = n_windows;
    const long long grid = per_head * heads;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<(unsigned)grid, P::NW * 32, smem, stream>>>((const T*)x, (const T*)wqkv, bqkv, (T*)out, n_windows,
                                                        heads, d, ks, iters, sl2, fault, bias);
    return cudaGetLastError();
}

// m in {8, 16} (square patches: m = 16); d_h read at run time; shared
// stages for C <= 64.
template <typename T, int M, int NCOL, int PW>
cudaError_t launch_qkv_m(const void* x, const void* wqkv, const float* bqkv, void* out, long long n_windows,
                         int heads, int d, int iters, cudaStream_t stream, unsigned int* fault, const NystraBias* bias) {
    const NystraBias b = bias ? *bias : NystraBias{};
    const bool pair = heads * d <= 64;
    if (bias)
        return pair ? launch_qkv_cfg<T, M, NCOL, PW, true, true>(x, wqkv, bqkv, out, n_windows, heads, d, iters,
                                                                  stream, fault, b)
                    : launch_qkv_cfg<T, M, NCOL, PW, true, false>(x, wqkv, bqkv, out, n_windows, heads, d, iters,
                                                                   stream, fault, b);
    return pair ? launch_qkv_cfg<T, M, NCOL, PW, false, true>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream,
                                                               fault, b)
                : launch_qkv_cfg<T, M, NCOL, PW, false, false>(x, wqkv, bqkv, out, n_windows, heads, d, iters,
                                                                stream, fault, b);
}

template <typename T>
cudaError_t launch_qkv(const void* x, const void* wqkv, const float* bqkv, void* out, long long n_windows,
                       int heads, int d, int m, int iters, int pool, cudaStream_t stream, unsigned int* fault,
                       const NystraBias* bias) {
    const bool wide = d > 30;  // the ones column needs a fifth n-tile when d_h = 32
    if (pool != 0) {
        if (m != 16) return cudaErrorInvalidValue;  // not reached: checked by the caller
        return wide ? launch_qkv_m<T, 16, 40, 8>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream, fault, bias)
                    : launch_qkv_m<T, 16, 32, 8>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream, fault, bias);
    }
    if (m == 8)
        return wide ? launch_qkv_m<T, 8, 40, 0>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream, fault, bias)
                    : launch_qkv_m<T, 8, 32, 0>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream, fault, bias);
    if (m == 16)
        return wide ? launch_qkv_m<T, 16, 40, 0>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream, fault, bias)
                    : launch_qkv_m<T, 16, 32, 0>(x, wqkv, bqkv, out, n_windows, heads, d, iters, stream, fault, bias);
    return cudaErrorInvalidValue;
}

}  // namespace tc
}  // namespace nystra

// Largest token width C = heads * d_h the fused kernel takes (nystra.h):
// its weight fragments fit beside the stages and the warps' state (shared
// stages only up to C = 64).
namespace nystra {
namespace tc {
constexpr int kQkvMaxC = 352;
static_assert(QkvLayout<__half, 16, 40, false>::bytes(kQkvMaxC / 16) <= kSmemLimit &&
                  QkvLayout<__half, 16, 32, false>::bytes(kQkvMaxC / 16) <= kSmemLimit &&
                  QkvLayout<__half, 8, 40, false>::bytes(kQkvMaxC / 16) <= kSmemLimit &&
                  QkvLayout<__half, 16, 40, true>::bytes(64 / 16) <= kSmemLimit &&
                  QkvLayout<__half, 8, 40, true>::bytes(64 / 16) <= kSmemLimit,
              "the widest projection must fit in shared memory");
}  // namespace tc
}  // namespace nystra

// One translation unit per I/O type defines its fault word and entry point.
#define NYSTRA_QKV_DEFINE(NAME, T)                                                                          \
    namespace nystra {                                                                                      \
    __device__ unsigned int g_fault_qkv_##NAME;                                                             \
    }                                                                                                       \
    namespace nystra_host {                                                                                 \
    cudaError_t launch_nystra_qkv_##NAME(const void* x, const void* wqkv, const float* bqkv, void* out,     \
                                         long long n_windows, int heads, int d, int m, int iters, int pool, \
                                         cudaStream_t stream, const nystra::NystraBias* bias) {             \
        static unsigned int* s_fault[nystra::kMaxDevices] = {}; /* fault word's address, per device */     \
        int dev = 0;                                                                                        \
        cudaError_t e = cudaGetDevice(&dev);                                                                \
        if (e != cudaSuccess) return e;                                                                     \
        if (dev < 0 || dev >= nystra::kMaxDevices) return cudaErrorInvalidDevice;                          \
        if (!s_fault[dev]) {                                                                                \
            e = cudaGetSymbolAddress((void**)&s_fault[dev], nystra::g_fault_qkv_##NAME);                    \
            if (e != cudaSuccess) return e;                                                                 \
        }                                                                                                   \
        return nystra::tc::launch_qkv<T>(x, wqkv, bqkv, out, n_windows, heads, d, m, iters, pool, stream,   \
                                         s_fault[dev], bias);                                               \
    }                                                                                                       \
    unsigned int take_fault_word_qkv_##NAME(cudaError_t* err) {                                             \
        unsigned int w = 0, zero = 0;                                                                       \
        *err = cudaMemcpyFromSymbol(&w, nystra::g_fault_qkv_##NAME, sizeof(w));                             \
        if (*err == cudaSuccess && w != 0)                                                                  \
            *err = cudaMemcpyToSymbol(nystra::g_fault_qkv_##NAME, &zero, sizeof(zero));                     \
        return w;                                                                                           \
    }                                                                                                       \
    }
