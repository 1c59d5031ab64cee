// The projections of Eq. (1), Q = X W_Q, K = X W_K, V = X W_V (+ an optional
// projection bias), as one GEMM on the fifth-generation tensor cores with the
// head split done in the epilogue: nystra_project_qkv writes Q, K and V in
// the [n_windows, heads, N, d_h] layout nystra_attention reads.
//
// GEMM: D[t][n] = sum_c X[t][c] W[o(n)][c] over the T = n_windows * N token
// rows of X [T, C] and a head group's output columns n.  Column layout of a
// head group (HB = 1 or 2 heads): head-local hl, part p (Q, K, V) and feature
// f < 32 at n = 96 hl + 32 p + f, i.e. W row o = p C + h d_h + f for f < d_h
// and zero padding above, so each (head, part) is one aligned 32-column block
// of the accumulator.
//
// CTA (one per SM, head-group stationary): the head group's weights B
// [96 HB, K] are staged once in shared memory (K-major core matrices); tiles
// of 128 token rows stream through a ring of NS k-blocks of 64 columns.
//   warps 0-3  epilogue: warp e reads TMEM lanes 32e..32e+31 (token rows),
//              adds the bias, rounds to the I/O type and bulk-stores each
//              (head, part) block of 32 rows x d_h (one contiguous run of the
//              head-split output) from a two-slot staging area;
//   warp 4     allocates TMEM (two accumulators of 96 HB fp32 columns); lane 0
//              issues tcgen05.mma (M = 128, N = 96 HB, K = 16) and commits
//              each k-block to the ring's "empty" barrier and each tile to an
//              accumulator's "full" barrier;
//   warps 5-8  loaders: X rows are C 16-bit values (360 bytes at C = 180, not
//              16-byte aligned, so no tensor-map copy can move them); each
//              k-block goes in as 8-byte (or 4-byte) cp.async granules placed
//              in the core-matrix layout, completed by cp.async.wait_group,
//              made visible to the tensor cores by a proxy fence, then
//              signalled on the stage's "full" barrier.
// Ring stage s always holds k-block s mod KB (NS is a multiple of KB), so the
// zero padding beyond C is written once.  Every mbarrier wait is bounded
// (2 s); on expiry a warp records the fault and leaves its loop, the others
// follow at their next bounded wait, and the MMA thread drains its MMAs
// before TMEM is freed.
#include <atomic>

#include "common.cuh"
#include "ptx.cuh"
#include "tcgen05.cuh"

namespace nystra {

__device__ unsigned int g_fault_proj;  // bit 0: a bounded wait gave up

namespace proj {

constexpr uint64_t kWaitNs = 2000000000ull;
constexpr int BM = 128, KBLK = 64, STAGE = BM * KBLK * 2, HEAD_COLS = 96;
constexpr int EPI = 4, MMAW = 4, LOAD0 = 5, WARPS = 9, THREADS = WARPS * 32, LOADERS = 4 * 32;
constexpr int SLOT = 2048;  // one (head, part) block of 32 rows x d_h <= 32 16-bit values
constexpr int LAG = 3;      // k-blocks a loader keeps in flight before signalling the oldest

struct Geo {
    int C, heads, d, N, HB, NHG, KB, NS, KSTEPS, NTILE, KP;
    long long T, n_tiles;
    // shared-memory offsets (bytes from the 1024-aligned base)
    int oB, oA, oStage, oBias, oBar, oTmem, bytes;
};

__host__ __device__ inline int align_up(int x, int a) { return (x + a - 1) / a * a; }

__host__ inline Geo geometry(int C, int heads, int d, int N, long long T, int HB) {
    Geo g{};
    g.C = C;
    g.heads = heads;
    g.d = d;
    g.N = N;
    g.T = T;
    g.HB = HB;
    g.NHG = (heads + HB - 1) / HB;
    g.KB = (C + KBLK - 1) / KBLK;
    g.NS = g.KB * (6 / g.KB);
    g.KSTEPS = (C + 15) / 16;
    g.NTILE = HEAD_COLS * HB;
    g.KP = g.KB * KBLK;
    g.n_tiles = (T + BM - 1) / BM;
    g.oB = 0;
    g.oA = align_up(g.NTILE * g.KP * 2, 1024);
    g.oStage = g.oA + g.NS * STAGE;
    g.oBias = g.oStage + EPI * 2 * SLOT;
    g.oBar = align_up(g.oBias + g.NTILE * 4, 16);
    g.oTmem = g.oBar + (2 * g.NS + 5) * 8;
    g.bytes = align_up(g.oTmem + 16, 128);
    return g;
}

// Offset of element (row r, column k) in a K-major core-matrix operand whose
// rows hold kc_row core matrices (8 columns each) back to back.
__device__ __forceinline__ int cm_off(int r, int k, int kc_row) {
    return (((r >> 3) * kc_row + (k >> 3)) << 7) + ((r & 7) << 4) + ((k & 7) << 1);
}

template <typename T>
struct Pack;
template <>
struct Pack<__nv_bfloat16> {
    static constexpr bool kBF16 = true;
    static __device__ __forceinline__ uint32_t pk(float a, float b) {
        __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
        return *reinterpret_cast<uint32_t*>(&h);
    }
};
template <>
struct Pack<__half> {
    static constexpr bool kBF16 = false;
    static __device__ __forceinline__ uint32_t pk(float a, float b) {
        __half2 h = __floats2half2_rn(a, b);
        return *reinterpret_cast<uint32_t*>(&h);
    }
};

__device__ __forceinline__ bool wait_all(uint64_t* bar, uint32_t parity) {
    return __all_sync(0xffffffffu, mbar_wait_bounded(bar, parity, kWaitNs));
}

template <typename T, bool G8>
__global__ void __launch_bounds__(THREADS, 1)
project_qkv_kernel(const T* __restrict__ x, const T* __restrict__ w, const float* __restrict__ bqkv, T* __restrict__ q,
                   T* __restrict__ k, T* __restrict__ v, Geo geo, unsigned int* fault) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    unsigned char* sm = smem_raw;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int C = geo.C, d = geo.d, N = geo.N, heads = geo.heads, HB = geo.HB, KB = geo.KB, NS = geo.NS;
    const int NTILE = geo.NTILE, KCB = geo.KP / 8;
    unsigned char* sB = sm + geo.oB;
    unsigned char* sA = sm + geo.oA;
    float* sBias = reinterpret_cast<float*>(sm + geo.oBias);
    uint64_t* full = reinterpret_cast<uint64_t*>(sm + geo.oBar);
    uint64_t* empty = full + NS;
    uint64_t* accf = empty + NS;
    uint64_t* acce = accf + 2;
    uint64_t* drain = acce + 2;
    uint32_t* tslot = reinterpret_cast<uint32_t*>(sm + geo.oTmem);

    const int P = gridDim.x / geo.NHG;  // CTAs per head group
    const int hg = blockIdx.x % geo.NHG, slot = blockIdx.x / geo.NHG;
    const uint32_t ncols = 2 * NTILE <= 256 ? 256u : 512u;

    if (tid == 0) {
        for (int s = 0; s < NS; ++s) {
            mbar_init(full + s, LOADERS);
            mbar_init(empty + s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf + b, 1);
            mbar_init(acce + b, EPI);
        }
        mbar_init(drain, 1);
        fence_mbar_init();
    }
    if (warp == MMAW) {
        t5::tmem_alloc(tslot, ncols);
        t5::tmem_relinquish();
    }
    // Zero the ring (its padding beyond C is never written again), stage the
    // head group's weights in the core-matrix layout (zero rows for padding
    // features and absent heads, zero columns beyond C) and its bias.
    for (int i = tid; i < NS * STAGE / 16; i += THREADS) reinterpret_cast<uint4*>(sA)[i] = make_uint4(0, 0, 0, 0);
    for (int i = tid; i < NTILE * (geo.KP / 2); i += THREADS) {
        const int n = i / (geo.KP / 2), kk = 2 * (i - n * (geo.KP / 2));
        const int hl = n / HEAD_COLS, p = (n % HEAD_COLS) / 32, f = n % 32, h = hg * HB + hl;
        uint32_t val = 0;
        if (f < d && h < heads && kk < C)
            val = __ldg(reinterpret_cast<const uint32_t*>(w + ((size_t)p * C + (size_t)h * d + f) * C + kk));
        *reinterpret_cast<uint32_t*>(sB + cm_off(n, kk, KCB)) = val;
    }
    for (int n = tid; n < NTILE; n += THREADS) {
        const int hl = n / HEAD_COLS, p = (n % HEAD_COLS) / 32, f = n % 32, h = hg * HB + hl;
        sBias[n] = (bqkv && f < d && h < heads) ? __ldg(bqkv + (size_t)p * C + (size_t)h * d + f) : 0.f;
    }
    fence_proxy_async_smem();  // generic writes of the ring and B before the tensor cores read them
    t5::fence_before_sync();
    __syncthreads();
    t5::fence_after_sync();
    const uint32_t tmem = *tslot;

    if (warp >= LOAD0) {
        // ======================= loaders =======================
        const int lt = tid - LOAD0 * 32;
        constexpr int GB = G8 ? 8 : 4, GPC = 128 / GB, RPC = 16 / GB;  // granule bytes, per core matrix, per row
        uint32_t it = 0, done = 0;
        bool failed = false;
        for (long long j = slot; j < geo.n_tiles && !failed; j += P) {
            const long long m0 = j * BM;
            for (int kb = 0; kb < KB; ++kb, ++it) {
                const int s = (int)(it % NS);
                if (it >= (uint32_t)NS && !wait_all(empty + s, ((it / NS) - 1) & 1u)) {
                    failed = true;
                    if (lane == 0) atomicOr(fault, 1u);
                    break;
                }
                unsigned char* st = sA + s * STAGE;
                for (int g = lt; g < 16 * 8 * GPC; g += LOADERS) {
                    const int cm = g / GPC, wg = g - cm * GPC;
                    const int rg = cm >> 3, kc = cm & 7, row = rg * 8 + wg / RPC, piece = wg % RPC;
                    const int kk = kb * KBLK + kc * 8 + piece * (GB / 2);
                    if (kk < C && m0 + row < geo.T) {
                        if constexpr (G8)
                            t5::cp_async8(st + ((rg * 8 + kc) << 7) + ((wg / RPC) << 4) + piece * GB,
                                          x + (size_t)(m0 + row) * C + kk);
                        else
                            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(
                                             st + ((rg * 8 + kc) << 7) + ((wg / RPC) << 4) + piece * GB)),
                                         "l"(x + (size_t)(m0 + row) * C + kk)
                                         : "memory");
                    }
                }
                t5::cp_async_commit();
                if (it >= (uint32_t)LAG) {  // k-block it - LAG has landed: hand it to the tensor cores
                    t5::cp_async_wait<LAG>();
                    fence_proxy_async_smem();
                    mbar_arrive(full + (done % NS));
                    ++done;
                }
            }
        }
        t5::cp_async_wait<0>();
        fence_proxy_async_smem();
        if (!failed)
            for (; done < it; ++done) mbar_arrive(full + (done % NS));
    } else if (warp == MMAW) {
        // ======================= MMA issue =======================
        if (lane == 0) {
            const uint32_t idesc = t5::idesc_f16(Pack<T>::kBF16, BM, NTILE);
            const uint32_t aBase = smem_addr(sA), bBase = smem_addr(sB);
            uint32_t it = 0, a = 0;
            bool failed = false;
            for (long long j = slot; j < geo.n_tiles && !failed; j += P, ++a) {
                const int buf = (int)(a & 1);
                if (a >= 2 && !mbar_wait_bounded(acce + buf, ((a >> 1) - 1) & 1u, kWaitNs)) {
                    failed = true;
                    atomicOr(fault, 1u);
                    break;
                }
                t5::fence_after_sync();
                const uint32_t dt = tmem + (uint32_t)(buf * NTILE);
                for (int kb = 0; kb < KB; ++kb, ++it) {
                    const int s = (int)(it % NS);
                    if (!mbar_wait_bounded(full + s, (it / NS) & 1u, kWaitNs)) {
                        failed = true;
                        atomicOr(fault, 1u);
                        break;
                    }
                    t5::fence_after_sync();
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const int ks = kb * 4 + kk;
                        if (ks < geo.KSTEPS) {
                            const uint64_t ad = t5::sdesc(aBase + s * STAGE + kk * 256, 128, 8 * 128);
                            const uint64_t bd = t5::sdesc(bBase + ks * 256, 128, KCB * 128);
                            t5::mma_f16(dt, ad, bd, idesc, (kb | kk) != 0);
                        }
                    }
                    t5::commit(empty + s);  // the stage is free once these MMAs have read it
                }
                if (!failed) t5::commit(accf + buf);
            }
            t5::commit(drain);  // every MMA issued above has completed before TMEM is freed
            if (!mbar_wait_bounded(drain, 0, kWaitNs)) atomicOr(fault, 1u);
        }
        __syncwarp();
    } else {
        // ======================= epilogue (warp e: TMEM lanes 32e..) =======================
        const int e = warp;
        unsigned char* stg = sm + geo.oStage + e * 2 * SLOT;
        T* const dst_base[3] = {q, k, v};
        uint32_t a = 0, nst = 0;
        for (long long j = slot; j < geo.n_tiles; j += P, ++a) {
            const int buf = (int)(a & 1);
            if (!wait_all(accf + buf, (a >> 1) & 1u)) {
                if (lane == 0) atomicOr(fault, 1u);
                break;
            }
            t5::fence_after_sync();
            const long long T0 = j * BM + 32 * e;  // first token row of this warp (32 rows share a window)
            const bool valid = T0 < geo.T;
            const long long wi = T0 / N;
            const int t0 = (int)(T0 - wi * N);
            for (int hl = 0; hl < HB; ++hl) {
                const int h = hg * HB + hl;
                for (int p = 0; p < 3; ++p) {
                    uint32_t r[32];
                    const int col = buf * NTILE + hl * HEAD_COLS + p * 32;
                    t5::ld_32x32b_x32(tmem + ((uint32_t)(32 * e) << 16) + (uint32_t)col, r);
                    t5::wait_ld();
                    if (!valid || h >= heads) continue;  // warp-uniform
                    unsigned char* sl = stg + (nst & 1) * SLOT;
                    if (nst >= 2) {
                        if (lane == 0) t5::bulk_wait_read_1();  // the slot's previous store has read it
                        __syncwarp();
                    }
                    uint32_t* row = reinterpret_cast<uint32_t*>(sl) + lane * (d / 2);
                    const float* bs = sBias + hl * HEAD_COLS + p * 32;
#pragma unroll
                    for (int f = 0; f < 16; ++f)
                        if (2 * f < d)
                            row[f] = Pack<T>::pk(__uint_as_float(r[2 * f]) + bs[2 * f],
                                                 __uint_as_float(r[2 * f + 1]) + bs[2 * f + 1]);
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        T* dst = dst_base[p] + (((size_t)wi * heads + h) * N + t0) * d;
                        bulk_s2g(dst, sl, (uint32_t)(64 * d));
                        bulk_commit();
                    }
                    ++nst;
                }
            }
            t5::fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(acce + buf);
        }
        if (lane == 0) bulk_wait_all();
        __syncwarp();
    }
    t5::fence_before_sync();
    __syncthreads();
    t5::fence_after_sync();
    if (warp == MMAW) t5::tmem_dealloc(tmem, ncols);
}

}  // namespace proj
}  // namespace nystra

namespace nystra_host {

namespace {
std::atomic<int> s_sms[nystra::kMaxDevices];
unsigned int* s_fault[nystra::kMaxDevices];

template <typename T, bool G8>
cudaError_t launch_proj_t(const void* x, const void* w, const float* b, void* q, void* k, void* v,
                          const nystra::proj::Geo& g, cudaStream_t stream, unsigned int* fault, int sms) {
    auto kern = nystra::proj::project_qkv_kernel<T, G8>;
    static std::atomic<int> s_attr[nystra::kMaxDevices];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (!s_attr[dev].load(std::memory_order_relaxed)) {
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448)) != cudaSuccess)
            return e;
        s_attr[dev].store(1, std::memory_order_relaxed);
    }
    long long per = sms / g.NHG;
    if (per < 1) per = 1;
    if (per > g.n_tiles) per = g.n_tiles;
    const unsigned grid = (unsigned)(per * g.NHG);
    // at least 120 KB of shared memory: one CTA per SM, so the TMEM
    // allocations of co-resident CTAs never wait on one another
    const size_t smem = (size_t)(g.bytes + 1024 > 122880 ? g.bytes + 1024 : 122880);
    kern<<<grid, nystra::proj::THREADS, smem, stream>>>((const T*)x, (const T*)w, b, (T*)q, (T*)k, (T*)v, g, fault);
    return cudaGetLastError();
}
}  // namespace

// Shared memory (bytes) the projection needs for C inputs and HB heads per CTA.
int project_qkv_smem(int C, int heads, int HB) {
    return nystra::proj::geometry(C, heads, 2, 64, 64, HB).bytes + 1024;
}

cudaError_t launch_project_qkv(const void* x, const void* w, const float* b, void* q, void* k, void* v,
                               long long n_windows, int heads, int N, int d, int dtype, cudaStream_t stream) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= nystra::kMaxDevices) return cudaErrorInvalidDevice;
    int sms = s_sms[dev].load(std::memory_order_relaxed);
    if (!sms) {
        if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
        s_sms[dev].store(sms, std::memory_order_relaxed);
    }
    if (!s_fault[dev]) {
        if ((e = cudaGetSymbolAddress((void**)&s_fault[dev], nystra::g_fault_proj)) != cudaSuccess) return e;
    }
    const int C = heads * d;
    // two heads per CTA where both fit (fewer passes over X), else one
    const int HB = (heads >= 2 && project_qkv_smem(C, heads, 2) <= 232448) ? 2 : 1;
    const nystra::proj::Geo g = nystra::proj::geometry(C, heads, d, N, n_windows * N, HB);
    const bool g8 = C % 4 == 0;
    if (dtype == 1)
        return g8 ? launch_proj_t<__nv_bfloat16, true>(x, w, b, q, k, v, g, stream, s_fault[dev], sms)
                  : launch_proj_t<__nv_bfloat16, false>(x, w, b, q, k, v, g, stream, s_fault[dev], sms);
    return g8 ? launch_proj_t<__half, true>(x, w, b, q, k, v, g, stream, s_fault[dev], sms)
              : launch_proj_t<__half, false>(x, w, b, q, k, v, g, stream, s_fault[dev], sms);
}

unsigned int take_fault_word_proj(cudaError_t* err) {
    unsigned int w = 0, zero = 0;
    *err = cudaMemcpyFromSymbol(&w, nystra::g_fault_proj, sizeof(w));
    if (*err == cudaSuccess && w != 0) *err = cudaMemcpyToSymbol(nystra::g_fault_proj, &zero, sizeof(zero));
    return w;
}

}  // namespace nystra_host
