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
// [96 HB, K] are staged once in shared memory (K-major core matrices).  A
// tile of 128 token rows is 128 C contiguous 16-bit values in HBM, so one
// 1-D bulk copy brings it into a row-major staging buffer (two buffers where
// they fit); the rows are C values long (360 bytes at C = 180, not 16-byte
// aligned, so neither a tensor-map copy nor the MMA can take them as they
// are), and the loader warps rewrite each k-block of 64 columns into a ring
// stage in the core-matrix layout the MMA reads.
//   warps 0-11 epilogue: warp w reads TMEM lanes 32 (w mod 4) .. + 31 (token
//              rows) of part w / 4 (Q, K or V) of each head, adds the bias,
//              rounds to the I/O type into a private slot (32 rows x d_h, the
//              contiguous run of the head-split output those rows form) and
//              copies the slot out with coalesced 16-byte stores;
//   warp 12    allocates TMEM (two accumulators of 96 HB fp32 columns); lane 0
//              issues tcgen05.mma (M = 128, N = 96 HB, K = 16) and commits
//              each k-block to the ring's "empty" barrier and each tile to an
//              accumulator's "full" barrier;
//   warps 13-20 loaders: thread 0 issues the tile's bulk copy; all rewrite the
//              staged rows k-block by k-block (a 16-byte core-matrix row from
//              two 8-byte loads when C % 4 == 0, else 4-byte pieces; zeros
//              beyond C), fence them for the tensor cores and signal the
//              stage's "full" barrier.
// Every mbarrier wait is bounded (2 s); on expiry a warp records the fault
// and leaves its loop, the others follow at their next bounded wait, and the
// MMA thread drains its MMAs before TMEM is freed.
#include <atomic>

#include "common.cuh"
#include "ptx.cuh"
#include "tcgen05.cuh"

namespace nystra {

__device__ unsigned int g_fault_proj;  // bit 0: a bounded wait gave up

namespace proj {

constexpr uint64_t kWaitNs = 2000000000ull;
constexpr int BM = 128, KBLK = 64, STAGE = BM * KBLK * 2, HEAD_COLS = 96;
constexpr int EPI = 12, MMAW = 12, LOAD0 = 13, WARPS = 21, THREADS = WARPS * 32, LOADERS = 8 * 32;
constexpr int ESLOT = 32 * 32 * 2;  // an epilogue warp's block of 32 rows x d_h <= 32 16-bit values
constexpr int kSmemMax = 232448 - 1024;
constexpr int kBarLoad = 1;  // named barrier of the loader warps

struct Geo {
    int C, heads, d, N, HB, NHG, KB, NS, SD, KSTEPS, NTILE, KP, XT;
    long long T, n_tiles;
    // shared-memory offsets (bytes from the 1024-aligned base)
    int oB, oX, oA, oE, oBias, oBar, oTmem, bytes;
};

__host__ __device__ inline int align_up(int x, int a) { return (x + a - 1) / a * a; }

__host__ inline Geo geometry(int C, int heads, int d, int N, long long T, int HB, int SD, int NS) {
    Geo g{};
    g.C = C;
    g.heads = heads;
    g.d = d;
    g.N = N;
    g.T = T;
    g.HB = HB;
    g.SD = SD;
    g.NS = NS;
    g.NHG = (heads + HB - 1) / HB;
    g.KB = (C + KBLK - 1) / KBLK;
    g.KSTEPS = (C + 15) / 16;
    g.NTILE = HEAD_COLS * HB;
    g.KP = g.KB * KBLK;
    g.XT = align_up(BM * C * 2, 128);  // one staged tile of token rows
    g.n_tiles = (T + BM - 1) / BM;
    g.oB = 0;
    g.oX = align_up(g.NTILE * g.KP * 2, 1024);
    g.oA = g.oX + SD * g.XT;
    g.oE = g.oA + NS * STAGE;
    g.oBias = g.oE + EPI * ESLOT;
    g.oBar = align_up(g.oBias + g.NTILE * 4, 16);
    g.oTmem = g.oBar + (2 * NS + SD + 5) * 8;
    g.bytes = align_up(g.oTmem + 16, 128);
    return g;
}

// The largest configuration that fits: two staging buffers, two heads per
// CTA and a four-deep ring where possible, in that order of preference.
__host__ inline Geo fit(int C, int heads, int d, int N, long long T) {
    const int cand[9][3] = {{2, 2, 4}, {2, 2, 3}, {2, 2, 2}, {2, 1, 4}, {2, 1, 2},
                            {1, 2, 4}, {1, 2, 2}, {1, 1, 4}, {1, 1, 2}};  // SD, HB, NS
    Geo g{};
    for (const auto& c : cand) {
        if (c[1] == 2 && heads < 2) continue;
        g = geometry(C, heads, d, N, T, c[1], c[0], c[2]);
        if (g.bytes <= kSmemMax) return g;
    }
    g.bytes = -1;
    return g;
}

// Offset of element (row r, column k) in a K-major core-matrix operand whose
// rows hold kc_row core matrices (8 columns each) back to back.
__device__ __forceinline__ int cm_off(int r, int k, int kc_row) {
    return (((r >> 3) * kc_row + (k >> 3)) << 7) + ((r & 7) << 4) + ((k & 7) << 1);
}

// Two fp32 values rounded (nearest-even) to the I/O type and packed, the
// first in the low half (the lower address).
template <typename T>
struct Pack;
template <>
struct Pack<__nv_bfloat16> {
    static constexpr bool kBF16 = true;
    static __device__ __forceinline__ uint32_t pk(float a, float b) {
        uint32_t r;
        asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(b), "f"(a));
        return r;
    }
};
template <>
struct Pack<__half> {
    static constexpr bool kBF16 = false;
    static __device__ __forceinline__ uint32_t pk(float a, float b) {
        uint32_t r;
        asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(b), "f"(a));
        return r;
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
    const int SD = geo.SD, NTILE = geo.NTILE, KCB = geo.KP / 8;
    unsigned char* sB = sm + geo.oB;
    unsigned char* sX = sm + geo.oX;
    unsigned char* sA = sm + geo.oA;
    unsigned char* sE = sm + geo.oE;
    float* sBias = reinterpret_cast<float*>(sm + geo.oBias);
    uint64_t* full = reinterpret_cast<uint64_t*>(sm + geo.oBar);
    uint64_t* empty = full + NS;
    uint64_t* xfull = empty + NS;  // staged tile landed, per staging buffer
    uint64_t* accf = xfull + SD;
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
        for (int b = 0; b < SD; ++b) mbar_init(xfull + b, 1);
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
    // Stage the head group's weights in the core-matrix layout (zero rows for
    // padding features and absent heads, zero columns beyond C) and its bias.
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
    fence_proxy_async_smem();  // generic writes of B before the tensor cores read them
    t5::fence_before_sync();
    __syncthreads();
    t5::fence_after_sync();
    const uint32_t tmem = *tslot;

    if (warp >= LOAD0) {
        // ======================= loaders =======================
        const int lt = tid - LOAD0 * 32;
        auto issue_tile = [&](long long j, int b) {  // thread lt == 0: bulk copy of tile j into buffer b
            const long long m0 = j * BM;
            const long long rows = geo.T - m0 < BM ? geo.T - m0 : BM;  // a multiple of 32
            const uint32_t bytes = (uint32_t)(rows * C * 2);
            mbar_arrive_expect_tx(xfull + b, bytes);
            bulk_g2s(sX + b * geo.XT, x + (size_t)m0 * C, bytes, xfull + b);
        };
        long long j = slot;
        uint32_t issued = 0, landed = 0;  // copies into the staging buffers, in tile order (thread lt == 0)
        if (lt == 0)
            for (int b = 0; b < SD && j + (long long)b * P < geo.n_tiles; ++b) {
                issue_tile(j + (long long)b * P, b);
                ++issued;
            }
        uint32_t it = 0, a = 0;
        bool failed = false;  // a bounded wait of this warp gave up (warp-uniform)
        for (; j < geo.n_tiles; j += P, ++a) {
            const int xb = (int)(a % SD);
            if (!wait_all(xfull + xb, (a / SD) & 1u)) failed = true;
            else ++landed;
            const unsigned char* xs = sX + xb * geo.XT;
            for (int kb = 0; kb < KB; ++kb, ++it) {
                const int s = (int)(it % NS);
                if (!failed && it >= (uint32_t)NS && !wait_all(empty + s, ((it / NS) - 1) & 1u)) failed = true;
                if (failed) continue;
                unsigned char* st = sA + s * STAGE;
                if constexpr (G8) {
                    // one core-matrix row (8 columns, 16 bytes) per lane and step:
                    // a quarter-warp fills one core matrix (128 contiguous
                    // bytes), the two quarters of a half-warp take row groups
                    // 8 rows apart, whose 360-byte-pitch rows fall in disjoint
                    // banks (C = 180); two 8-byte loads (odd rows are only
                    // 8-byte aligned), one 16-byte store
                    const int wq = lt >> 3, i8 = lt & 7;  // quarter-warp of the loaders, row in the group
                    constexpr int QW = LOADERS / 8;       // quarter-warps of the loaders
#pragma unroll
                    for (int i = 0; i < 128 / QW; ++i) {
                        const int cm = i * QW + wq, rg = cm & 15, kc = cm >> 4;
                        const int row = (rg << 3) + i8, kk = kb * KBLK + (kc << 3);
                        const unsigned char* src = xs + ((size_t)row * C + kk) * 2;
                        uint2 lo = make_uint2(0u, 0u), hi = make_uint2(0u, 0u);
                        if (kk < C) lo = *reinterpret_cast<const uint2*>(src);
                        if (kk + 4 < C) hi = *reinterpret_cast<const uint2*>(src + 8);
                        *reinterpret_cast<uint4*>(st + (((rg << 3) + kc) << 7) + (i8 << 4)) =
                            make_uint4(lo.x, lo.y, hi.x, hi.y);
                    }
                } else {  // 4-byte pieces: 32 per core matrix
#pragma unroll 4
                    for (int i = 0; i < 16 * 8 * 32 / LOADERS; ++i) {
                        const int g = lt + LOADERS * i, cm = g >> 5, w32 = g & 31;
                        const int row = ((cm >> 3) << 3) + (w32 >> 2), kk = kb * KBLK + ((cm & 7) << 3) + ((w32 & 3) << 1);
                        uint32_t val = 0u;
                        if (kk < C) val = *reinterpret_cast<const uint32_t*>(xs + ((size_t)row * C + kk) * 2);
                        *reinterpret_cast<uint32_t*>(st + (cm << 7) + ((w32 >> 2) << 4) + ((w32 & 3) << 2)) = val;
                    }
                }
                fence_proxy_async_smem();  // the rewritten stage before the tensor cores read it
                mbar_arrive(full + s);
            }
            // Every loader has read staging buffer xb (the loaders leave
            // together if any of them gave up): refill it with the tile SD ahead.
            fence_proxy_async_smem();
            if (named_barrier_or(kBarLoad, LOADERS, failed)) {
                if (lt == 0) atomicOr(fault, 1u);
                break;
            }
            const long long jn = j + (long long)SD * P;
            if (jn < geo.n_tiles) {
                if (lt == 0) issue_tile(jn, xb);
                ++issued;
            }
        }
        // Fault path: copies in flight land before the CTA's memory is released
        // (tile a' goes to buffer a' mod SD; its landing is that buffer's
        // (a' / SD)-th phase).
        if (lt == 0)
            for (uint32_t t2 = landed; t2 < issued; ++t2)
                (void)mbar_wait_bounded(xfull + (t2 % SD), (t2 / SD) & 1u, kWaitNs);
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
        // ============ epilogue (warp w: TMEM lanes 32 (w mod 4).., part w / 4 of each head) ============
        const int e = warp & 3, p = warp >> 2;
        unsigned char* slot_e = sE + warp * ESLOT;  // this warp's 32 rows x d_h of one (head, part) block
        const int words = d / 2;                    // 32-bit words per row
        const int chunks = 4 * d;                   // 16-byte pieces of the block (32 rows x 2 d bytes)
        T* const dst = p == 0 ? q : (p == 1 ? k : v);
        const bool biased = bqkv != nullptr;
        uint32_t a = 0;
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
            if (!valid) {  // rows past the end: release the accumulator and go on (warp-uniform)
                t5::fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(acce + buf);
                continue;
            }
#pragma unroll 1
            for (int hl = 0; hl < HB; ++hl) {
                const int h = hg * HB + hl;
                uint32_t r[32];
                t5::ld_32x32b_x32(tmem + ((uint32_t)(32 * e) << 16) + (uint32_t)(buf * NTILE + hl * HEAD_COLS + p * 32),
                                  r);
                t5::wait_ld();
                if (hl == HB - 1) {  // this warp's last TMEM read of the tile: release the accumulator
                    t5::fence_before_sync();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(acce + buf);
                }
                if (h >= heads) break;  // warp-uniform
                // row `lane` of the block, rounded, into the slot (odd word
                // counts: conflict-free 4-byte stores)
                uint32_t* row = reinterpret_cast<uint32_t*>(slot_e) + lane * words;
                const float* bs = sBias + hl * HEAD_COLS + p * 32;
#pragma unroll
                for (int f = 0; f < 16; ++f)
                    if (2 * f < d) {
                        float x0 = __uint_as_float(r[2 * f]), x1 = __uint_as_float(r[2 * f + 1]);
                        if (biased) {
                            x0 += bs[2 * f];
                            x1 += bs[2 * f + 1];
                        }
                        row[f] = Pack<T>::pk(x0, x1);
                    }
                __syncwarp();
                // the block is one contiguous run of the head-split output:
                // coalesced 16-byte copies out
                const uint4* src4 = reinterpret_cast<const uint4*>(slot_e);
                uint4* dst4 = reinterpret_cast<uint4*>(dst + (((size_t)wi * heads + h) * N + t0) * d);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int c = lane + 32 * i;
                    if (c < chunks) dst4[c] = src4[c];
                }
                __syncwarp();  // the slot is read before the next block overwrites it
            }
        }
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
    const nystra::proj::Geo g = nystra::proj::fit(C, heads, d, N, n_windows * N);
    if (g.bytes < 0) return cudaErrorInvalidValue;
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
