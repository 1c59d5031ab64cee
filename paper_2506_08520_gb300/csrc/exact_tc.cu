// Tensor-core exact window attention, Eq. 1: O = softmax(Q K^T / sqrt(d_h)) V,
// even d_h <= 32; 16-bit I/O for windows of N = 64, 256 or 1024 tokens, fp32
// I/O (split bf16 operands, three MMAs per product) for N = 64 and 256.
//
// A group of WPU = N/64 warps processes one (window, head) unit; warp r
// bulk-copies rows [64r, 64r+64) of Q, K and V into its private stage (one
// mbarrier, bounded wait), and after a group barrier every warp reads all of
// the group's K and V.  Warp r computes the output rows it staged, one
// 16-row tile at a time, streaming the keys in 64-token chunks with the
// online (running-max) softmax: S = Q K_c^T (mma.sync, fp32 accumulate),
// P = exp(S - m) in registers fed directly as the A operand of P [V_c | 1],
// whose last column accumulates the row sums of the same rounded P.  Scores
// are scaled by log2(e)/sqrt(d_h) so each exponential is one FFMA and one ex2.
// This is the computation PnP-Nystra replaces; it is the in-library
// comparator.
#include "common.cuh"
#include "ptx.cuh"

namespace nystra {

__device__ unsigned int g_fault_exact_tc;  // bit 0: a bounded wait gave up

namespace {

constexpr uint64_t kWaitNs = 2000000000ull;
constexpr size_t kSmemLimit = 232448;

template <typename T, int NCOL, int WPU>
struct ExactLayout {
    static constexpr int DS = (NCOL == 32) ? 30 : 32;
    static constexpr size_t STAGE = 3 * 64 * (size_t)DS * sizeof(T);
    static constexpr size_t WARP_BYTES = ((STAGE + 127) / 128) * 128;
    static constexpr size_t GROUP_BYTES = ((8 * WPU + 16 + 127) / 128) * 128;  // mbarriers + flag
    static constexpr size_t PER_GROUP = GROUP_BYTES + WPU * WARP_BYTES;
};

template <typename T, int NCOL, int WPU, int GROUPS>
__global__ void __launch_bounds__(GROUPS * WPU * 32, 1)
exact_tc_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                T* __restrict__ out, long long n_units, int d, float sl2, unsigned int* fault) {
    using Lay = ExactLayout<T, NCOL, WPU>;
    using O = Opnd<T>;
    using R = typename O::Reg;
    constexpr int N = 64 * WPU, NTO = NCOL / 8;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = warp / WPU, r = warp - grp * WPU;
    const int g = lane >> 2, t = lane & 3;
    unsigned char* gb = smem_raw + (size_t)grp * Lay::GROUP_BYTES;
    unsigned char* wbase0 = smem_raw + (size_t)GROUPS * Lay::GROUP_BYTES + (size_t)(grp * WPU) * Lay::WARP_BYTES;
    const int td = 64 * d;
    auto stage_q = [&](int s) { return reinterpret_cast<T*>(wbase0 + (size_t)s * Lay::WARP_BYTES); };
    T* Qs = stage_q(r);
    uint64_t* bar = reinterpret_cast<uint64_t*>(gb) + r;
    volatile unsigned int* gflag = reinterpret_cast<volatile unsigned int*>(gb + 8 * WPU);

    auto gsync = [&]() {
        if constexpr (WPU == 1) __syncwarp();
        else named_barrier(1 + grp, WPU * 32);
    };
    const long long stride = (long long)gridDim.x * GROUPS;
    long long u = (long long)blockIdx.x * GROUPS + grp;
    const uint32_t tile_bytes = (uint32_t)(td * sizeof(T));
    auto issue = [&](long long unit) {
        const size_t off = (size_t)unit * N * d + (size_t)r * td;
        mbar_arrive_expect_tx(bar, 3u * tile_bytes);
        bulk_g2s(Qs, q + off, tile_bytes, bar);
        bulk_g2s(Qs + td, k + off, tile_bytes, bar);
        bulk_g2s(Qs + 2 * td, v + off, tile_bytes, bar);
    };
    if (lane == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
        if (r == 0) *gflag = 0u;
    }
    gsync();
    if (u < n_units && lane == 0) issue(u);
    uint32_t phase = 0;
    const int jd = d >> 3, tdn = (d & 7) >> 1, src = (lane & ~3) | tdn;

    for (; u < n_units; u += stride) {
        const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(bar, phase, kWaitNs));
        if (!ok && lane == 0) {
            atomicOr(fault, 1u);
            *gflag = 1u;
        }
        phase ^= 1u;
        gsync();  // every warp's K and V rows are in place
        if (*gflag != 0u) break;

        T* obase = out + (size_t)u * N * d + (size_t)r * td;
#pragma unroll 1
        for (int tm = 0; tm < 4; ++tm) {
            R aq[2][4];
            const T* q0 = Qs + (16 * tm + g) * d;
            const T* q1 = q0 + 8 * d;
#pragma unroll
            for (int kk = 0; kk < 2; ++kk) {
                const int c0 = 16 * kk + 2 * t, c1 = c0 + 8;
                aq[kk][0] = c0 < d ? O::ld(q0 + c0) : O::zero();
                aq[kk][1] = c0 < d ? O::ld(q1 + c0) : O::zero();
                aq[kk][2] = c1 < d ? O::ld(q0 + c1) : O::zero();
                aq[kk][3] = c1 < d ? O::ld(q1 + c1) : O::zero();
            }
            float o[NTO][4];
#pragma unroll
            for (int j = 0; j < NTO; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
            float run0 = -INFINITY, run1 = -INFINITY;
#pragma unroll 1
            for (int c = 0; c < WPU; ++c) {
                const T* Kc = stage_q(c) + td;
                const T* Vc = stage_q(c) + 2 * td;
                float s[8][4];
#pragma unroll
                for (int nt = 0; nt < 8; ++nt) {
                    s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
                    const T* kr = Kc + (8 * nt + g) * d;
#pragma unroll
                    for (int kk = 0; kk < 2; ++kk) {
                        const int c0 = 16 * kk + 2 * t, c1 = c0 + 8;
                        O::mma(s[nt], aq[kk], c0 < d ? O::ld(kr + c0) : O::zero(),
                               c1 < d ? O::ld(kr + c1) : O::zero());
                    }
                }
                float mx0 = run0, mx1 = run1;
#pragma unroll
                for (int nt = 0; nt < 8; ++nt) {
                    mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]) * sl2);
                    mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]) * sl2);
                }
                mx0 = quad_max(mx0);
                mx1 = quad_max(mx1);
                const float f0 = ex2(run0 - mx0), f1 = ex2(run1 - mx1);
#pragma unroll
                for (int j = 0; j < NTO; ++j) {
                    o[j][0] *= f0; o[j][1] *= f0; o[j][2] *= f1; o[j][3] *= f1;
                }
                run0 = mx0;
                run1 = mx1;
#pragma unroll
                for (int kt = 0; kt < 4; ++kt) {
                    R a[4];
                    a[0] = O::pk(ex2(fmaf(s[2 * kt][0], sl2, -mx0)), ex2(fmaf(s[2 * kt][1], sl2, -mx0)));
                    a[1] = O::pk(ex2(fmaf(s[2 * kt][2], sl2, -mx1)), ex2(fmaf(s[2 * kt][3], sl2, -mx1)));
                    a[2] = O::pk(ex2(fmaf(s[2 * kt + 1][0], sl2, -mx0)), ex2(fmaf(s[2 * kt + 1][1], sl2, -mx0)));
                    a[3] = O::pk(ex2(fmaf(s[2 * kt + 1][2], sl2, -mx1)), ex2(fmaf(s[2 * kt + 1][3], sl2, -mx1)));
#pragma unroll
                    for (int j = 0; j < NTO; ++j) {
                        const int c0 = 8 * j + 2 * t;
                        const R x0 = c0 < d ? O::ld(Vc + (16 * kt + g) * d + c0) : (c0 == d ? O::one() : O::zero());
                        const R x1 =
                            c0 < d ? O::ld(Vc + (16 * kt + 8 + g) * d + c0) : (c0 == d ? O::one() : O::zero());
                        O::mma(o[j], a, O::tr(x0), O::tr(x1));
                    }
                }
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
            T* o0 = obase + (16 * tm + g) * d;
            T* o1 = o0 + 8 * d;
#pragma unroll
            for (int j = 0; j < NTO; ++j) {
                const int c = 8 * j + 2 * t;
                if (c < d) {
                    O::st2(o0 + c, o[j][0] * i0, o[j][1] * i0);
                    O::st2(o1 + c, o[j][2] * i1, o[j][3] * i1);
                }
            }
        }
        gsync();  // no warp reads another warp's stage any more
        const long long un = u + stride;
        if (un < n_units && lane == 0) {
            fence_proxy_async_smem();
            issue(un);
        }
    }
}

template <typename T, int NCOL, int WPU>
cudaError_t launch_cfg(const void* q, const void* k, const void* v, void* out, long long n_units, int d,
                       cudaStream_t stream, unsigned int* fault) {
    using Lay = ExactLayout<T, NCOL, WPU>;
    constexpr int by_smem = (int)(kSmemLimit / Lay::PER_GROUP);
    // at most 512 threads (registers stay <= 128), 256 with split fp32 operands
    constexpr int by_threads = (sizeof(T) == 4 ? 8 : 16) / WPU;
    constexpr int kGroups = by_smem < by_threads ? by_smem : by_threads;
    static_assert(kGroups >= 1, "does not fit");
    auto kern = exact_tc_kernel<T, NCOL, WPU, kGroups>;
    const size_t smem = (size_t)kGroups * Lay::PER_GROUP;
    static std::atomic<int> s_blocks[kMaxDevices];  // persistent grid size per device
    int blocks = 0;
    if (cudaError_t e = persistent_grid(kern, kGroups * WPU * 32, smem, s_blocks, &blocks); e != cudaSuccess)
        return e;
    const long long want = (n_units + kGroups - 1) / kGroups;
    const long long grid = want < blocks ? want : blocks;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<(unsigned)grid, kGroups * WPU * 32, smem, stream>>>((const T*)q, (const T*)k, (const T*)v, (T*)out,
                                                              n_units, d, sl2, fault);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_t(const void* q, const void* k, const void* v, void* out, long long n_units, int N, int d,
                     cudaStream_t stream, unsigned int* fault) {
    const bool wide = d > 30;
    switch (N) {
        case 64:
            return wide ? launch_cfg<T, 40, 1>(q, k, v, out, n_units, d, stream, fault)
                        : launch_cfg<T, 32, 1>(q, k, v, out, n_units, d, stream, fault);
        case 256:
            return wide ? launch_cfg<T, 40, 4>(q, k, v, out, n_units, d, stream, fault)
                        : launch_cfg<T, 32, 4>(q, k, v, out, n_units, d, stream, fault);
        default:
            if constexpr (sizeof(T) == 4) return cudaErrorInvalidValue;  // not offered (see supports)
            else
                return wide ? launch_cfg<T, 40, 16>(q, k, v, out, n_units, d, stream, fault)
                            : launch_cfg<T, 32, 16>(q, k, v, out, n_units, d, stream, fault);
    }
}

}  // namespace
}  // namespace nystra

namespace nystra_host {
bool exact_tc_supports(int N, int d, int dtype) {
    const bool shape = d >= 2 && d <= 32 && d % 2 == 0;
    if (dtype == 0) return shape && (N == 64 || N == 256);
    return (dtype == 1 || dtype == 2) && (N == 64 || N == 256 || N == 1024) && shape;
}

cudaError_t launch_exact_tc(const void* q, const void* k, const void* v, void* out, long long n_units, int N,
                            int d, int dtype, cudaStream_t stream) {
    static unsigned int* s_fault[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!s_fault[dev]) {
        e = cudaGetSymbolAddress((void**)&s_fault[dev], nystra::g_fault_exact_tc);
        if (e != cudaSuccess) return e;
    }
    if (dtype == 0) return nystra::launch_t<float>(q, k, v, out, n_units, N, d, stream, s_fault[dev]);
    if (dtype == 1)
        return nystra::launch_t<__nv_bfloat16>(q, k, v, out, n_units, N, d, stream, s_fault[dev]);
    return nystra::launch_t<__half>(q, k, v, out, n_units, N, d, stream, s_fault[dev]);
}

unsigned int take_fault_word_exact_tc(cudaError_t* err) {
    unsigned int w = 0, zero = 0;
    *err = cudaMemcpyFromSymbol(&w, nystra::g_fault_exact_tc, sizeof(w));
    if (*err == cudaSuccess && w != 0) *err = cudaMemcpyToSymbol(nystra::g_fault_exact_tc, &zero, sizeof(zero));
    return w;
}
}  // namespace nystra_host
