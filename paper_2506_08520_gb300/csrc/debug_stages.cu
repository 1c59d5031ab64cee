// Test-only stage dump of the tensor-core path for 8x8 windows (N = 64,
// m in {8, 16}, even d_h <= 32; square-patch landmarks with m = 16): one warp
// runs, for one unit, the same phase functions the stage-pool kernel runs
// (landmarks_mma, gl_tile, front_su_w, core_warp, output_rows) and writes
// every intermediate in fp32, so tests can hold each step of Algorithm 1
// against the float64 oracle on its own.  The paper has no counterpart;
// nystra_attention never calls this.
#include "common.cuh"
#include "nystra_tc.cuh"

namespace nystra {
namespace tc {
namespace {

// Two elements of a derived operand register (hi + lo pair in the MMA type
// of T: bf16 for fp32 I/O), widened to fp32.
template <typename T>
__device__ __forceinline__ float2 reg_f2(RegPair r) {
    using Op = typename Opnd<T>::Op;
    const float2 h = Op::unpack(r.hi), l = Op::unpack(r.lo);
    return make_float2(h.x + l.x, h.y + l.y);
}
// A stored derived value (landmark) widened to fp32.
template <typename T>
__device__ __forceinline__ float lm_f32(const T* p) {
    if constexpr (sizeof(T) == 2) return to_f32(p[0]) + to_f32(p[LmS<T>::LO]);
    else return p[0];
}

template <typename T, int M, int NCOL>
struct StageLayout {
    static constexpr int ES = (int)sizeof(T);
    static constexpr int DS = 32, MP = 16, LS = LmS<T>::LS, WS = NCOL + 4;
    static constexpr int KTL = (M >= 16) ? M / 16 : 1;
    static constexpr size_t QKV = 0;                                   // Q, K, V rows (64 x d each)
    static constexpr size_t QB = QKV + 3 * 64 * DS * ES;               // Qbar, MP x LS
    static constexpr size_t KB = QB + LmS<T>::bytes(MP);               // Kbar, MP x LS
    static constexpr size_t GLF = (KB + LmS<T>::bytes(MP) + 15) / 16 * 16;  // parked G_L^n fragments
    static constexpr size_t W = GLF + 4 * KTL * 32 * GlPark<T, M>::BYTES;  // fp32 MP x WS
    static constexpr size_t YT = W + MP * WS * 4;                      // Y^T (YtS layout)
    static constexpr size_t OUT = (YT + YtS<T, M>::bytes(NCOL) + 15) / 16 * 16;  // output rows, 64 x d
    static constexpr size_t DBG = OUT + 64 * DS * ES;                  // core dump: 2 M^2 + M NCOL floats
    static constexpr size_t BYTES = DBG + (2 * M * M + M * NCOL) * 4;
};

// Offsets (in floats) of the dump regions; the order and shapes are those
// nystra.h documents for nystra_debug_stages.
struct DumpOffsets {
    long long qbar, kbar, gl, mu, w, ga, z, y, out, total;
    __host__ __device__ DumpOffsets(int N, int d, int m) {
        qbar = 0;
        kbar = qbar + (long long)m * d;
        gl = kbar + (long long)m * d;
        mu = gl + (long long)N * m;
        w = mu + m;
        ga = w + (long long)m * (d + 1);
        z = ga + (long long)m * m;
        y = z + (long long)m * m;
        out = y + (long long)m * (d + 1);
        total = out + (long long)N * d;
    }
};

// RS: token order of the staged rows, as the product kernel takes it for
// this d_h (row_step of its compile-time width), so that the dumped output
// is the product kernel's bit for bit.
template <typename T, int M, int NCOL, int PW, int RS>
__global__ void __launch_bounds__(32, 1)
nystra_stage_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v, long long unit,
                    int d, int iters, float sl2, float* __restrict__ dump) {
    using P = StageLayout<T, M, NCOL>;
    constexpr int L = 64 / M;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    const int lane = threadIdx.x, g = lane >> 2, t = lane & 3;
    T* Qs = reinterpret_cast<T*>(smem_raw + P::QKV);
    T* Ks = Qs + 64 * d;
    T* Vs = Qs + 128 * d;
    T* qbar = reinterpret_cast<T*>(smem_raw + P::QB);
    T* kbar = reinterpret_cast<T*>(smem_raw + P::KB);
    uint32_t* glf = reinterpret_cast<uint32_t*>(smem_raw + P::GLF);
    float* mW = reinterpret_cast<float*>(smem_raw + P::W);
    T* yT = reinterpret_cast<T*>(smem_raw + P::YT);
    T* ob = reinterpret_cast<T*>(smem_raw + P::OUT);
    float* dbg = reinterpret_cast<float*>(smem_raw + P::DBG);
    const DumpOffsets off(64, d, M);

    const size_t base = (size_t)unit * 64 * d;
    for (int i = lane; i < 64 * d; i += 32) {
        Qs[i] = q[base + i];
        Ks[i] = k[base + i];
        Vs[i] = v[base + i];
    }
    __syncwarp();

    // step 1: landmarks
    landmarks_mma<T, 64, L, PW, RS>(Qs, qbar, 0, d, g, t);
    landmarks_mma<T, 64, L, PW, RS>(Ks, kbar, 0, d, g, t);
    if constexpr (M < P::MP) {
        landmarks_zero<T>(qbar, M, P::MP, lane, 32);
        landmarks_zero<T>(kbar, M, P::MP, lane, 32);
    }
    __syncwarp();
    for (int i = lane; i < M * d; i += 32) {
        dump[off.qbar + i] = lm_f32<T>(qbar + (i / d) * P::LS + i % d);
        dump[off.kbar + i] = lm_f32<T>(kbar + (i / d) * P::LS + i % d);
    }

    // steps 2-3: S_L, m_L, G_L^n (the operand registers of O = G_L^n Y)
#pragma unroll
    for (int tm = 0; tm < 4; ++tm) {
        typename Opnd<T>::DReg f[P::KTL][4];
        gl_tile<T, M, P::KTL, false, RS>(Qs + mtok<RS>(tm, g) * d, kbar, d, g, t, sl2, f);
#pragma unroll
        for (int kk = 0; kk < P::KTL; ++kk) {
            GlPark<T, M>::put(glf, (tm * P::KTL + kk) * 32 + lane, f[kk]);
#pragma unroll
            for (int r = 0; r < (M >= 16 ? 4 : 2); ++r) {
                const float2 x = reg_f2<T>(f[kk][r]);
                const int row = mtok<RS>(tm, g) + (r & 1) * mrow<RS>(), col = 16 * kk + 8 * (r >> 1) + 2 * t;
                dump[off.gl + row * M + col] = x.x;
                dump[off.gl + row * M + col + 1] = x.y;
            }
        }
    }

    // steps 2-3, 5: S_U, m_U, W = G_U^n [V | 1]
    float mU[1][2];
    front_su_w<T, M, NCOL, 1, false, RS>(qbar, Ks, Vs, d, g, t, sl2, mW, P::WS, mU);
    __syncwarp();
    if (t == 0) {  // m_U is kept in the log2 domain
        if (g < M) dump[off.mu + g] = mU[0][0] * 0.69314718055994531f;
        if (g + 8 < M) dump[off.mu + g + 8] = mU[0][1] * 0.69314718055994531f;
    }
    for (int i = lane; i < M * (d + 1); i += 32) dump[off.w + i] = mW[(i / (d + 1)) * P::WS + i % (d + 1)];

    // steps 3-4, 6: G_A^n, the pseudo-inverse iteration, Y = Z W
    core_warp<T, M, NCOL, true>(qbar, kbar, mU, mW, yT, iters, sl2, g, t, dbg);
    __syncwarp();
    for (int i = lane; i < M * M; i += 32) {
        dump[off.ga + i] = dbg[i];
        dump[off.z + i] = dbg[M * M + i];
    }
    for (int i = lane; i < M * (d + 1); i += 32) dump[off.y + i] = dbg[2 * M * M + (i / (d + 1)) * NCOL + i % (d + 1)];

    // step 7: O = (G_L^n Y_:d) / (G_L^n Y_d)
    output_rows<T, M, NCOL, 1, true, false, RS>(glf, Qs, kbar, yT, ob, d, g, t, lane, sl2);
    __syncwarp();
    for (int i = lane; i < 64 * d; i += 32) dump[off.out + i] = to_f32(ob[i]);
}

template <typename T, int M, int NCOL, int PW>
cudaError_t launch_stage(const void* q, const void* k, const void* v, long long unit, int d, int iters,
                         float* dump, cudaStream_t stream) {
    using P = StageLayout<T, M, NCOL>;
    // the product kernel compiles d_h = 30 in (row_step(30)); other widths keep token order
    auto kern = d == 30 ? nystra_stage_kernel<T, M, NCOL, PW, row_step(30)> : nystra_stage_kernel<T, M, NCOL, PW, 1>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)P::BYTES);
    if (e != cudaSuccess) return e;
    const float sl2 = 1.4426950408889634f / sqrtf((float)d);
    kern<<<1, 32, P::BYTES, stream>>>((const T*)q, (const T*)k, (const T*)v, unit, d, iters, sl2, dump);
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_stage_t(const void* q, const void* k, const void* v, long long unit, int d, int m, int iters,
                           int pool, float* dump, cudaStream_t stream) {
    const bool wide = d > 30;  // the ones column needs a fifth n-tile when d_h = 32
    if (pool != 0) {  // square patches: 16-bit I/O, m = 16, 2x2 patches of the 8x8 window
        if constexpr (sizeof(T) == 2)
            return wide ? launch_stage<T, 16, 40, 8>(q, k, v, unit, d, iters, dump, stream)
                        : launch_stage<T, 16, 32, 8>(q, k, v, unit, d, iters, dump, stream);
        return cudaErrorInvalidValue;  // not reached: checked by the caller
    }
    if (m == 8)
        return wide ? launch_stage<T, 8, 40, 0>(q, k, v, unit, d, iters, dump, stream)
                    : launch_stage<T, 8, 32, 0>(q, k, v, unit, d, iters, dump, stream);
    return wide ? launch_stage<T, 16, 40, 0>(q, k, v, unit, d, iters, dump, stream)
                : launch_stage<T, 16, 32, 0>(q, k, v, unit, d, iters, dump, stream);
}

}  // namespace
}  // namespace tc
}  // namespace nystra

namespace nystra_host {

long long debug_stages_size(int N, int d, int m) { return nystra::tc::DumpOffsets(N, d, m).total; }

cudaError_t launch_debug_stages(const void* q, const void* k, const void* v, long long unit, int d, int m,
                                int iters, int pool, int dtype, float* dump, cudaStream_t stream) {
    using namespace nystra::tc;
    if (dtype == 0) return launch_stage_t<float>(q, k, v, unit, d, m, iters, pool, dump, stream);
    if (dtype == 1) return launch_stage_t<__nv_bfloat16>(q, k, v, unit, d, m, iters, pool, dump, stream);
    return launch_stage_t<__half>(q, k, v, unit, d, m, iters, pool, dump, stream);
}

}  // namespace nystra_host
