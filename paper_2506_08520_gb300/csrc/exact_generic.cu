// Generic exact window attention, Eq. (1): O = softmax(Q K^T / sqrt(d_h)) V.
//
// One CTA (256 threads) per (window, head) unit; one thread per query row.
// Keys and values are staged through shared memory in chunks of 32 tokens;
// each thread keeps its query row and output accumulator in registers and
// applies the online (running-max) form of the row softmax, which equals the
// max-shifted Eq. (2) up to rounding.  fp32 arithmetic, correctly rounded expf.
// Always available for any N <= 1024 and d_h <= 64.
#include "common.cuh"

namespace nystra {
namespace {

constexpr int kThreads = 256;
constexpr int kChunk = 32;

template <typename T, int DMAX>
__global__ void __launch_bounds__(kThreads)
exact_generic_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                     T* __restrict__ out, long long n_units, int N, int d, float scale) {
    __shared__ float kb[kChunk * DMAX];
    __shared__ float vb[kChunk * DMAX];
    __shared__ float sc[kChunk * kThreads];
    const int tid = threadIdx.x;
    for (long long u = blockIdx.x; u < n_units; u += gridDim.x) {
        const size_t base = (size_t)u * N * d;
        for (int r0 = 0; r0 < N; r0 += kThreads) {
            const int row = r0 + tid;
            const bool active = row < N;
            float qr[DMAX], acc[DMAX];
#pragma unroll
            for (int c = 0; c < DMAX; ++c) {
                qr[c] = (active && c < d) ? scale * ldg_f32(q + base + (size_t)row * d + c) : 0.f;
                acc[c] = 0.f;
            }
            float mx = -INFINITY, den = 0.f;
            for (int t0 = 0; t0 < N; t0 += kChunk) {
                const int nt = min(kChunk, N - t0);
                __syncthreads();
                for (int idx = tid; idx < nt * d; idx += blockDim.x) {
                    const int t = idx / d, c = idx - (idx / d) * d;
                    kb[t * DMAX + c] = ldg_f32(k + base + (size_t)t0 * d + idx);
                    vb[t * DMAX + c] = ldg_f32(v + base + (size_t)t0 * d + idx);
                }
                __syncthreads();
                if (!active) continue;
                // this thread's scores for the chunk, kept in shared memory
                float* s = sc + tid;
                float cmx = -INFINITY;
#pragma unroll 2
                for (int t = 0; t < nt; ++t) {
                    float a = 0.f;
#pragma unroll
                    for (int c = 0; c < DMAX; ++c)
                        if (c < d) a = fmaf(qr[c], kb[t * DMAX + c], a);
                    s[t * kThreads] = a;
                    cmx = fmaxf(cmx, a);
                }
                const float nmx = fmaxf(mx, cmx);
                const float r = (mx == -INFINITY) ? 0.f : expf(mx - nmx);
                den *= r;
#pragma unroll
                for (int c = 0; c < DMAX; ++c) acc[c] *= r;
                mx = nmx;
#pragma unroll 2
                for (int t = 0; t < nt; ++t) {
                    const float p = expf(s[t * kThreads] - mx);
                    den += p;
#pragma unroll
                    for (int c = 0; c < DMAX; ++c)
                        if (c < d) acc[c] = fmaf(p, vb[t * DMAX + c], acc[c]);
                }
            }
            if (active) {
                const float inv = 1.f / den;
#pragma unroll
                for (int c = 0; c < DMAX; ++c)
                    if (c < d) out[base + (size_t)row * d + c] = from_f32<T>(acc[c] * inv);
            }
        }
    }
}

template <typename T>
cudaError_t launch_t(const void* q, const void* k, const void* v, void* out, long long n_units, int N,
                     int d, cudaStream_t stream) {
    const long long grid = n_units < (1LL << 30) ? n_units : (1LL << 30);
    const float scale = 1.0f / sqrtf((float)d);
    if (d <= 32)
        exact_generic_kernel<T, 32><<<(unsigned)grid, kThreads, 0, stream>>>(
            (const T*)q, (const T*)k, (const T*)v, (T*)out, n_units, N, d, scale);
    else
        exact_generic_kernel<T, 64><<<(unsigned)grid, kThreads, 0, stream>>>(
            (const T*)q, (const T*)k, (const T*)v, (T*)out, n_units, N, d, scale);
    return cudaGetLastError();
}

}  // namespace
}  // namespace nystra

namespace nystra_host {
cudaError_t launch_exact_generic(const void* q, const void* k, const void* v, void* out,
                                 long long n_units, int N, int d, int dtype, cudaStream_t stream) {
    using namespace nystra;
    switch (dtype) {
        case 0: return launch_t<float>(q, k, v, out, n_units, N, d, stream);
        case 1: return launch_t<__nv_bfloat16>(q, k, v, out, n_units, N, d, stream);
        default: return launch_t<__half>(q, k, v, out, n_units, N, d, stream);
    }
}
}  // namespace nystra_host
