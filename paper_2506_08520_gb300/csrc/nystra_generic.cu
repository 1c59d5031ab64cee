// Generic PnP-Nystra kernel: any N <= 1024, m | N with m <= 64, d_h <= 64.
//
// One CTA (256 threads) per (window, head) unit, all arithmetic in fp32 with
// correctly rounded expf.  Q, K and V are streamed from global memory in
// token chunks, so shared memory only holds the O(m^2 + m d) state:
//   pass 1  landmarks Qbar, Kbar (segment or square-patch means, Algorithm 1 step 1);
//   pass 2  K and V chunks: S_U = s Qbar K^T with a running row max m_U and
//           W = G_U^n [V | 1] accumulated with the usual online rescaling,
//           so that at the end W = exp(S_U - m_U) [V | 1] for the final m_U;
//   core    G_A^n = exp(s Qbar Kbar^T - m_U), the third-order iteration for
//           Z ~ (G_A^n)^+ (step 4), Y = Z W;
//   pass 3  Q chunks: G_L^n = exp(S_L - m_L) and O = (G_L^n Y_:d) / (G_L^n Y_d)
//           (steps 5-7, re-associated as G_L^n (Z (G_U^n [V | 1]))).
// This is the always-available path (and the fp32-exact one); shape-specialised
// tensor-core kernels take the common shapes.
#include "common.cuh"

namespace nystra {
namespace {

constexpr int kThreads = 256;
constexpr int kChunk = 32;  // tokens per streamed chunk

// C[r x c] = A[r x n] B[n x c], row-major, all in shared memory.
__device__ void block_matmul(const float* A, const float* B, float* C, int r, int n, int c) {
    for (int idx = threadIdx.x; idx < r * c; idx += blockDim.x) {
        const int i = idx / c, j = idx - (idx / c) * c;
        float acc = 0.f;
        for (int t = 0; t < n; ++t) acc = fmaf(A[i * n + t], B[t * c + j], acc);
        C[idx] = acc;
    }
}

// T = alpha I - X for an m x m matrix.
__device__ void shifted_identity_minus(const float* X, float* T, int m, float alpha) {
    for (int idx = threadIdx.x; idx < m * m; idx += blockDim.x) {
        const int i = idx / m, j = idx - (idx / m) * m;
        T[idx] = (i == j ? alpha : 0.f) - X[idx];
    }
}

__device__ float warp_max(float x) {
    for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
    return x;
}

template <typename T>
__global__ void __launch_bounds__(kThreads)
nystra_generic_kernel(const T* __restrict__ q, const T* __restrict__ k, const T* __restrict__ v,
                      T* __restrict__ out, long long n_units, int N, int d, int m, int iters,
                      int pw, float scale, NystraBias bias) {
    extern __shared__ float sm[];
    const int d1 = d + 1, L = N / m, tid = threadIdx.x;
    int pp = 0;  // patches per patch row (square-patch landmarks)
    if (pw > 0)
        while ((pp + 1) * (pp + 1) <= m) ++pp;
    float* qbar = sm;              // m*d
    float* kbar = qbar + m * d;    // m*d
    float* W = kbar + m * d;       // m*d1   G_U^n [V | 1]
    float* Y = W + m * d1;         // m*d1   Z W
    float* A = Y + m * d1;         // m*m    G_A^n
    float* Z = A + m * m;          // m*m
    float* X = Z + m * m;          // m*m
    float* T1 = X + m * m;         // m*m
    float* T2 = T1 + m * m;        // m*m
    float* mU = T2 + m * m;        // m
    float* rs = mU + m;            // m      rescale factors
    float* cb = rs + m;            // kChunk*d   K or Q chunk
    float* vb = cb + kChunk * d;   // kChunk*d   V chunk
    float* S = vb + kChunk * d;    // kChunk*m   scores of a chunk
    float* rowv = S + kChunk * m;  // kChunk     per-token max / denominator
    float* red = rowv + kChunk;    // 2          1/(||A||_1 ||A||_inf)

    for (long long u = blockIdx.x; u < n_units; u += gridDim.x) {
        const size_t base = (size_t)u * N * d;
        const T* qu = q + base;
        const T* ku = k + base;
        const T* vu = v + base;
        T* ou = out + base;
        // score bias through the landmarks (null without one): slice of this unit
        const long long bs = bias.per_window ? u : u % bias.heads;
        const float* bLu = bias.L ? bias.L + (size_t)bs * N * m : nullptr;
        const float* bUu = bias.U ? bias.U + (size_t)bs * m * N : nullptr;
        const float* bAu = bias.A ? bias.A + (size_t)bs * m * m : nullptr;

        // ---- pass 1: landmarks (Algorithm 1 step 1): segments of L tokens,
        // or (pw > 0) pb x pb patches of the pw-wide window, pb^2 = L ----
        for (int idx = tid; idx < m * d; idx += blockDim.x) {
            const int j = idx / d, c = idx - (idx / d) * d;
            float a = 0.f, b = 0.f;
            if (pw == 0) {
                for (int t = j * L; t < (j + 1) * L; ++t) {
                    a += ldg_f32(qu + (size_t)t * d + c);
                    b += ldg_f32(ku + (size_t)t * d + c);
                }
            } else {
                const int pb = pw / pp, r0 = (j / pp) * pb, s0 = (j % pp) * pb;
                for (int r = r0; r < r0 + pb; ++r)
                    for (int s = s0; s < s0 + pb; ++s) {
                        a += ldg_f32(qu + (size_t)(r * pw + s) * d + c);
                        b += ldg_f32(ku + (size_t)(r * pw + s) * d + c);
                    }
            }
            qbar[idx] = a / (float)L;
            kbar[idx] = b / (float)L;
        }
        for (int idx = tid; idx < m * d1; idx += blockDim.x) W[idx] = 0.f;
        for (int i = tid; i < m; i += blockDim.x) mU[i] = -INFINITY;
        __syncthreads();

        // ---- pass 2: S_U, running m_U, W = G_U^n [V | 1] ----
        for (int t0 = 0; t0 < N; t0 += kChunk) {
            const int nt = min(kChunk, N - t0);
            for (int idx = tid; idx < nt * d; idx += blockDim.x) {
                cb[idx] = ldg_f32(ku + (size_t)t0 * d + idx);
                vb[idx] = ldg_f32(vu + (size_t)t0 * d + idx);
            }
            __syncthreads();
            for (int idx = tid; idx < m * nt; idx += blockDim.x) {
                const int i = idx / nt, t = idx - (idx / nt) * nt;
                float a = 0.f;
                for (int c = 0; c < d; ++c) a = fmaf(qbar[i * d + c], cb[t * d + c], a);
                S[i * kChunk + t] = scale * a + (bUu ? __ldg(bUu + (size_t)i * N + t0 + t) : 0.f);
            }
            __syncthreads();
            for (int i = tid; i < m; i += blockDim.x) {
                float mx = mU[i];
                for (int t = 0; t < nt; ++t) mx = fmaxf(mx, S[i * kChunk + t]);
                rs[i] = (mU[i] == -INFINITY) ? 0.f : expf(mU[i] - mx);
                mU[i] = mx;
            }
            __syncthreads();
            for (int idx = tid; idx < m * nt; idx += blockDim.x) {
                const int i = idx / nt, t = idx - (idx / nt) * nt;
                S[i * kChunk + t] = expf(S[i * kChunk + t] - mU[i]);
            }
            __syncthreads();
            for (int idx = tid; idx < m * d1; idx += blockDim.x) {
                const int i = idx / d1, c = idx - (idx / d1) * d1;
                float acc = W[idx] * rs[i];
                if (c < d) {
                    for (int t = 0; t < nt; ++t) acc = fmaf(S[i * kChunk + t], vb[t * d + c], acc);
                } else {
                    for (int t = 0; t < nt; ++t) acc += S[i * kChunk + t];
                }
                W[idx] = acc;
            }
            __syncthreads();
        }

        // ---- core: G_A^n, pseudo-inverse iteration, Y = Z W ----
        for (int idx = tid; idx < m * m; idx += blockDim.x) {
            const int i = idx / m, j = idx - (idx / m) * m;
            float a = 0.f;
            for (int c = 0; c < d; ++c) a = fmaf(qbar[i * d + c], kbar[j * d + c], a);
            A[idx] = expf(scale * a + (bAu ? __ldg(bAu + idx) : 0.f) - mU[i]);
        }
        __syncthreads();
        if (tid < 32) {
            // ||A||_1 (max column sum) and ||A||_inf (max row sum); A > 0.
            float cmax = 0.f, rmax = 0.f;
            for (int j = tid; j < m; j += 32) {
                float cs = 0.f, rsum = 0.f;
                for (int i = 0; i < m; ++i) {
                    cs += A[i * m + j];
                    rsum += A[j * m + i];
                }
                cmax = fmaxf(cmax, cs);
                rmax = fmaxf(rmax, rsum);
            }
            cmax = warp_max(cmax);
            rmax = warp_max(rmax);
            if (tid == 0) red[0] = 1.f / (cmax * rmax);
        }
        __syncthreads();
        for (int idx = tid; idx < m * m; idx += blockDim.x) {
            const int i = idx / m, j = idx - (idx / m) * m;
            Z[idx] = red[0] * A[j * m + i];
        }
        __syncthreads();
        for (int it = 0; it < iters; ++it) {
            block_matmul(A, Z, X, m, m, m);          // X = A Z
            __syncthreads();
            shifted_identity_minus(X, T1, m, 7.f);   // 7I - X
            __syncthreads();
            block_matmul(X, T1, T2, m, m, m);
            __syncthreads();
            shifted_identity_minus(T2, T1, m, 15.f); // 15I - X(7I - X)
            __syncthreads();
            block_matmul(X, T1, T2, m, m, m);
            __syncthreads();
            shifted_identity_minus(T2, T1, m, 13.f); // 13I - X(15I - ...)
            __syncthreads();
            block_matmul(Z, T1, T2, m, m, m);
            __syncthreads();
            for (int idx = tid; idx < m * m; idx += blockDim.x) Z[idx] = 0.25f * T2[idx];
            __syncthreads();
        }
        block_matmul(Z, W, Y, m, m, d1);
        __syncthreads();

        // ---- pass 3: G_L^n and the normalised output ----
        for (int t0 = 0; t0 < N; t0 += kChunk) {
            const int nt = min(kChunk, N - t0);
            for (int idx = tid; idx < nt * d; idx += blockDim.x) cb[idx] = ldg_f32(qu + (size_t)t0 * d + idx);
            __syncthreads();
            for (int idx = tid; idx < nt * m; idx += blockDim.x) {
                const int t = idx / m, j = idx - (idx / m) * m;
                float a = 0.f;
                for (int c = 0; c < d; ++c) a = fmaf(cb[t * d + c], kbar[j * d + c], a);
                S[t * m + j] = scale * a + (bLu ? __ldg(bLu + (size_t)(t0 + t) * m + j) : 0.f);
            }
            __syncthreads();
            for (int t = tid; t < nt; t += blockDim.x) {
                float mx = -INFINITY;
                for (int j = 0; j < m; ++j) mx = fmaxf(mx, S[t * m + j]);
                rowv[t] = mx;
            }
            __syncthreads();
            for (int idx = tid; idx < nt * m; idx += blockDim.x) {
                const int t = idx / m;
                S[idx] = expf(S[idx] - rowv[t]);
            }
            __syncthreads();
            for (int t = tid; t < nt; t += blockDim.x) {
                float den = 0.f;
                for (int j = 0; j < m; ++j) den = fmaf(S[t * m + j], Y[j * d1 + d], den);
                rowv[t] = den;
            }
            __syncthreads();
            for (int idx = tid; idx < nt * d; idx += blockDim.x) {
                const int t = idx / d, c = idx - (idx / d) * d;
                float num = 0.f;
                for (int j = 0; j < m; ++j) num = fmaf(S[t * m + j], Y[j * d1 + c], num);
                ou[(size_t)(t0 + t) * d + c] = from_f32<T>(num / rowv[t]);
            }
            __syncthreads();
        }
    }
}

size_t generic_smem_bytes(int d, int m) {
    const int d1 = d + 1;
    const size_t floats = 2 * (size_t)m * d + 2 * (size_t)m * d1 + 5 * (size_t)m * m + 2 * (size_t)m +
                          2 * (size_t)kChunk * d + (size_t)kChunk * m + kChunk + 2;
    return floats * sizeof(float);
}

template <typename T>
cudaError_t launch_t(const void* q, const void* k, const void* v, void* out, long long n_units, int N,
                     int d, int m, int iters, int pool, const NystraBias& bias, cudaStream_t stream) {
    int pw = 0;  // window width for square patches
    if (pool != 0)
        while ((pw + 1) * (pw + 1) <= N) ++pw;
    const size_t smem = generic_smem_bytes(d, m);
    cudaError_t e = cudaFuncSetAttribute(nystra_generic_kernel<T>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const long long grid = n_units < (1LL << 30) ? n_units : (1LL << 30);
    nystra_generic_kernel<T><<<(unsigned)grid, kThreads, smem, stream>>>(
        (const T*)q, (const T*)k, (const T*)v, (T*)out, n_units, N, d, m, iters, pw, 1.0f / sqrtf((float)d),
        bias);
    return cudaGetLastError();
}

}  // namespace
}  // namespace nystra

namespace nystra_host {
cudaError_t launch_nystra_generic(const void* q, const void* k, const void* v, void* out,
                                  long long n_units, int N, int d, int m, int iters, int pool, int dtype,
                                  cudaStream_t stream, const nystra::NystraBias& bias) {
    using namespace nystra;
    switch (dtype) {
        case 0: return launch_t<float>(q, k, v, out, n_units, N, d, m, iters, pool, bias, stream);
        case 1: return launch_t<__nv_bfloat16>(q, k, v, out, n_units, N, d, m, iters, pool, bias, stream);
        default: return launch_t<__half>(q, k, v, out, n_units, N, d, m, iters, pool, bias, stream);
    }
}
}  // namespace nystra_host
