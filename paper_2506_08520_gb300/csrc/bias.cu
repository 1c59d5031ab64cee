// An additive score bias (window attention's relative-position bias and
// masks) seen through the landmarks: every entry of a landmark block is the
// mean of the bias over the tokens the landmark averages, as the landmark
// itself is the mean of those tokens (Algorithm 1 step 1):
//   L[i][j] = mean_{t in j} B[i][t]   (N x m)
//   U[j][t] = mean_{s in j} B[s][t]   (m x N)
//   A[i][j] = mean_{s in i, t in j} B[s][t]   (m x m)
// Runs once per model constant, so a plain SIMT kernel suffices.
#include "common.cuh"

namespace nystra {
namespace {

// The l-th token of landmark j: segments of L tokens (pw = 0) or b x b
// patches of the pw-wide window (pp patches per row).
__device__ __forceinline__ int token_of(int j, int l, int L, int pw, int pp) {
    if (pw == 0) return j * L + l;
    const int b = pw / pp;
    return ((j / pp) * b + l / b) * pw + (j % pp) * b + l % b;
}

__global__ void pool_bias_kernel(const float* __restrict__ B, long long n_bias, int N, int m, int pw, int pp,
                                 float* __restrict__ bL, float* __restrict__ bU, float* __restrict__ bA) {
    const int L = N / m;
    const long long per = 2LL * N * m + (long long)m * m;  // outputs per slice
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < n_bias * per;
         idx += (long long)gridDim.x * blockDim.x) {
        const long long n = idx / per;
        const int e = (int)(idx - n * per);
        const float* Bn = B + (size_t)n * N * N;
        float acc = 0.f;
        if (e < N * m) {  // L[i][j]
            const int i = e / m, j = e % m;
            for (int l = 0; l < L; ++l) acc += Bn[(size_t)i * N + token_of(j, l, L, pw, pp)];
            bL[(size_t)n * N * m + e] = acc / (float)L;
        } else if (e < 2 * N * m) {  // U[j][t]
            const int f = e - N * m, j = f / N, t = f % N;
            for (int l = 0; l < L; ++l) acc += Bn[(size_t)token_of(j, l, L, pw, pp) * N + t];
            bU[(size_t)n * m * N + f] = acc / (float)L;
        } else {  // A[i][j]
            const int f = e - 2 * N * m, i = f / m, j = f % m;
            for (int a = 0; a < L; ++a) {
                const int s = token_of(i, a, L, pw, pp);
                for (int b = 0; b < L; ++b) acc += Bn[(size_t)s * N + token_of(j, b, L, pw, pp)];
            }
            bA[(size_t)n * m * m + f] = acc / ((float)L * (float)L);
        }
    }
}

}  // namespace
}  // namespace nystra

namespace nystra_host {
cudaError_t launch_pool_bias(const float* bias, long long n_bias, int N, int m, int pool, float* bias_L,
                             float* bias_U, float* bias_A, cudaStream_t stream) {
    int pw = 0, pp = 0;
    if (pool != 0) {
        while ((pw + 1) * (pw + 1) <= N) ++pw;
        while ((pp + 1) * (pp + 1) <= m) ++pp;
    }
    const long long total = n_bias * (2LL * N * m + (long long)m * m);
    const long long blocks = (total + 255) / 256;
    nystra::pool_bias_kernel<<<(unsigned)(blocks < 65536 ? blocks : 65536), 256, 0, stream>>>(
        bias, n_bias, N, m, pw, pp, bias_L, bias_U, bias_A);
    return cudaGetLastError();
}
}  // namespace nystra_host
