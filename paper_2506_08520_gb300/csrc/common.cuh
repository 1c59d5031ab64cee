// Shared device helpers for the PnP-Nystra kernels (sm_103a).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

namespace nystra {

// Element I/O: 16-bit inputs are widened exactly; outputs are rounded to
// nearest-even.
__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }
__device__ __forceinline__ float to_f32(__half x) { return __half2float(x); }

template <typename T> __device__ __forceinline__ T from_f32(float x);
template <> __device__ __forceinline__ float from_f32<float>(float x) { return x; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
    return __float2bfloat16_rn(x);
}
template <> __device__ __forceinline__ __half from_f32<__half>(float x) { return __float2half_rn(x); }

// 16-bit I/O whose derived factors (landmarks, G_L^n, G_U^n, Y) are rounded
// to that 16-bit type instead of being carried as hi + lo pairs: the faster,
// less accurate arithmetic a caller selects with NYSTRA_FACTORS_16.  Same
// size and bits as T; only the kernels' operand policies differ (Opnd).
template <typename T>
struct Single16 {
    T v;
};
__device__ __forceinline__ float to_f32(Single16<__nv_bfloat16> x) { return __bfloat162float(x.v); }
__device__ __forceinline__ float to_f32(Single16<__half> x) { return __half2float(x.v); }
template <> __device__ __forceinline__ Single16<__nv_bfloat16> from_f32<Single16<__nv_bfloat16>>(float x) {
    return {__float2bfloat16_rn(x)};
}
template <> __device__ __forceinline__ Single16<__half> from_f32<Single16<__half>>(float x) {
    return {__float2half_rn(x)};
}

template <typename T> __device__ __forceinline__ float ldg_f32(const T* p) { return to_f32(p[0]); }
template <> __device__ __forceinline__ float ldg_f32<float>(const float* p) { return __ldg(p); }

// An additive score bias seen through the landmarks (null pointers: none):
// per slice, L is N x m, U is m x N and A is m x m (fp32, row-major).  Unit
// u = window * heads + head uses slice u (per_window) or u % heads.
struct NystraBias {
    const float* L = nullptr;
    const float* U = nullptr;
    const float* A = nullptr;
    int heads = 1;
    int per_window = 0;
};

// Persistent grid size of `kern` on the current device: SMs x CTAs resident
// at `smem` bytes of dynamic shared memory, after opting the kernel in to that
// much.  Both are per device, so both are cached per device ordinal in
// `cache` (a zero-initialised static of the launcher).
constexpr int kMaxDevices = 64;
template <typename K>
cudaError_t persistent_grid(K kern, int threads, size_t smem, std::atomic<int> (&cache)[kMaxDevices], int* blocks) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    int b = cache[dev].load(std::memory_order_relaxed);
    if (b == 0) {
        if ((e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
            return e;
        int sms = 0, per_sm = 0;
        if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
        if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem)) != cudaSuccess) return e;
        if (per_sm < 1) return cudaErrorInvalidConfiguration;
        b = sms * per_sm;
        cache[dev].store(b, std::memory_order_relaxed);
    }
    *blocks = b;
    return cudaSuccess;
}

}  // namespace nystra

// Host-side launchers (one per kernel family), defined in their .cu files.
// Each returns a cudaError_t of the launch.
namespace nystra_host {
// pool: landmark pooling, 0 = segments, 1 = square patches of a square window.
cudaError_t launch_nystra_generic(const void* q, const void* k, const void* v, void* out,
                                  long long n_units, int N, int d, int m, int iters, int pool, int dtype,
                                  cudaStream_t stream, const nystra::NystraBias& bias = {});
// Pools bias [n_bias, N, N] into its landmark blocks (bias.cu).
cudaError_t launch_pool_bias(const float* bias, long long n_bias, int N, int m, int pool, float* bias_L,
                             float* bias_U, float* bias_A, cudaStream_t stream);
cudaError_t launch_exact_generic(const void* q, const void* k, const void* v, void* out,
                                 long long n_units, int N, int d, int dtype, cudaStream_t stream);
// Tensor-core kernels, windows of 64 / 256 / 1024 tokens (nystra_tc_n*.cu):
// 16-bit I/O with m in {8, 16, 32, 64}, fp32 I/O at N = 64 with m in {8, 16};
// even d_h <= 32.  Square-patch landmarks (pool = 1): 16-bit I/O, m = 16.  A
// score bias (bias != nullptr): m in {8, 16}.
cudaError_t launch_nystra_tc_n64(const void* q, const void* k, const void* v, void* out, long long n_units,
                                 int d, int m, int iters, int pool, int dtype, cudaStream_t stream,
                                 const nystra::NystraBias* bias = nullptr);
cudaError_t launch_nystra_tc_n256(const void* q, const void* k, const void* v, void* out, long long n_units,
                                  int d, int m, int iters, int pool, int dtype, cudaStream_t stream,
                                 const nystra::NystraBias* bias = nullptr);
cudaError_t launch_nystra_tc_n1024(const void* q, const void* k, const void* v, void* out, long long n_units,
                                   int d, int m, int iters, int pool, int dtype, cudaStream_t stream,
                                 const nystra::NystraBias* bias = nullptr);
// The same with the derived factors rounded to 16 bits (Single16; 16-bit I/O
// only, nystra_tc_n*_s16.cu).
cudaError_t launch_nystra_tc_n64_s16(const void* q, const void* k, const void* v, void* out, long long n_units,
                                     int d, int m, int iters, int pool, int dtype, cudaStream_t stream,
                                     const nystra::NystraBias* bias = nullptr);
cudaError_t launch_nystra_tc_n256_s16(const void* q, const void* k, const void* v, void* out, long long n_units,
                                      int d, int m, int iters, int pool, int dtype, cudaStream_t stream,
                                      const nystra::NystraBias* bias = nullptr);
cudaError_t launch_nystra_tc_n1024_s16(const void* q, const void* k, const void* v, void* out, long long n_units,
                                       int d, int m, int iters, int pool, int dtype, cudaStream_t stream,
                                       const nystra::NystraBias* bias = nullptr);
unsigned int take_fault_word_tc_n64(cudaError_t* err);
unsigned int take_fault_word_tc_n256(cudaError_t* err);
unsigned int take_fault_word_tc_n1024(cudaError_t* err);
unsigned int take_fault_word_tc_n64_s16(cudaError_t* err);
unsigned int take_fault_word_tc_n256_s16(cudaError_t* err);
unsigned int take_fault_word_tc_n1024_s16(cudaError_t* err);
// Tensor-core exact attention, 16-bit I/O, N in {64, 256, 1024}, even d_h <= 32 (exact_tc.cu).
bool exact_tc_supports(int N, int d, int dtype);
cudaError_t launch_exact_tc(const void* q, const void* k, const void* v, void* out, long long n_units, int N,
                            int d, int dtype, cudaStream_t stream);
unsigned int take_fault_word_exact_tc(cudaError_t* err);
// Device-side fault words (bit 0: a bounded wait gave up) of the translation
// units whose kernels wait on barriers: OR-ed together, then cleared.
unsigned int take_fault_words(cudaStream_t stream, cudaError_t* err);
cudaError_t launch_debug_wait(unsigned long long limit_ns, cudaStream_t stream);
// Fused Q/K/V projection + PnP-Nystra, 8x8 windows, m in {8, 16} (square
// patches: m = 16), even d_h <= 32, heads * d_h <= 352 (nystra_qkv_*.cu).
cudaError_t launch_nystra_qkv_bf16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                   long long n_windows, int heads, int d, int m, int iters, int pool,
                                   cudaStream_t stream, const nystra::NystraBias* bias);
cudaError_t launch_nystra_qkv_f16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                  long long n_windows, int heads, int d, int m, int iters, int pool,
                                  cudaStream_t stream, const nystra::NystraBias* bias);
cudaError_t launch_nystra_qkv_bf16_s16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                       long long n_windows, int heads, int d, int m, int iters, int pool,
                                       cudaStream_t stream, const nystra::NystraBias* bias);
cudaError_t launch_nystra_qkv_f16_s16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                      long long n_windows, int heads, int d, int m, int iters, int pool,
                                      cudaStream_t stream, const nystra::NystraBias* bias);
// Fused Q/K/V projection + PnP-Nystra for N = 256 or 1024 (nystra_qkvs_*.cu).
cudaError_t launch_nystra_qkvs_bf16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                    long long n_windows, int heads, int N, int d, int m, int iters, int pool,
                                    cudaStream_t stream, const nystra::NystraBias* bias);
cudaError_t launch_nystra_qkvs_f16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                   long long n_windows, int heads, int N, int d, int m, int iters, int pool,
                                   cudaStream_t stream, const nystra::NystraBias* bias);
cudaError_t launch_nystra_qkvs_bf16_s16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                        long long n_windows, int heads, int N, int d, int m, int iters, int pool,
                                        cudaStream_t stream, const nystra::NystraBias* bias);
cudaError_t launch_nystra_qkvs_f16_s16(const void* x, const void* wqkv, const float* bqkv, void* out,
                                       long long n_windows, int heads, int N, int d, int m, int iters, int pool,
                                       cudaStream_t stream, const nystra::NystraBias* bias);
unsigned int take_fault_word_qkvs_bf16(cudaError_t* err);
unsigned int take_fault_word_qkvs_f16(cudaError_t* err);
unsigned int take_fault_word_qkvs_bf16_s16(cudaError_t* err);
unsigned int take_fault_word_qkvs_f16_s16(cudaError_t* err);
unsigned int take_fault_word_qkv_bf16(cudaError_t* err);
unsigned int take_fault_word_qkv_f16(cudaError_t* err);
unsigned int take_fault_word_qkv_bf16_s16(cudaError_t* err);
unsigned int take_fault_word_qkv_f16_s16(cudaError_t* err);
// Q/K/V projection with the head split on the fifth-generation tensor cores
// (project_qkv.cu): x [n_windows * N, heads * d] -> q, k, v [n_windows, heads, N, d].
cudaError_t launch_project_qkv(const void* x, const void* w, const float* b, void* q, void* k, void* v,
                               long long n_windows, int heads, int N, int d, int dtype, cudaStream_t stream);
unsigned int take_fault_word_proj(cudaError_t* err);
// Test-only stage dump of the 8x8-window tensor-core path (debug_stages.cu).
long long debug_stages_size(int N, int d, int m);
cudaError_t launch_debug_stages(const void* q, const void* k, const void* v, long long unit, int d, int m,
                                int iters, int pool, int dtype, float* dump, cudaStream_t stream);
unsigned int take_fault_word_debug(cudaError_t* err);
}  // namespace nystra_host
