// Fused Q/K/V projection + PnP-Nystra for 8x8 windows, bf16 I/O (nystra_qkv.cuh).
#include "nystra_qkv.cuh"

namespace nystra_host {
cudaError_t launch_nystra_qkv_bf16(const void* x, const void* wqkv, const float* bqkv, void* out, long long n_windows,
                                 int heads, int d, int m, int iters, int pool, cudaStream_t stream,
                                 const nystra::NystraBias* bias) {
    return nystra::tc::launch_qkv<__nv_bfloat16>(x, wqkv, bqkv, out, n_windows, heads, d, m, iters, pool, stream, bias);
}
}  // namespace nystra_host
