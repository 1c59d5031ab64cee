// Test-only kernel for the failure-detection path: one warp waits, through
// the kernels' bounded mbarrier wait, on an mbarrier that nothing arrives on,
// gives up after the given limit and records the timeout in its fault word.
#include "common.cuh"
#include "ptx.cuh"

namespace nystra {
__device__ unsigned int g_fault_debug;

__global__ void debug_wait_kernel(unsigned long long limit_ns, unsigned int* fault) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
    }
    __syncwarp();
    // Phase 0 never completes: no thread arrives and no copy is armed.
    const bool ok = __all_sync(0xffffffffu, mbar_wait_bounded(&bar, 0u, limit_ns));
    if (!ok && threadIdx.x == 0) atomicOr(fault, 1u);
}
}  // namespace nystra

namespace nystra_host {
cudaError_t launch_debug_wait(unsigned long long limit_ns, cudaStream_t stream) {
    static unsigned int* s_fault[64] = {};  // device address of the fault word, per device
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    if (!s_fault[dev]) {
        e = cudaGetSymbolAddress((void**)&s_fault[dev], nystra::g_fault_debug);
        if (e != cudaSuccess) return e;
    }
    nystra::debug_wait_kernel<<<1, 32, 0, stream>>>(limit_ns, s_fault[dev]);
    return cudaGetLastError();
}

unsigned int take_fault_word_debug(cudaError_t* err) {
    unsigned int w = 0, zero = 0;
    *err = cudaMemcpyFromSymbol(&w, nystra::g_fault_debug, sizeof(w));
    if (*err == cudaSuccess && w != 0) *err = cudaMemcpyToSymbol(nystra::g_fault_debug, &zero, sizeof(zero));
    return w;
}
}  // namespace nystra_host
