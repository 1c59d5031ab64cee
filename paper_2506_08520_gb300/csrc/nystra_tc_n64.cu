// Tensor-core PnP-Nystra kernels for windows of 64 tokens: the stage-pool
// kernel (nystra_pool.cuh) for m <= 16, the grouped kernel (nystra_tc.cuh,
// one warp per unit) for m = 32.
#include "nystra_tc.cuh"
#include "nystra_pool.cuh"

NYSTRA_TC_DEFINE(n64, 64, 1, __nv_bfloat16, __half, true)
