// Tensor-core PnP-Nystra kernels for windows of 1024 tokens: the streaming
// team kernel (nystra_stream.cuh) for m <= 16, the grouped kernel
// (nystra_tc.cuh) for m = 32 and 64.
#include "nystra_tc.cuh"
#include "nystra_stream.cuh"

NYSTRA_TC_DEFINE(n1024, 128, 8, __nv_bfloat16, __half, false)
