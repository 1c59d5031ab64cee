// Tensor-core PnP-Nystra kernels for windows of 256 tokens: the team kernel
// (nystra_team.cuh) for m <= 16, the grouped kernel (nystra_tc.cuh, four
// warps of 64 tokens per unit) for m = 32.
#include "nystra_tc.cuh"
#include "nystra_team.cuh"

NYSTRA_TC_DEFINE(n256, 64, 4, __nv_bfloat16, __half, false)
