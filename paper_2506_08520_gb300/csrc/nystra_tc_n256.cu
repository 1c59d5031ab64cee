// Tensor-core PnP-Nystra kernels for windows of 256 tokens (see nystra_tc.cuh):
// each unit is handled by 4 warp(s) of 64 tokens.
#include "nystra_tc.cuh"

NYSTRA_TC_DEFINE(n256, 64, 4)
