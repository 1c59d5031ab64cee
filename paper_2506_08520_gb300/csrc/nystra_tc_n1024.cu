// Tensor-core PnP-Nystra kernels for windows of 1024 tokens (see nystra_tc.cuh):
// each unit is handled by 8 warp(s) of 128 tokens.
#include "nystra_tc.cuh"

NYSTRA_TC_DEFINE(n1024, 128, 8)
