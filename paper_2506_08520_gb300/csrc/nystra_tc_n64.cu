// Tensor-core PnP-Nystra kernels for windows of 64 tokens (see nystra_tc.cuh):
// each unit is handled by 1 warp(s) of 64 tokens.
#include "nystra_tc.cuh"

NYSTRA_TC_DEFINE(n64, 64, 1)
