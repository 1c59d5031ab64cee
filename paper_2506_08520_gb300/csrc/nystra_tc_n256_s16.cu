// The kernels of nystra_tc_n256.cu with the derived factors (landmarks,
// G_L^n, G_U^n, Y) rounded to the 16-bit I/O type: the faster arithmetic
// a caller selects with NYSTRA_FACTORS_16 (16-bit I/O only).
#include "nystra_tc.cuh"
#include "nystra_team.cuh"

NYSTRA_TC_DEFINE(n256_s16, 64, 4, nystra::Single16<__nv_bfloat16>, nystra::Single16<__half>, false)
