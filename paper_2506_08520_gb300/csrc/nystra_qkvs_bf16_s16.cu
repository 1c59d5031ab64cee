// Fused Q/K/V projection + PnP-Nystra for 16x16 and 32x32 windows, bf16 I/O, derived factors rounded to bf16
// (NYSTRA_FACTORS_16);
// the kernels of nystra_qkv_stream.cuh.
#include "nystra_qkv_stream.cuh"

NYSTRA_QKVS_DEFINE(bf16_s16, nystra::Single16<__nv_bfloat16>)
