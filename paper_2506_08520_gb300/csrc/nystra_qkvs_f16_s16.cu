// Fused Q/K/V projection + PnP-Nystra for 16x16 and 32x32 windows, fp16 I/O, derived factors rounded to fp16
// (NYSTRA_FACTORS_16);
// the kernels of nystra_qkv_stream.cuh.
#include "nystra_qkv_stream.cuh"

NYSTRA_QKVS_DEFINE(f16_s16, nystra::Single16<__half>)
