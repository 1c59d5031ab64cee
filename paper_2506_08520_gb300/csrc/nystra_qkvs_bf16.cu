// Fused Q/K/V projection + PnP-Nystra for 16x16 and 32x32 windows, bf16 I/O;
// the kernels of nystra_qkv_stream.cuh.
#include "nystra_qkv_stream.cuh"

NYSTRA_QKVS_DEFINE(bf16, __nv_bfloat16)
