// Fused Q/K/V projection + PnP-Nystra for 8x8 windows, bf16 I/O, derived
// factors rounded to bf16 (NYSTRA_FACTORS_16; nystra_qkv.cuh).
#include "nystra_qkv.cuh"

NYSTRA_QKV_DEFINE(bf16_s16, nystra::Single16<__nv_bfloat16>)
