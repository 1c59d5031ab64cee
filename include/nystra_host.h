/*
 * nystra_host.h -- C ABI of the multi-core CPU path of the PnP-Nystra
 * window-attention library (libnystra_host.so).
 *
 * The paper reports its method's speedup on CPUs as well as GPUs (abstract;
 * Table 2's CPU columns).  This is that path for the host cores: fp32, one
 * OpenMP thread per group of (window, head) units, loops laid out so the
 * compiler vectorises them over landmarks or features.  It is a separate
 * library with its own entry points: the GPU library never calls it, and it
 * never stands in for the GPU path.
 *
 * Conventions (as nystra.h, except for the memory space)
 *  Layout   q, k, v and out are contiguous row-major fp32 tensors of shape
 *           [n_windows, heads, N, d_h] in HOST memory owned by the caller;
 *           out must not overlap an input.
 *  Method   Algorithm 1 in the stabilised form of Sec. 2.2 (Eq. 8), evaluated
 *           per unit as G_L^n (Z (G_U^n [V | 1])) with the landmark pooling
 *           and pseudo-inverse iteration of nystra.h (segments or square
 *           patches; Z_0 = A^T/(||A||_1 ||A||_inf), `iters` third-order
 *           steps), all in fp32 (exponentials: nystra_host_exp's, within a
 *           few ulp of exp).
 *  Threads  `threads` OpenMP threads (<= 0: the OpenMP default, normally
 *           every core).  Each unit is computed by one thread in a fixed
 *           order, so results do not depend on the thread count.
 *  Errors   the status codes of nystra.h; invalid arguments are rejected
 *           before any work and leave `out` untouched.  Synchronous.
 */
#ifndef NYSTRA_HOST_H
#define NYSTRA_HOST_H

#include "nystra.h"

#ifdef __cplusplus
extern "C" {
#endif

/*
 * nystra_attention_host -- PnP-Nystra attention (Algorithm 1, Sec. 2.2) of
 * every unit on the host cores.  N in [1, NYSTRA_MAX_N], d_h in
 * [1, NYSTRA_MAX_DH], m in [1, min(N, NYSTRA_MAX_M)] dividing N, iters in
 * [0, NYSTRA_MAX_ITERS], landmarks a nystra_landmarks value (square patches:
 * N and m perfect squares whose roots divide); anything else, null
 * pointers and an out that overlaps an input return NYSTRA_EINVAL.
 * Returns NYSTRA_OK or NYSTRA_EINVAL.
 */
NYSTRA_API int nystra_attention_host(const float* q, const float* k, const float* v, float* out, int n_windows,
                                     int heads, int N, int d_h, int m, int iters, int landmarks, int threads);

/*
 * nystra_pool_bias_host -- the three landmark blocks of n_bias additive score
 * biases (the reading of nystra.h's nystra_pool_bias): bias [n_bias, N, N]
 * in, bias_L [n_bias, N, m], bias_U [n_bias, m, N], bias_A [n_bias, m, m]
 * out, all fp32 host memory, no overlaps; means over each landmark's tokens.
 * Returns NYSTRA_OK or NYSTRA_EINVAL.
 */
NYSTRA_API int nystra_pool_bias_host(const float* bias, int n_bias, int N, int m, int landmarks, float* bias_L,
                                     float* bias_U, float* bias_A, int threads);

/*
 * nystra_attention_bias_host -- nystra_attention_host with a pooled score
 * bias added to the scaled scores of S_L, S_U and S_A before their row
 * maxima (nystra.h, nystra_attention_bias).  bias_windows = 1: one slice per
 * head, shared by every window; = n_windows: one per (window, head) unit.
 * Returns NYSTRA_OK or NYSTRA_EINVAL (also for a bias that overlaps out).
 */
NYSTRA_API int nystra_attention_bias_host(const float* q, const float* k, const float* v, float* out,
                                          int n_windows, int heads, int N, int d_h, int m, int iters,
                                          int landmarks, const float* bias_L, const float* bias_U,
                                          const float* bias_A, int bias_windows, int threads);

/*
 * exact_window_attention_host -- exact softmax attention per unit, Eq. (1)
 * with row-max-shifted exponentials (Eq. 2), on the host cores: the CPU
 * computation PnP-Nystra replaces, for comparison.  Arguments and return
 * codes as nystra_attention_host (no m, iters, landmarks).
 */
NYSTRA_API int exact_window_attention_host(const float* q, const float* k, const float* v, float* out,
                                           int n_windows, int heads, int N, int d_h, int threads);

/*
 * nystra_host_exp -- test-only: y[i] = exp(x[i]) for i < n, by the
 * vectorisable exponential every entry point above uses for its softmax
 * blocks (Cody-Waite range reduction and a degree-7 Taylor polynomial;
 * arguments are taken as min(x, 88), results below exp(-104) are 0, NaN is
 * kept).  Host memory, no overlap checks, no return value.
 */
NYSTRA_API void nystra_host_exp(const float* x, float* y, int n);

/* Threads the host path uses when `threads` <= 0. */
NYSTRA_API int nystra_host_threads(void);

#ifdef __cplusplus
}
#endif
#endif /* NYSTRA_HOST_H */
