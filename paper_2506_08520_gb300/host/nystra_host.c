/*
 * Multi-core CPU path of PnP-Nystra window attention (fp32), declared in
 * include/nystra_host.h.
 *
 * Per (window, head) unit, Algorithm 1 in the stabilised form of Sec. 2.2,
 * evaluated as G_L^n (Z (G_U^n [V | 1])):
 *   1. landmarks Qbar, Kbar: means of the m segments of N/m tokens (or of
 *      the square patches of the window);
 *   2. S_U = s Qbar K^T (kept transposed, N x m) with the row maxima m_U over
 *      all N keys; G_U^n = exp(S_U - m_U); W = G_U^n [V | 1] (m x (d+1));
 *   3. A = G_A^n = exp(s Qbar Kbar^T - m_U);
 *   4. Z_0 = A^T / (||A||_1 ||A||_inf), then `iters` steps
 *      Z <- Z (13 I - X (15 I - X (7 I - X))) / 4 with X = A Z;
 *   5. Y = Z W;
 *   6. per token i: S_L = s q_i Kbar^T, G_L^n = exp(S_L - max), and
 *      o_i = (G_L^n Y_:d) / (G_L^n Y_d).
 * s = 1/sqrt(d).  Every inner loop runs over a contiguous landmark or feature
 * index with no reduction carried along it (dot products accumulate one
 * input dimension per pass over a vector of outputs), so -O3 vectorises it
 * for the host's SIMD unit without reassociating any sum.  Units are spread
 * over OpenMP threads; each unit runs on one thread in a fixed order.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#include "nystra_host.h"

enum { MAXN = NYSTRA_MAX_N, MAXD = NYSTRA_MAX_DH, MAXM = NYSTRA_MAX_M, NBLK = 64, MAXDP = 80 };

static int isqrt_exact(int n) {
    int r = 0;
    while ((r + 1) * (r + 1) <= n) ++r;
    return r * r == n ? r : -1;
}

static int overlaps(const void* a, const void* b, size_t bytes) {
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return x < y + bytes && y < x + bytes;
}

/* exp(x) for x <= 88, written so that a loop of calls vectorises (glibc's
 * scalar expf does not).  Cody-Waite range reduction (W. J. Cody and W. Waite,
 * Software Manual for the Elementary Functions, 1980): x = k ln 2 + r with k
 * the nearest integer to x / ln 2, so |r| <= ln 2 / 2, and ln 2 split into a
 * 9-bit part whose products with k are exact plus a correction.  exp(r) is
 * its Taylor series to degree 7 (truncation below 1e-8 relative) in Horner
 * form, and 2^k is applied as two exact powers of two, so results in the
 * subnormal range round once.  Arguments below -104 give 0 (exp(-104) is
 * below half the smallest subnormal); a NaN is returned as it is.  Max error
 * a few ulp (tested against float64 exp). */
static inline float exp_cw(float x) {
    const float xc = x > -104.f ? (x < 88.f ? x : 88.f) : -104.f;
    const float shifter = 12582912.f;  /* 1.5 * 2^23: adding it rounds to an integer */
    const float kf = (xc * 1.44269504088896341f + shifter) - shifter;
    const float r = (xc - kf * 0.693359375f) - kf * -2.12194440054690583e-4f;
    float p = 1.f / 5040.f;
    p = p * r + 1.f / 720.f;
    p = p * r + 1.f / 120.f;
    p = p * r + 1.f / 24.f;
    p = p * r + 1.f / 6.f;
    p = p * r + 0.5f;
    p = p * r + 1.f;
    p = p * r + 1.f;
    const int32_t k = (int32_t)kf, k1 = k / 2, k2 = k - k1;  /* both in [-75, 64] */
    union { int32_t i; float f; } s1, s2;
    s1.i = (k1 + 127) * (1 << 23);
    s2.i = (k2 + 127) * (1 << 23);
    const float y = p * s1.f * s2.f;
    return x == x ? y : x;
}

/* max(x[0..n)) (NaNs skipped), as eight running maxima compared elementwise:
 * the loop vectorises, and the maximum does not depend on the order. */
static inline float row_max(const float* x, int n) {
    float acc[8];
    for (int b = 0; b < 8; ++b) acc[b] = -INFINITY;
    int j = 0;
    for (; j + 8 <= n; j += 8)
        for (int b = 0; b < 8; ++b) acc[b] = x[j + b] > acc[b] ? x[j + b] : acc[b];
    float mx = acc[0];
    for (int b = 1; b < 8; ++b) mx = acc[b] > mx ? acc[b] : mx;
    for (; j < n; ++j) mx = x[j] > mx ? x[j] : mx;
    return mx;
}

void nystra_host_exp(const float* x, float* y, int n) {
    if (!x || !y) return;
    for (int i = 0; i < n; ++i) y[i] = exp_cw(x[i]);
}

/* Per-thread scratch of one unit. */
typedef struct {
    float qbar[MAXM * MAXD], kbar[MAXM * MAXD];
    float qbarT[MAXD * MAXM], kbarT[MAXD * MAXM], kbarTs[MAXD * MAXM];  /* qbar: scaled by s */
    float st[MAXN * MAXM];            /* S_U^T, then G_U^n transposed (N x m) */
    float vp[MAXN * MAXDP];           /* [V | 1 | 0]: d + 1 columns padded to DP, a multiple of 16 */
    float w[MAXM * MAXDP];            /* W = G_U^n [V | 1] (padded columns: zero) */
    float a[MAXM * MAXM], z[MAXM * MAXM], x[MAXM * MAXM], t1[MAXM * MAXM], t2[MAXM * MAXM];
    float y[MAXM * MAXDP];            /* Y = Z W */
    float mu[MAXM];
    float num[NBLK * MAXDP];          /* G_L^n Y for a block of tokens */
    int seg[MAXN];                    /* landmark of each token */
} Scratch;

/* C[r x c] = A[r x n] B[n x c] (row-major), inner loop over c. */
static void mm(const float* A, const float* B, float* C, int r, int n, int c) {
    for (int i = 0; i < r; ++i) {
        float* ci = C + (size_t)i * c;
        for (int j = 0; j < c; ++j) ci[j] = 0.f;
        for (int l = 0; l < n; ++l) {
            const float av = A[(size_t)i * n + l];
            const float* bl = B + (size_t)l * c;
            for (int j = 0; j < c; ++j) ci[j] += av * bl[j];
        }
    }
}

/* C[r x c] (+)= A[r x n] B[n x c], all row-major with leading dimensions
 * lda, ldb, ldc: blocks of 4 rows x 16 columns of C accumulate in registers
 * over n (the 16 columns are one vector loop), remainders element by element. */
static void gemm_nn(const float* A, int lda, const float* B, int ldb, float* C, int ldc, int r, int n, int c,
                    int accumulate) {
    int i = 0;
    for (; i + 4 <= r; i += 4) {
        int j = 0;
        for (; j + 16 <= c; j += 16) {
            float acc[4][16];
            for (int a = 0; a < 4; ++a)
                for (int b = 0; b < 16; ++b) acc[a][b] = accumulate ? C[(size_t)(i + a) * ldc + j + b] : 0.f;
            for (int l = 0; l < n; ++l) {
                const float* bl = B + (size_t)l * ldb + j;
                const float a0 = A[(size_t)i * lda + l], a1 = A[(size_t)(i + 1) * lda + l];
                const float a2 = A[(size_t)(i + 2) * lda + l], a3 = A[(size_t)(i + 3) * lda + l];
                for (int b = 0; b < 16; ++b) {
                    acc[0][b] += a0 * bl[b];
                    acc[1][b] += a1 * bl[b];
                    acc[2][b] += a2 * bl[b];
                    acc[3][b] += a3 * bl[b];
                }
            }
            for (int a = 0; a < 4; ++a)
                for (int b = 0; b < 16; ++b) C[(size_t)(i + a) * ldc + j + b] = acc[a][b];
        }
        for (; j < c; ++j)
            for (int a = 0; a < 4; ++a) {
                float acc = accumulate ? C[(size_t)(i + a) * ldc + j] : 0.f;
                for (int l = 0; l < n; ++l) acc += A[(size_t)(i + a) * lda + l] * B[(size_t)l * ldb + j];
                C[(size_t)(i + a) * ldc + j] = acc;
            }
    }
    for (; i < r; ++i)
        for (int j = 0; j < c; ++j) {
            float acc = accumulate ? C[(size_t)i * ldc + j] : 0.f;
            for (int l = 0; l < n; ++l) acc += A[(size_t)i * lda + l] * B[(size_t)l * ldb + j];
            C[(size_t)i * ldc + j] = acc;
        }
}

/* C[r x c] = A^T B with A [n x r] and B [n x c] row-major (leading
 * dimensions lda, ldb; C dense): 4 x 16 register blocks accumulated over n. */
static void gemm_tn(const float* A, int lda, const float* B, int ldb, float* C, int r, int n, int c) {
    int i = 0;
    for (; i + 4 <= r; i += 4) {
        int j = 0;
        for (; j + 16 <= c; j += 16) {
            float acc[4][16];
            for (int a = 0; a < 4; ++a)
                for (int b = 0; b < 16; ++b) acc[a][b] = 0.f;
            for (int l = 0; l < n; ++l) {
                const float* al = A + (size_t)l * lda + i;
                const float* bl = B + (size_t)l * ldb + j;
                for (int b = 0; b < 16; ++b) {
                    acc[0][b] += al[0] * bl[b];
                    acc[1][b] += al[1] * bl[b];
                    acc[2][b] += al[2] * bl[b];
                    acc[3][b] += al[3] * bl[b];
                }
            }
            for (int a = 0; a < 4; ++a)
                for (int b = 0; b < 16; ++b) C[(size_t)(i + a) * c + j + b] = acc[a][b];
        }
        for (; j < c; ++j)
            for (int a = 0; a < 4; ++a) {
                float acc = 0.f;
                for (int l = 0; l < n; ++l) acc += A[(size_t)l * lda + i + a] * B[(size_t)l * ldb + j];
                C[(size_t)(i + a) * c + j] = acc;
            }
    }
    for (; i < r; ++i)
        for (int j = 0; j < c; ++j) {
            float acc = 0.f;
            for (int l = 0; l < n; ++l) acc += A[(size_t)l * lda + i] * B[(size_t)l * ldb + j];
            C[(size_t)i * c + j] = acc;
        }
}

/* One unit.  bL, bU, bA: its pooled score-bias blocks (N x m, m x N, m x m;
 * all null: no bias), added to the scaled scores before the row maxima. */
static void one_unit(const float* Q, const float* K, const float* V, float* O, int N, int d, int m, int iters,
                     const float* bL, const float* bU, const float* bA, Scratch* S) {
    const float s = 1.0f / sqrtf((float)d);
    const int dp = (d + 1 + 15) / 16 * 16;  /* columns of [V | 1] padded for full register blocks */
    /* 1. landmarks: sums over each landmark's tokens, then the mean */
    memset(S->qbar, 0, sizeof(float) * (size_t)m * d);
    memset(S->kbar, 0, sizeof(float) * (size_t)m * d);
    int cnt[MAXM];
    for (int j = 0; j < m; ++j) cnt[j] = 0;
    for (int t = 0; t < N; ++t) {
        const int j = S->seg[t];
        ++cnt[j];
        float* qb = S->qbar + (size_t)j * d;
        float* kb = S->kbar + (size_t)j * d;
        const float* qt = Q + (size_t)t * d;
        const float* kt = K + (size_t)t * d;
        for (int c = 0; c < d; ++c) {
            qb[c] += qt[c];
            kb[c] += kt[c];
        }
    }
    /* the means; s is folded into Qbar (the scores of S_U and A) and into a
     * copy of Kbar^T (the scores of S_L), so no pass scales a score block */
    for (int j = 0; j < m; ++j) {
        const float inv = 1.0f / (float)cnt[j];
        for (int c = 0; c < d; ++c) {
            S->qbar[(size_t)j * d + c] *= inv;
            S->kbar[(size_t)j * d + c] *= inv;
            S->qbar[(size_t)j * d + c] *= s;
            S->qbarT[(size_t)c * m + j] = S->qbar[(size_t)j * d + c];
            S->kbarT[(size_t)c * m + j] = S->kbar[(size_t)j * d + c];
            S->kbarTs[(size_t)c * m + j] = S->kbar[(size_t)j * d + c] * s;
        }
    }
    /* 2. S_U^T = K (s Qbar)^T (N x m), the maxima over all N keys,
     *    G_U^n, and W = G_U^n [V | 1] (the ones column: the row sums) */
    gemm_nn(K, d, S->qbarT, m, S->st, m, N, d, m, 0);
    for (int i = 0; i < m; ++i) S->mu[i] = -INFINITY;
    for (int t = 0; t < N; ++t) {
        float* row = S->st + (size_t)t * m;
        if (bU)
            for (int i = 0; i < m; ++i) row[i] += bU[(size_t)i * N + t];
        for (int i = 0; i < m; ++i) S->mu[i] = row[i] > S->mu[i] ? row[i] : S->mu[i];
    }
    for (int t = 0; t < N; ++t) {
        float* row = S->st + (size_t)t * m;
        for (int i = 0; i < m; ++i) row[i] = exp_cw(row[i] - S->mu[i]);
        float* vr = S->vp + (size_t)t * dp;
        const float* vt = V + (size_t)t * d;
        for (int c = 0; c < d; ++c) vr[c] = vt[c];
        vr[d] = 1.f;
        for (int c = d + 1; c < dp; ++c) vr[c] = 0.f;
    }
    gemm_tn(S->st, m, S->vp, dp, S->w, m, N, dp);
    /* 3. A = exp((s Qbar) Kbar^T - m_U), row-wise */
    mm(S->qbar, S->kbarT, S->a, m, d, m);
    for (int i = 0; i < m; ++i)
        for (int j = 0; j < m; ++j)
            S->a[(size_t)i * m + j] =
                exp_cw(S->a[(size_t)i * m + j] + (bA ? bA[(size_t)i * m + j] : 0.f) - S->mu[i]);
    /* 4. Z_0 = A^T / (||A||_1 ||A||_inf), then the iteration */
    float n1 = 0.f, ninf = 0.f;
    for (int j = 0; j < m; ++j) {
        float col = 0.f;
        for (int i = 0; i < m; ++i) col += fabsf(S->a[(size_t)i * m + j]);
        n1 = col > n1 ? col : n1;
    }
    for (int i = 0; i < m; ++i) {
        float rw = 0.f;
        for (int j = 0; j < m; ++j) rw += fabsf(S->a[(size_t)i * m + j]);
        ninf = rw > ninf ? rw : ninf;
    }
    const float a0 = 1.0f / (n1 * ninf);
    for (int i = 0; i < m; ++i)
        for (int j = 0; j < m; ++j) S->z[(size_t)i * m + j] = a0 * S->a[(size_t)j * m + i];
    for (int k = 0; k < iters; ++k) {
        mm(S->a, S->z, S->x, m, m, m);                        /* X = A Z */
        for (int e = 0; e < m * m; ++e) S->t1[e] = -S->x[e];  /* 7I - X */
        for (int i = 0; i < m; ++i) S->t1[(size_t)i * m + i] += 7.f;
        mm(S->x, S->t1, S->t2, m, m, m);                      /* X (7I - X) */
        for (int e = 0; e < m * m; ++e) S->t2[e] = -S->t2[e]; /* 15I - X (7I - X) */
        for (int i = 0; i < m; ++i) S->t2[(size_t)i * m + i] += 15.f;
        mm(S->x, S->t2, S->t1, m, m, m);                      /* X (15I - ...) */
        for (int e = 0; e < m * m; ++e) S->t1[e] = -S->t1[e]; /* 13I - X (...) */
        for (int i = 0; i < m; ++i) S->t1[(size_t)i * m + i] += 13.f;
        mm(S->z, S->t1, S->t2, m, m, m);                      /* Z (13I - ...) */
        for (int e = 0; e < m * m; ++e) S->z[e] = 0.25f * S->t2[e];
    }
    /* 5. Y = Z W */
    mm(S->z, S->w, S->y, m, m, dp);
    /* 6. outputs: S_L = Q (s Kbar)^T (N x m, into st), G_L^n row by row, then
     *    (G_L^n Y) into st's room after it, divided by its last column */
    gemm_nn(Q, d, S->kbarTs, m, S->st, m, N, d, m, 0);
    for (int t = 0; t < N; ++t) {
        float* row = S->st + (size_t)t * m;
        if (bL)
            for (int j = 0; j < m; ++j) row[j] += bL[(size_t)t * m + j];
        const float mx = row_max(row, m);
        for (int j = 0; j < m; ++j) row[j] = exp_cw(row[j] - mx);
    }
    float* num = S->num;
    for (int t0 = 0; t0 < N; t0 += NBLK) {
        const int nb = N - t0 < NBLK ? N - t0 : NBLK;
        gemm_nn(S->st + (size_t)t0 * m, m, S->y, dp, num, dp, nb, m, dp, 0);
        for (int t = 0; t < nb; ++t) {
            const float inv = 1.0f / num[(size_t)t * dp + d];
            float* ot = O + (size_t)(t0 + t) * d;
            for (int c = 0; c < d; ++c) ot[c] = num[(size_t)t * dp + c] * inv;
        }
    }
}

static int threads_or_default(int threads) {
#ifdef _OPENMP
    return threads > 0 ? threads : omp_get_max_threads();
#else
    (void)threads;
    return 1;
#endif
}

int nystra_host_threads(void) { return threads_or_default(0); }

/* Landmark of token t: segments of N/m tokens, or b x b patches of the w x w
 * window (landmark (row / b) * p + col / b). */
static int landmark_of(int t, int N, int m, int landmarks, int wdt, int pgrid) {
    if (landmarks == NYSTRA_LANDMARKS_SEGMENTS) return t / (N / m);
    const int b = wdt / pgrid, row = t / wdt, col = t % wdt;
    return (row / b) * pgrid + col / b;
}

static int shape_ok(int N, int m, int landmarks, int* wdt, int* pgrid) {
    if (N < 1 || N > MAXN || m < 1 || m > N || m > MAXM || N % m != 0) return 0;
    if (landmarks != NYSTRA_LANDMARKS_SEGMENTS && landmarks != NYSTRA_LANDMARKS_PATCHES) return 0;
    *wdt = *pgrid = 0;
    if (landmarks == NYSTRA_LANDMARKS_PATCHES) {
        *wdt = isqrt_exact(N);
        *pgrid = isqrt_exact(m);
        if (*wdt < 0 || *pgrid < 0 || *wdt % *pgrid != 0) return 0;
    }
    return 1;
}

static int attention_host(const float* q, const float* k, const float* v, float* out, int n_windows, int heads,
                          int N, int d_h, int m, int iters, int landmarks, const float* bias_L, const float* bias_U,
                          const float* bias_A, int bias_windows, int threads);

int nystra_attention_host(const float* q, const float* k, const float* v, float* out, int n_windows, int heads,
                          int N, int d_h, int m, int iters, int landmarks, int threads) {
    return attention_host(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, NULL, NULL, NULL, 0, threads);
}

int nystra_attention_bias_host(const float* q, const float* k, const float* v, float* out, int n_windows,
                               int heads, int N, int d_h, int m, int iters, int landmarks, const float* bias_L,
                               const float* bias_U, const float* bias_A, int bias_windows, int threads) {
    if (n_windows > 0 && heads > 0) {
        if (bias_windows != 1 && bias_windows != n_windows) return NYSTRA_EINVAL;
        if (!bias_L || !bias_U || !bias_A) return NYSTRA_EINVAL;
        if (N >= 1 && N <= MAXN && m >= 1 && m <= MAXM && d_h >= 1 && d_h <= MAXD && out) {
            const size_t ob = (size_t)n_windows * heads * N * d_h * sizeof(float);
            const size_t nm = (size_t)bias_windows * heads * N * m * sizeof(float);
            const size_t mm2 = (size_t)bias_windows * heads * m * m * sizeof(float);
            const uintptr_t o = (uintptr_t)out;
            if ((o < (uintptr_t)bias_L + nm && (uintptr_t)bias_L < o + ob) ||
                (o < (uintptr_t)bias_U + nm && (uintptr_t)bias_U < o + ob) ||
                (o < (uintptr_t)bias_A + mm2 && (uintptr_t)bias_A < o + ob))
                return NYSTRA_EINVAL;
        }
    }
    return attention_host(q, k, v, out, n_windows, heads, N, d_h, m, iters, landmarks, bias_L, bias_U, bias_A,
                          bias_windows, threads);
}

int nystra_pool_bias_host(const float* bias, int n_bias, int N, int m, int landmarks, float* bias_L, float* bias_U,
                          float* bias_A, int threads) {
    int wdt, pgrid;
    if (n_bias < 0 || !shape_ok(N, m, landmarks, &wdt, &pgrid)) return NYSTRA_EINVAL;
    if (n_bias == 0) return NYSTRA_OK;
    if (!bias || !bias_L || !bias_U || !bias_A) return NYSTRA_EINVAL;
    const size_t in = (size_t)n_bias * N * N * sizeof(float), nm = (size_t)n_bias * N * m * sizeof(float),
                 mm2 = (size_t)n_bias * m * m * sizeof(float);
    const void* outs[3] = {bias_L, bias_U, bias_A};
    const size_t sz[3] = {nm, nm, mm2};
    for (int i = 0; i < 3; ++i) {
        const uintptr_t a = (uintptr_t)outs[i];
        if (a < (uintptr_t)bias + in && (uintptr_t)bias < a + sz[i]) return NYSTRA_EINVAL;
        for (int j = i + 1; j < 3; ++j) {
            const uintptr_t b = (uintptr_t)outs[j];
            if (a < b + sz[j] && b < a + sz[i]) return NYSTRA_EINVAL;
        }
    }
    const int nt = threads_or_default(threads);
    const float inv = (float)m / (float)N;  /* 1 / (tokens per landmark) */
#pragma omp parallel for num_threads(nt) schedule(static)
    for (int u = 0; u < n_bias; ++u) {
        const float* B = bias + (size_t)u * N * N;
        float* L = bias_L + (size_t)u * N * m;
        float* U = bias_U + (size_t)u * m * N;
        float* A = bias_A + (size_t)u * m * m;
        memset(L, 0, sizeof(float) * (size_t)N * m);
        memset(U, 0, sizeof(float) * (size_t)m * N);
        memset(A, 0, sizeof(float) * (size_t)m * m);
        /* sums over each landmark's tokens (as keys for L, as queries for U, both for A), then means */
        for (int s2 = 0; s2 < N; ++s2) {
            const int i = landmark_of(s2, N, m, landmarks, wdt, pgrid);
            for (int t = 0; t < N; ++t) {
                const float b = B[(size_t)s2 * N + t];
                const int j = landmark_of(t, N, m, landmarks, wdt, pgrid);
                L[(size_t)s2 * m + j] += b;
                U[(size_t)i * N + t] += b;
                A[(size_t)i * m + j] += b;
            }
        }
        for (size_t e = 0; e < (size_t)N * m; ++e) {
            L[e] *= inv;
            U[e] *= inv;
        }
        for (int e = 0; e < m * m; ++e) A[e] *= inv * inv;
    }
    return NYSTRA_OK;
}

static int attention_host(const float* q, const float* k, const float* v, float* out, int n_windows, int heads,
                          int N, int d_h, int m, int iters, int landmarks, const float* bias_L, const float* bias_U,
                          const float* bias_A, int bias_windows, int threads) {
    if (n_windows < 0 || heads < 0) return NYSTRA_EINVAL;
    if (d_h < 1 || d_h > MAXD) return NYSTRA_EINVAL;
    int wdt = 0, pgrid = 0;
    if (!shape_ok(N, m, landmarks, &wdt, &pgrid)) return NYSTRA_EINVAL;
    if (iters < 0 || iters > NYSTRA_MAX_ITERS) return NYSTRA_EINVAL;
    const long long units = (long long)n_windows * heads;
    if (units == 0) return NYSTRA_OK;
    if (!q || !k || !v || !out) return NYSTRA_EINVAL;
    const size_t bytes = (size_t)units * N * d_h * sizeof(float);
    if (overlaps(out, q, bytes) || overlaps(out, k, bytes) || overlaps(out, v, bytes)) return NYSTRA_EINVAL;
    const int nt = threads_or_default(threads);
    int status = NYSTRA_OK;
#pragma omp parallel num_threads(nt)
    {
        Scratch* S = (Scratch*)malloc(sizeof(Scratch));
        if (!S) {
#pragma omp atomic write
            status = NYSTRA_EINVAL;
        } else {
            for (int t = 0; t < N; ++t) S->seg[t] = landmark_of(t, N, m, landmarks, wdt, pgrid);
#pragma omp for schedule(static)
            for (long long u = 0; u < units; ++u) {
                const size_t off = (size_t)u * N * d_h;
                /* the unit's bias slice: its head's (shared) or its own (per window) */
                const long long sl = bias_L ? (bias_windows == 1 ? u % heads : u) : 0;
                one_unit(q + off, k + off, v + off, out + off, N, d_h, m, iters,
                         bias_L ? bias_L + (size_t)sl * N * m : NULL, bias_U ? bias_U + (size_t)sl * m * N : NULL,
                         bias_A ? bias_A + (size_t)sl * m * m : NULL, S);
            }
            free(S);
        }
    }
    return status;
}

int exact_window_attention_host(const float* q, const float* k, const float* v, float* out, int n_windows,
                                int heads, int N, int d_h, int threads) {
    if (n_windows < 0 || heads < 0) return NYSTRA_EINVAL;
    if (N < 1 || N > MAXN || d_h < 1 || d_h > MAXD) return NYSTRA_EINVAL;
    const long long units = (long long)n_windows * heads;
    if (units == 0) return NYSTRA_OK;
    if (!q || !k || !v || !out) return NYSTRA_EINVAL;
    const size_t bytes = (size_t)units * N * d_h * sizeof(float);
    if (overlaps(out, q, bytes) || overlaps(out, k, bytes) || overlaps(out, v, bytes)) return NYSTRA_EINVAL;
    const int nt = threads_or_default(threads);
    int status = NYSTRA_OK;
    const float s = 1.0f / sqrtf((float)d_h);
    const int dp = (d_h + 1 + 15) / 16 * 16;  /* [V | 1] padded for full register blocks */
#pragma omp parallel num_threads(nt)
    {
        /* per thread: s K^T (d x N), [V | 1 | 0] (N x dp), scores and numerators of a block of queries */
        float* kT = (float*)malloc(sizeof(float) * (size_t)MAXD * MAXN);
        float* vp = (float*)malloc(sizeof(float) * (size_t)MAXN * MAXDP);
        float* p = (float*)malloc(sizeof(float) * (size_t)NBLK * MAXN);
        float* num = (float*)malloc(sizeof(float) * (size_t)NBLK * MAXDP);
        if (!kT || !vp || !p || !num) {
#pragma omp atomic write
            status = NYSTRA_EINVAL;
        } else {
#pragma omp for schedule(static)
            for (long long u = 0; u < units; ++u) {
                const size_t off = (size_t)u * N * d_h;
                const float *Q = q + off, *K = k + off, *V = v + off;
                float* O = out + off;
                for (int t = 0; t < N; ++t) {
                    for (int c = 0; c < d_h; ++c) {
                        kT[(size_t)c * N + t] = K[(size_t)t * d_h + c] * s;
                        vp[(size_t)t * dp + c] = V[(size_t)t * d_h + c];
                    }
                    vp[(size_t)t * dp + d_h] = 1.f;  /* the ones column: the softmax denominators */
                    for (int c = d_h + 1; c < dp; ++c) vp[(size_t)t * dp + c] = 0.f;
                }
                for (int i0 = 0; i0 < N; i0 += NBLK) {
                    const int nb = N - i0 < NBLK ? N - i0 : NBLK;
                    gemm_nn(Q + (size_t)i0 * d_h, d_h, kT, N, p, N, nb, d_h, N, 0);  /* scores Q (s K)^T */
                    for (int i = 0; i < nb; ++i) {
                        float* pr = p + (size_t)i * N;
                        const float mx = row_max(pr, N);
                        for (int t = 0; t < N; ++t) pr[t] = exp_cw(pr[t] - mx);
                    }
                    gemm_nn(p, N, vp, dp, num, dp, nb, N, dp, 0);  /* exp(scores) [V | 1] */
                    for (int i = 0; i < nb; ++i) {
                        const float inv = 1.0f / num[(size_t)i * dp + d_h];
                        for (int c = 0; c < d_h; ++c) O[(size_t)(i0 + i) * d_h + c] = num[(size_t)i * dp + c] * inv;
                    }
                }
            }
        }
        free(kT);
        free(vp);
        free(p);
        free(num);
    }
    return status;
}
