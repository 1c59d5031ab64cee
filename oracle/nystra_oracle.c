/*
 * Float64 CPU oracle for PnP-Nystra window attention.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file; only the test-suite, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no code, header or constant with the CUDA
 * library: it is a plain, slow, literal restatement of the paper's method so
 * that a reader can check it against the paper by eye.
 *
 * Paper: "Plug-and-Play Linear Attention with Provable Guarantees for
 * Training-Free Image Restoration" (PnP-Nystra, arXiv 2506.08520).
 *
 * Every function works on one or more independent "units".  A unit is one
 * (window, head) pair with Q, K, V in R^{N x d}, stored row-major and
 * contiguous; unit u starts at offset u*N*d.  All arithmetic is float64.
 *
 * Readings where the paper is silent:
 *   - landmarks are means over m contiguous, non-overlapping segments of
 *     L = N/m tokens in the window's token order (Sec. 2.2 "average pooling
 *     over non-overlapping windows"); m must divide N.  The other reading,
 *     pool = 1: a square window of w x w tokens (N = w^2, row-major) pooled
 *     over a p x p grid of square b x b patches (m = p^2, b = w/p), landmark
 *     j = (row j/p, column j%p) of that grid;
 *   - the scale is 1/sqrt(d) with d the per-head dimension (Eq. 1, Sec. 1);
 *   - the pseudo-inverse is the third-order iteration
 *       Z_{k+1} = 1/4 Z_k (13 I - A Z_k (15 I - A Z_k (7 I - A Z_k)))
 *     started from Z_0 = A^T / (||A||_1 ||A||_inf) and run for `iters`
 *     steps, applied to the normalised core block A = G_A^n (Sec. 2.2);
 *   - no guard on the denominator (Alg. 1 step 7 divides as written);
 *   - an additive score bias B (N x N, the relative-position bias and masks
 *     of window attention; Eq. 1 has none) enters every block the way the
 *     landmarks enter it: a landmark stands for the mean of its tokens, so
 *     S_L[i][j] += mean_{t in j} B[i][t], S_U[j][t] += mean_{s in j} B[s][t]
 *     and S_A[i][j] += mean_{s in i, t in j} B[s][t].
 *
 * Parallelism: units are spread over OpenMP threads; each unit is computed
 * sequentially, so the result does not depend on the thread count.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Number of host threads the oracle's parallel loops use. */
int oracle_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------ */
/* Small dense helpers (row-major, float64).                           */
/* ------------------------------------------------------------------ */

/* C[r x c] = A[r x n] * B[n x c] */
static void matmul(const double* A, const double* B, double* C, int r, int n, int c) {
    for (int i = 0; i < r; ++i)
        for (int j = 0; j < c; ++j) {
            double acc = 0.0;
            for (int t = 0; t < n; ++t) acc += A[(size_t)i * n + t] * B[(size_t)t * c + j];
            C[(size_t)i * c + j] = acc;
        }
}

/* ------------------------------------------------------------------ */
/* Exact softmax attention, Eq. (1):  A = Q K^T / sqrt(d),             */
/* S = softmax(A) row-wise, O = S V.  Rows are max-shifted before exp; */
/* the shift cancels in the row normalisation (Eq. 2).                 */
/* ------------------------------------------------------------------ */
static void exact_unit(const double* q, const double* k, const double* v, double* o,
                       int N, int d, const double* B, double* row) {
    const double s = 1.0 / sqrt((double)d);
    for (int i = 0; i < N; ++i) {
        double mx = -INFINITY;
        for (int j = 0; j < N; ++j) {
            double a = 0.0;
            for (int c = 0; c < d; ++c) a += q[(size_t)i * d + c] * k[(size_t)j * d + c];
            row[j] = s * a + (B ? B[(size_t)i * N + j] : 0.0);
            if (row[j] > mx) mx = row[j];
        }
        double den = 0.0;
        for (int j = 0; j < N; ++j) {
            row[j] = exp(row[j] - mx);
            den += row[j];
        }
        for (int c = 0; c < d; ++c) {
            double num = 0.0;
            for (int j = 0; j < N; ++j) num += row[j] * v[(size_t)j * d + c];
            o[(size_t)i * d + c] = num / den;
        }
    }
}

/* Exact attention of every unit; bias (NULL or N x N per unit) is added to
 * the scaled scores before the softmax. */
void oracle_exact_attention_bias(const double* q, const double* k, const double* v, double* out,
                                 long n_units, int N, int d, const double* bias) {
    const size_t unit = (size_t)N * d;
#pragma omp parallel
    {
        double* row = (double*)malloc(sizeof(double) * (size_t)N);
#pragma omp for schedule(dynamic, 4)
        for (long u = 0; u < n_units; ++u)
            exact_unit(q + u * unit, k + u * unit, v + u * unit, out + u * unit, N, d,
                       bias ? bias + (size_t)u * N * N : 0, row);
        free(row);
    }
}

void oracle_exact_attention(const double* q, const double* k, const double* v, double* out,
                            long n_units, int N, int d) {
    oracle_exact_attention_bias(q, k, v, out, n_units, N, d, 0);
}

/* ------------------------------------------------------------------ */
/* Algorithm 1, step 1: landmarks by average pooling over m            */
/* non-overlapping contiguous segments of L = N/m tokens.              */
/* xbar[j][c] = (1/L) * sum_{t = jL}^{jL+L-1} x[t][c].                 */
/* ------------------------------------------------------------------ */
void oracle_landmarks(const double* x, int N, int d, int m, double* xbar) {
    const int L = N / m;
    for (int j = 0; j < m; ++j)
        for (int c = 0; c < d; ++c) {
            double acc = 0.0;
            for (int t = j * L; t < (j + 1) * L; ++t) acc += x[(size_t)t * d + c];
            xbar[(size_t)j * d + c] = acc / (double)L;
        }
}

/* Integer square root of n, or -1 if n is not a perfect square. */
static int exact_sqrt(int n) {
    int r = 0;
    while ((r + 1) * (r + 1) <= n) ++r;
    return r * r == n ? r : -1;
}

/* pool = 1 needs N = w^2, m = p^2 and p dividing w. */
static int pool_valid(int N, int m, int pool) {
    if (pool == 0) return N % m == 0;
    if (pool != 1) return 0;
    const int w = exact_sqrt(N), p = exact_sqrt(m);
    return w > 0 && p > 0 && w % p == 0;
}

/* Step 1 over square patches (pool = 1): token t = (t/w, t%w) of the w x w
 * window; landmark j averages the b x b tokens of patch (j/p, j%p),
 *   xbar[j][c] = (1/b^2) sum_{r = (j/p) b}^{(j/p) b + b-1}
 *                        sum_{s = (j%p) b}^{(j%p) b + b-1} x[r w + s][c]. */
void oracle_landmarks_patches(const double* x, int N, int d, int m, double* xbar) {
    const int w = exact_sqrt(N), p = exact_sqrt(m), b = w / p;
    for (int j = 0; j < m; ++j)
        for (int c = 0; c < d; ++c) {
            double acc = 0.0;
            for (int r = (j / p) * b; r < (j / p) * b + b; ++r)
                for (int s = (j % p) * b; s < (j % p) * b + b; ++s) acc += x[((size_t)r * w + s) * d + c];
            xbar[(size_t)j * d + c] = acc / (double)(b * b);
        }
}

/* Landmark of token t: its segment (pool = 0) or its square patch (pool = 1). */
static int landmark_of(int t, int N, int m, int pool) {
    if (pool == 0) return t / (N / m);
    const int w = exact_sqrt(N), p = exact_sqrt(m), b = w / p;
    return ((t / w) / b) * p + (t % w) / b;
}

/* The additive score bias B (N x N) of one unit seen through the landmarks:
 *   BL[i][j] = mean over tokens t of landmark j of B[i][t]          (N x m)
 *   BU[j][t] = mean over tokens s of landmark j of B[s][t]          (m x N)
 *   BA[i][j] = mean over s of landmark i, t of landmark j of B[s][t] (m x m)
 * Every landmark averages L = N/m tokens under either pooling. */
void oracle_pool_bias(const double* B, int N, int m, int pool, double* BL, double* BU, double* BA) {
    const double L = (double)(N / m);
    memset(BL, 0, sizeof(double) * (size_t)N * m);
    memset(BU, 0, sizeof(double) * (size_t)m * N);
    memset(BA, 0, sizeof(double) * (size_t)m * m);
    for (int s = 0; s < N; ++s)
        for (int t = 0; t < N; ++t) {
            const double b = B[(size_t)s * N + t];
            const int js = landmark_of(s, N, m, pool), jt = landmark_of(t, N, m, pool);
            BL[(size_t)s * m + jt] += b / L;
            BU[(size_t)js * N + t] += b / L;
            BA[(size_t)js * m + jt] += b / (L * L);
        }
}

/* ------------------------------------------------------------------ */
/* Algorithm 1, step 4: approximate (pseudo-)inverse of the m x m      */
/* matrix A by the third-order iteration of Razavi et al. (2014):      */
/*   Z_0     = A^T / (||A||_1 * ||A||_inf)                             */
/*   X       = A Z_k                                                   */
/*   Z_{k+1} = 1/4 * Z_k * (13 I - X (15 I - X (7 I - X)))             */
/* ||A||_1 is the largest absolute column sum, ||A||_inf the largest   */
/* absolute row sum.  `iters` = number of updates after Z_0.           */
/* ------------------------------------------------------------------ */
void oracle_pinv_iteration(const double* A, int m, int iters, double* Z) {
    const size_t mm = (size_t)m * m;
    double norm1 = 0.0, norminf = 0.0;
    for (int j = 0; j < m; ++j) {
        double col = 0.0;
        for (int i = 0; i < m; ++i) col += fabs(A[(size_t)i * m + j]);
        if (col > norm1) norm1 = col;
    }
    for (int i = 0; i < m; ++i) {
        double row = 0.0;
        for (int j = 0; j < m; ++j) row += fabs(A[(size_t)i * m + j]);
        if (row > norminf) norminf = row;
    }
    const double scale = 1.0 / (norm1 * norminf);
    for (int i = 0; i < m; ++i)
        for (int j = 0; j < m; ++j) Z[(size_t)i * m + j] = scale * A[(size_t)j * m + i];

    double* X = (double*)malloc(sizeof(double) * mm);
    double* T = (double*)malloc(sizeof(double) * mm);
    double* U = (double*)malloc(sizeof(double) * mm);
    for (int it = 0; it < iters; ++it) {
        matmul(A, Z, X, m, m, m);                     /* X = A Z            */
        for (size_t e = 0; e < mm; ++e) T[e] = -X[e]; /* T = 7I - X         */
        for (int i = 0; i < m; ++i) T[(size_t)i * m + i] += 7.0;
        matmul(X, T, U, m, m, m);                     /* U = X (7I - X)     */
        for (size_t e = 0; e < mm; ++e) T[e] = -U[e]; /* T = 15I - U        */
        for (int i = 0; i < m; ++i) T[(size_t)i * m + i] += 15.0;
        matmul(X, T, U, m, m, m);                     /* U = X (15I - ...)  */
        for (size_t e = 0; e < mm; ++e) T[e] = -U[e]; /* T = 13I - U        */
        for (int i = 0; i < m; ++i) T[(size_t)i * m + i] += 13.0;
        matmul(Z, T, U, m, m, m);                     /* U = Z (13I - ...)  */
        for (size_t e = 0; e < mm; ++e) Z[e] = 0.25 * U[e];
    }
    free(X);
    free(T);
    free(U);
}

/* ------------------------------------------------------------------ */
/* One unit of PnP-Nystra, Algorithm 1 in the stabilised form of       */
/* Eq. 8.  Any stage pointer may be NULL.                               */
/*   qbar, kbar : m x d   landmarks (step 1)                           */
/*   mL  : N   row maxima of S_L = Q Kbar^T / sqrt(d)                  */
/*   mU  : m   row maxima of S_U = Qbar K^T / sqrt(d), over all N keys */
/*   GLn : N x m   exp(S_L - mL)          = M_L^{-1} G_L               */
/*   GUn : m x N   exp(S_U - mU)          = M_U^{-1} G_U               */
/*   GAn : m x m   exp(Qbar Kbar^T/sqrt(d) - mU) = M_U^{-1} G_A        */
/*   Z   : m x m   iterative pseudo-inverse of GAn (step 4)            */
/*   num : N x d   O_N = P (G_U^n V), P = G_L^n Z (steps 5-6)          */
/*   den : N       O_D = P (G_U^n 1_N)                 (step 6)        */
/*   o   : N x d   O_N / O_D row-wise                  (step 7)        */
/* ------------------------------------------------------------------ */
typedef struct {
    double *qbar, *kbar, *mL, *mU, *GLn, *GUn, *GAn, *Z, *num, *den;
} stage_ptrs;

static void nystra_unit(const double* q, const double* k, const double* v, double* o,
                        int N, int d, int m, int iters, int pool, const double* B, stage_ptrs st) {
    const double s = 1.0 / sqrt((double)d);
    double* qbar = (double*)malloc(sizeof(double) * (size_t)m * d);
    double* kbar = (double*)malloc(sizeof(double) * (size_t)m * d);
    double* mL = (double*)malloc(sizeof(double) * (size_t)N);
    double* mU = (double*)malloc(sizeof(double) * (size_t)m);
    double* GL = (double*)malloc(sizeof(double) * (size_t)N * m);
    double* GU = (double*)malloc(sizeof(double) * (size_t)m * N);
    double* GA = (double*)malloc(sizeof(double) * (size_t)m * m);
    double* Z = (double*)malloc(sizeof(double) * (size_t)m * m);
    double* P = (double*)malloc(sizeof(double) * (size_t)N * m);
    double* GUV = (double*)malloc(sizeof(double) * (size_t)m * d);
    double* GU1 = (double*)malloc(sizeof(double) * (size_t)m);
    double* num = (double*)malloc(sizeof(double) * (size_t)N * d);
    double* den = (double*)malloc(sizeof(double) * (size_t)N);

    /* Step 1: landmark queries and keys. */
    if (pool == 1) {
        oracle_landmarks_patches(q, N, d, m, qbar);
        oracle_landmarks_patches(k, N, d, m, kbar);
    } else {
        oracle_landmarks(q, N, d, m, qbar);
        oracle_landmarks(k, N, d, m, kbar);
    }

    /* The score bias through the landmarks (zero without a bias). */
    double* BL = (double*)calloc((size_t)N * m, sizeof(double));
    double* BU = (double*)calloc((size_t)m * N, sizeof(double));
    double* BA = (double*)calloc((size_t)m * m, sizeof(double));
    if (B) oracle_pool_bias(B, N, m, pool, BL, BU, BA);

    /* Steps 2-3 with row-max stabilisation.  S_L, its row max m_L. */
    for (int i = 0; i < N; ++i) {
        double mx = -INFINITY;
        for (int j = 0; j < m; ++j) {
            double a = 0.0;
            for (int c = 0; c < d; ++c) a += q[(size_t)i * d + c] * kbar[(size_t)j * d + c];
            const double sl = s * a + BL[(size_t)i * m + j];
            GL[(size_t)i * m + j] = sl;
            if (sl > mx) mx = sl;
        }
        mL[i] = mx;
    }
    /* S_U and its row max m_U, taken over all N keys. */
    for (int i = 0; i < m; ++i) {
        double mx = -INFINITY;
        for (int j = 0; j < N; ++j) {
            double a = 0.0;
            for (int c = 0; c < d; ++c) a += qbar[(size_t)i * d + c] * k[(size_t)j * d + c];
            const double su = s * a + BU[(size_t)i * N + j];
            GU[(size_t)i * N + j] = su;
            if (su > mx) mx = su;
        }
        mU[i] = mx;
    }
    /* Normalised blocks: G_L^n = M_L^{-1} G_L, G_U^n = M_U^{-1} G_U,
     * G_A^n = M_U^{-1} G_A (row i of G_A scaled by exp(-m_U(i))). */
    for (int i = 0; i < N; ++i)
        for (int j = 0; j < m; ++j) GL[(size_t)i * m + j] = exp(GL[(size_t)i * m + j] - mL[i]);
    for (int i = 0; i < m; ++i)
        for (int j = 0; j < N; ++j) GU[(size_t)i * N + j] = exp(GU[(size_t)i * N + j] - mU[i]);
    for (int i = 0; i < m; ++i)
        for (int j = 0; j < m; ++j) {
            double a = 0.0;
            for (int c = 0; c < d; ++c) a += qbar[(size_t)i * d + c] * kbar[(size_t)j * d + c];
            GA[(size_t)i * m + j] = exp(s * a + BA[(size_t)i * m + j] - mU[i]);
        }

    /* Step 4: pseudo-inverse of G_A^n. */
    oracle_pinv_iteration(GA, m, iters, Z);

    /* Step 5: premultiplier P = G_L^n Z. */
    matmul(GL, Z, P, N, m, m);

    /* Step 6: O_N = P (G_U^n V), O_D = P (G_U^n 1_N). */
    matmul(GU, v, GUV, m, N, d);
    for (int i = 0; i < m; ++i) {
        double acc = 0.0;
        for (int j = 0; j < N; ++j) acc += GU[(size_t)i * N + j];
        GU1[i] = acc;
    }
    matmul(P, GUV, num, N, m, d);
    matmul(P, GU1, den, N, m, 1);

    /* Step 7: row-wise normalisation. */
    for (int i = 0; i < N; ++i)
        for (int c = 0; c < d; ++c) o[(size_t)i * d + c] = num[(size_t)i * d + c] / den[i];

    if (st.qbar) memcpy(st.qbar, qbar, sizeof(double) * (size_t)m * d);
    if (st.kbar) memcpy(st.kbar, kbar, sizeof(double) * (size_t)m * d);
    if (st.mL) memcpy(st.mL, mL, sizeof(double) * (size_t)N);
    if (st.mU) memcpy(st.mU, mU, sizeof(double) * (size_t)m);
    if (st.GLn) memcpy(st.GLn, GL, sizeof(double) * (size_t)N * m);
    if (st.GUn) memcpy(st.GUn, GU, sizeof(double) * (size_t)m * N);
    if (st.GAn) memcpy(st.GAn, GA, sizeof(double) * (size_t)m * m);
    if (st.Z) memcpy(st.Z, Z, sizeof(double) * (size_t)m * m);
    if (st.num) memcpy(st.num, num, sizeof(double) * (size_t)N * d);
    if (st.den) memcpy(st.den, den, sizeof(double) * (size_t)N);

    free(BL); free(BU); free(BA);
    free(qbar); free(kbar); free(mL); free(mU); free(GL); free(GU); free(GA);
    free(Z); free(P); free(GUV); free(GU1); free(num); free(den);
}

/* Batched PnP-Nystra output with landmark pooling `pool` (0 = segments,
 * 1 = square patches) and an additive score bias (NULL, or N x N per unit).
 * Returns 0, or -1 for an m the pooling cannot form. */
int oracle_nystra_attention_bias(const double* q, const double* k, const double* v, double* out,
                                 long n_units, int N, int d, int m, int iters, int pool, const double* bias) {
    if (m < 1 || m > N || !pool_valid(N, m, pool) || iters < 0) return -1;
    const size_t unit = (size_t)N * d;
    const stage_ptrs none = {0};
#pragma omp parallel for schedule(dynamic, 4)
    for (long u = 0; u < n_units; ++u)
        nystra_unit(q + u * unit, k + u * unit, v + u * unit, out + u * unit, N, d, m, iters, pool,
                    bias ? bias + (size_t)u * N * N : 0, none);
    return 0;
}

/* Without a bias. */
int oracle_nystra_attention_pool(const double* q, const double* k, const double* v, double* out,
                                 long n_units, int N, int d, int m, int iters, int pool) {
    return oracle_nystra_attention_bias(q, k, v, out, n_units, N, d, m, iters, pool, 0);
}

/* Batched PnP-Nystra output, segment landmarks.  -1 if m does not divide N. */
int oracle_nystra_attention(const double* q, const double* k, const double* v, double* out,
                            long n_units, int N, int d, int m, int iters) {
    return oracle_nystra_attention_pool(q, k, v, out, n_units, N, d, m, iters, 0);
}

/* Single-unit PnP-Nystra exposing every intermediate (NULL to skip). */
int oracle_nystra_stages(const double* q, const double* k, const double* v, double* out,
                         int N, int d, int m, int iters, int pool,
                         double* qbar, double* kbar, double* mL, double* mU,
                         double* GLn, double* GUn, double* GAn, double* Z,
                         double* num, double* den) {
    if (m < 1 || m > N || !pool_valid(N, m, pool) || iters < 0) return -1;
    stage_ptrs st = {qbar, kbar, mL, mU, GLn, GUn, GAn, Z, num, den};
    nystra_unit(q, k, v, out, N, d, m, iters, pool, 0, st);
    return 0;
}
