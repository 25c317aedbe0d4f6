/*
 * gs_oracle.c -- float64 CPU oracle for the Gram-Space codebook path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the checker, not the product: only
 * the tests, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
 * arm may load it.  It shares no code, header, table or constant with the CUDA
 * library under paper_2608_01528_gb300/csrc, and never calls it.
 *
 * It is written for a reader checking it against the paper by eye: plain
 * loops, float64 throughout, no blocking or reordering of arithmetic beyond
 * what each definition states.  OpenMP only distributes independent rows.
 *
 * Notation (paper -> here).  The paper stores the codebook as W (D x M, one
 * atom per column), the basis as U (D x k) and the Gram-loc codebook as
 * T = U^T W (k x M) (Sec. 3.1, Eq. 1).  Here every matrix is row-major with
 * one vector per row:
 *     C = W^T (M x D),  Q = U^T (r x D, r = k),  R = T^T (M x r),  C = R Q.
 * A query x is represented by its Gram-loc t = U^T x (Sec. 3.1), which is the
 * row y = x Q^T here; reconstruction x = U t (Sec. 3.1, Sec. 3.3) is
 * xhat = t Q.
 *
 * Readings of the paper that this file fixes (the paper is silent on them):
 *  - Gram-Schmidt variant: modified Gram-Schmidt in codeword (row) order,
 *    each row projected twice against the basis built so far
 *    ("reorthogonalisation"; Sec. 3.1 and Sec. 3.3 name Gram-Schmidt, Sec. 3.2
 *    notes the loss of orthogonality of classical GS).
 *  - Rank decision: a row is dependent when the norm left after both passes
 *    is <= tau * ||c_i|| (its own original norm).  Zero rows are always
 *    dependent.  The rank k of Sec. 3.2 is the number of accepted rows.
 *  - Sign: each new basis vector is v/||v|| with a positive coefficient
 *    R[i][r] = ||v||, so for a full-rank C the result is the unique LQ
 *    factorisation with positive diagonal.
 *  - Cosine similarity uses the full D-dimensional ||x|| of the query and
 *    ||c_i|| = ||R_i|| (Eq. 2 gives ||R_i|| = ||c_i||).
 *  - argmax returns the lowest index among equal maxima.
 *
 * Build: gcc -O2 -fPIC -shared [-fopenmp] gs_oracle.c -lm -o liboracle.so
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* Score modes of orc_similarity. */
#define ORC_SCORE_RAW 0
#define ORC_SCORE_COSINE 1
#define ORC_SCORE_SOFTMAX 2

int orc_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void orc_set_num_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

static double dot(const double* a, const double* b, int n) {
    double s = 0.0;
    for (int d = 0; d < n; ++d) s += a[d] * b[d];
    return s;
}

/*
 * Basis construction (Sec. 3.1, Eq. 1; Sec. 3.3 builds the basis once, at
 * initialisation, by Gram-Schmidt orthogonalisation of the codebook).
 *
 * For each codeword row c_i in order:
 *   v = c_i (optionally c_i/||c_i||: Sec. 3.1 scales the atoms to unit
 *   length);
 *   `passes` times: for j = 0 .. r-1 in order, h = <q_j, v> with the current
 *   v (modified GS), v -= h q_j, R[i][j] += h;
 *   if ||v|| > tau * ||c_i||: q_r = v / ||v||, R[i][r] = ||v||, r += 1.
 * Rows judged dependent keep their projections R[i][0..r-1] and add no basis
 * vector, so C = R Q holds row by row (Eq. 4: b = sum_i <b, q_i> q_i).
 *
 * passes is 2 in every use; the argument exists so that a test can plant the
 * single-pass mistake and see a pin fail.
 *
 * Q: capacity min(M, D) rows of D; R: M x ldr (ldr >= min(M, D)), zeroed here;
 * cnorm: M norms of the (possibly normalised) rows.  Returns the rank r.
 */
int orc_build_mgs(const double* C, int M, int D, double tau, int normalize_rows,
                  int passes, double* Q, double* R, int ldr, double* cnorm) {
    int r = 0;
    int rmax = M < D ? M : D;
    double* v = (double*)malloc(sizeof(double) * (size_t)(D > 0 ? D : 1));
    if (!v) return -1;
    for (int i = 0; i < M; ++i) {
        const double* c = C + (size_t)i * D;
        double cn = sqrt(dot(c, c, D));
        double s = 1.0;
        if (normalize_rows && cn > 0.0) s = 1.0 / cn;
        for (int d = 0; d < D; ++d) v[d] = c[d] * s;
        cn = sqrt(dot(v, v, D));
        cnorm[i] = cn;
        double* Ri = R + (size_t)i * ldr;
        for (int j = 0; j < ldr; ++j) Ri[j] = 0.0;
        for (int p = 0; p < passes; ++p) {
            for (int j = 0; j < r; ++j) {
                const double* q = Q + (size_t)j * D;
                double h = dot(q, v, D);
                for (int d = 0; d < D; ++d) v[d] -= h * q[d];
                Ri[j] += h;
            }
        }
        double nu = sqrt(dot(v, v, D));
        if (nu > tau * cn && r < rmax) {
            double* q = Q + (size_t)r * D;
            for (int d = 0; d < D; ++d) q[d] = v[d] / nu;
            Ri[r] = nu;
            r += 1;
        }
    }
    free(v);
    return r;
}

/*
 * Gram-loc of queries (Sec. 3.1: t = U^T x), Y[n][j] = <x_n, q_j>,
 * and the full-dimension query norms ||x_n|| used by cosine scores.
 */
void orc_project(const double* X, long N, int D, int ldx, const double* Q, int r,
                 double* Y, double* xnorm) {
    long n;
#pragma omp parallel for schedule(static)
    for (n = 0; n < N; ++n) {
        const double* x = X + (size_t)n * ldx;
        for (int j = 0; j < r; ++j) Y[(size_t)n * r + j] = dot(x, Q + (size_t)j * D, D);
        if (xnorm) xnorm[n] = sqrt(dot(x, x, D));
    }
}

/*
 * Similarity in Gram-loc (Sec. 2.2 "scaled dot-product similarity"; Sec. 3.2,
 * Eq. 2-3: inner products and norm-based similarities are preserved by the
 * orthonormal basis).  Raw scores are S[n][i] = scale * <y_n, R_i>.
 *   RAW:     S = scale * <y, R_i>
 *   COSINE:  S = scale * <y, R_i> / (||x|| * ||c_i||), 0 when a norm is 0
 *   SOFTMAX: S = softmax_i(scale * <y, R_i>) over the M codewords
 * argmax[n] = lowest i attaining max_i S[n][i]; maxval[n] = S[n][argmax].
 * S, argmax, maxval may each be NULL.
 */
void orc_similarity(const double* Y, long N, int r, const double* R, int ldr, int M,
                    int mode, double scale, const double* xnorm, const double* cnorm,
                    double* S, int* argmax, double* maxval) {
    long n;
#pragma omp parallel for schedule(static)
    for (n = 0; n < N; ++n) {
        double* s = (double*)malloc(sizeof(double) * (size_t)(M > 0 ? M : 1));
        const double* y = Y + (size_t)n * r;
        for (int i = 0; i < M; ++i) {
            double g = scale * dot(y, R + (size_t)i * ldr, r);
            if (mode == ORC_SCORE_COSINE) {
                double den = xnorm[n] * cnorm[i];
                g = den > 0.0 ? g / den : 0.0;
            }
            s[i] = g;
        }
        if (mode == ORC_SCORE_SOFTMAX && M > 0) {
            double mx = s[0];
            for (int i = 1; i < M; ++i) if (s[i] > mx) mx = s[i];
            double sum = 0.0;
            for (int i = 0; i < M; ++i) { s[i] = exp(s[i] - mx); sum += s[i]; }
            for (int i = 0; i < M; ++i) s[i] /= sum;
        }
        int best = 0;
        for (int i = 1; i < M; ++i) if (s[i] > s[best]) best = i;
        if (argmax) argmax[n] = best;
        if (maxval) maxval[n] = M > 0 ? s[best] : 0.0;
        if (S) memcpy(S + (size_t)n * M, s, sizeof(double) * (size_t)M);
        free(s);
    }
}

/*
 * Probability vectorization in Gram-loc (Sec. 2.2: a weighted sum of codebook
 * vectors with the attribute probabilities as weights; Sec. 3.1/3.3: computed
 * on Gram-loc).  V[n][j] = sum_i P[n][i] R[i][j], i.e. the Gram-loc of P C.
 */
void orc_prob_vectorize(const double* P, long N, int M, int ldp, const double* R, int ldr,
                        int r, double* V) {
    long n;
#pragma omp parallel for schedule(static)
    for (n = 0; n < N; ++n) {
        const double* p = P + (size_t)n * ldp;
        double* v = V + (size_t)n * r;
        for (int j = 0; j < r; ++j) {
            double acc = 0.0;
            for (int i = 0; i < M; ++i) acc += p[i] * R[(size_t)i * ldr + j];
            v[j] = acc;
        }
    }
}

/*
 * Reconstruction ("decompose", Sec. 3.1 and Sec. 3.3: x = U t).
 * Xhat[n][d] = sum_j T[n][j] Q[j][d].
 */
void orc_reconstruct(const double* T, long N, int r, int ldt, const double* Q, int D,
                     double* Xhat) {
    long n;
#pragma omp parallel for schedule(static)
    for (n = 0; n < N; ++n) {
        const double* t = T + (size_t)n * ldt;
        double* x = Xhat + (size_t)n * D;
        for (int d = 0; d < D; ++d) {
            double acc = 0.0;
            for (int j = 0; j < r; ++j) acc += t[j] * Q[(size_t)j * D + d];
            x[d] = acc;
        }
    }
}

/*
 * Binding / unbinding (Sec. 2.2: the component-wise operators of rule
 * execution, with a modulo-style index computation; Sec. 3.3: the operations
 * after reconstruction are based on circular convolution).  Each row is cut
 * into blocks of L consecutive components (L divides D; L = D is one circular
 * convolution over the whole vector) and, within block b,
 *   bind:   Z[n][bL + k] = sum_j X[n][bL + j] * Y[n'][bL + ((k - j) mod L)]
 *   unbind: Z[n][bL + k] = sum_j X[n][bL + j] * Y[n'][bL + ((j - k) mod L)]
 * (circular convolution, and circular correlation: binding with the involution
 * of Y, the approximate inverse of binding).  n' = n, or 0 when ldy = 0 (one
 * partner for every row).  Reading fixed here: the paper names neither the
 * block length nor the direction of the index; the block length is the
 * caller's, and unbind(bind(x, y), y) = x for partners y whose block DFTs have
 * unit modulus.
 */
void orc_bind(const double* X, long N, int D, int ldx, const double* Y, long ldy, int L, int op,
              double* Z) {
    long n;
#pragma omp parallel for schedule(static)
    for (n = 0; n < N; ++n) {
        const double* x = X + (size_t)n * ldx;
        const double* y = Y + (size_t)n * ldy;
        double* z = Z + (size_t)n * D;
        for (int b0 = 0; b0 < D; b0 += L) {
            for (int k = 0; k < L; ++k) {
                double acc = 0.0;
                for (int j = 0; j < L; ++j) {
                    int m = op == 0 ? k - j : j - k;
                    if (m < 0) m += L;
                    acc += x[b0 + j] * y[b0 + m];
                }
                z[b0 + k] = acc;
            }
        }
    }
}

/*
 * Attention scores between compressed vectors (Sec. 2.2 "attention score";
 * Sec. 3.2: attention scores that use matrix multiplication are preserved).
 * For each sequence b: L[q][k] = scale * <Yq[b][q], Yk[b][k]>; with
 * apply_softmax the row over the Lk keys is replaced by softmax(L[q][.]).
 */
void orc_attention(const double* Yq, const double* Yk, int B, int Lq, int Lk, int r,
                   double scale, int apply_softmax, double* A) {
    long bq;
    long total = (long)B * Lq;
#pragma omp parallel for schedule(static)
    for (bq = 0; bq < total; ++bq) {
        long b = bq / Lq;
        const double* q = Yq + (size_t)bq * r;
        const double* kb = Yk + (size_t)b * Lk * r;
        double* a = A + (size_t)bq * Lk;
        for (int k = 0; k < Lk; ++k) a[k] = scale * dot(q, kb + (size_t)k * r, r);
        if (apply_softmax && Lk > 0) {
            double mx = a[0];
            for (int k = 1; k < Lk; ++k) if (a[k] > mx) mx = a[k];
            double sum = 0.0;
            for (int k = 0; k < Lk; ++k) { a[k] = exp(a[k] - mx); sum += a[k]; }
            for (int k = 0; k < Lk; ++k) a[k] /= sum;
        }
    }
}

/*
 * Memory model (Sec. 3.1): original storage M*D values, Gram-Space storage
 * D*k + M*k values.  out[0] = coefficient ratio (M*D)/(M*k) = D/k, the ratio
 * the paper quotes (D/k >= 6.4 for M = 40, D = 256); out[1] = total ratio
 * (M*D)/(D*k + M*k).
 */
void orc_memory_ratios(long M, long D, long k, double* out) {
    out[0] = k > 0 ? (double)(M * D) / (double)(M * k) : 0.0;
    out[1] = k > 0 ? (double)(M * D) / (double)(D * k + M * k) : 0.0;
}
