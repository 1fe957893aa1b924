/*
 * resbm_oracle.c -- plain fp64 CPU oracle of the ResBM boundary bottleneck.
 *
 * TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU
 * baseline leg may load this library. The product path (the CUDA library and
 * its Python binding) never calls it, and the two share no code.
 *
 * What it computes (all tensors fp64, row-major, "x . W" orientation of the
 * paper, Sec. 3.1 Eq. 1 and Eq. generalized_transformer_equation):
 *
 *   Rectangular identity   [I_{c x C}]_{ij} = 1 iff i == j      (Eq. rect_identity_definition)
 *   Identity projection    P^id(x) = x . I_{c x C}              (Eq. Pid_definition)
 *   Encoder (Sec. 3.2)     b = E(z) = phi(z . We1) . We2         two linear layers, one nonlinearity
 *   Decoder (Sec. 3.2)     z~ = D(b) = phi(b . Wd1) . Wd2
 *   Send side (Sec. 3.2 "Preserving the identity path", Eq. generalized_transformer_equation):
 *                          B = P^id(X; d -> r) + E(F)            X = x_l^Attn, F = z_l (FF output)
 *   Receive side           Y = P^id(B; r -> d) + D(B)            (merge = 1)
 *                          Y = D(B)                              (merge = 0: the caller adds the
 *                                                                 padded skip after attention)
 *   Backward               the chain rule of the above for the scalar  sum(dY * Y)  (decoder) and
 *                          sum(dB * B) (encoder); a gradient through y = x . M is dx = dy . M^T.
 *   Transfer rounding      B and dB cross the boundary in the transfer dtype (Appendix A.3 counts
 *                          them in bf16): oracle_round_array rounds them, nearest-even, before
 *                          the receiving side uses them.
 *
 * Readings where the paper is silent (listed with the same numbers in the design notes):
 *   - hidden width m of the two-layer encoder/decoder is a free argument (Sec. 3.2 does not fix it);
 *   - phi is SiLU by default, GELU(tanh) and identity selectable (Sec. 3.2 names no nonlinearity);
 *   - no biases; no normalisation inside the bottleneck;
 *   - P^id keeps the FIRST columns when truncating and zero-pads AFTER them (Eq. Pid bullets).
 *
 * Every matrix product is the textbook triple loop; every reduction runs over its summation
 * index in natural order. OpenMP only splits independent output rows between threads, so the
 * result does not depend on the thread count.
 *
 * Pins (tests/test_oracle_pins.py): the P^id truncate / pad / identity cases and the
 * composition-of-identities rank statement (Sec. 3.3), the zero-weight identity-path cases,
 * the byte counts of Appendix A.3, central finite differences for every gradient, the
 * act = identity case against numpy's matmul, and the activation derivatives against
 * finite differences.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORACLE_ACT_SILU = 0, ORACLE_ACT_GELU_TANH = 1, ORACLE_ACT_IDENTITY = 2 };

int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Number of OpenMP threads later calls use (results do not depend on it). */
void oracle_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ------------------------------------------------------------------------------------------ */
/* Nonlinearity phi and its derivative (Sec. 3.2: "a non-linearity applied between them").      */
/* SiLU: x * sigmoid(x).  GELU(tanh form): 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3))).      */
/* ------------------------------------------------------------------------------------------ */

static const double kSqrt2OverPi = 0.79788456080286535587989211986876;
static const double kGeluC = 0.044715;

double oracle_act(int act, double x)
{
    if (act == ORACLE_ACT_SILU) {
        double s = 1.0 / (1.0 + exp(-x));
        return x * s;
    }
    if (act == ORACLE_ACT_GELU_TANH) {
        double u = kSqrt2OverPi * (x + kGeluC * x * x * x);
        return 0.5 * x * (1.0 + tanh(u));
    }
    return x;
}

double oracle_dact(int act, double x)
{
    if (act == ORACLE_ACT_SILU) {
        /* d/dx [x s(x)] = s(x) + x s(x) (1 - s(x)) */
        double s = 1.0 / (1.0 + exp(-x));
        return s + x * s * (1.0 - s);
    }
    if (act == ORACLE_ACT_GELU_TANH) {
        double u = kSqrt2OverPi * (x + kGeluC * x * x * x);
        double th = tanh(u);
        double du = kSqrt2OverPi * (1.0 + 3.0 * kGeluC * x * x);
        return 0.5 * (1.0 + th) + 0.5 * x * (1.0 - th * th) * du;
    }
    return 1.0;
}

/* ------------------------------------------------------------------------------------------ */
/* Plain matrix products (row-major).                                                           */
/* ------------------------------------------------------------------------------------------ */

/* Z[M x N] = A[M x K] . B[K x N] */
static void mm_nn(int64_t M, int64_t N, int64_t K, const double *A, const double *B, double *Z)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        double *z = Z + i * N;
        for (int64_t j = 0; j < N; ++j) z[j] = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            const double a = A[i * K + k];
            const double *b = B + k * N;
            for (int64_t j = 0; j < N; ++j) z[j] += a * b[j];
        }
    }
}

/* Z[M x N] = A[M x K] . B^T, with B stored N x K */
static void mm_nt(int64_t M, int64_t N, int64_t K, const double *A, const double *B, double *Z)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        for (int64_t j = 0; j < N; ++j) {
            double acc = 0.0;
            for (int64_t k = 0; k < K; ++k) acc += A[i * K + k] * B[j * K + k];
            Z[i * N + j] = acc;
        }
    }
}

/* Z[M x N] = A^T . B, with A stored K x M and B stored K x N; the sum over k (the token
 * index for the weight gradients) runs k = 0, 1, ..., K-1 for every output element. */
static void mm_tn(int64_t M, int64_t N, int64_t K, const double *A, const double *B, double *Z)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        double *z = Z + i * N;
        for (int64_t j = 0; j < N; ++j) z[j] = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            const double a = A[k * M + i];
            const double *b = B + k * N;
            for (int64_t j = 0; j < N; ++j) z[j] += a * b[j];
        }
    }
}

/* ------------------------------------------------------------------------------------------ */
/* Rounding of the tensors that cross the boundary. Appendix A.3 counts the forward activation  */
/* b_l and the backward gradient d b_l in bf16: what the receiving side consumes is the value   */
/* rounded to the transfer dtype. Both roundings are to nearest, ties to even, taken directly    */
/* from the fp64 value (no intermediate fp32 rounding).                                         */
/* ------------------------------------------------------------------------------------------ */

/* Round x to `bits` significant bits (bf16: 8, fp32: 24), nearest-even; normal range only. */
static double round_significand(double x, int bits)
{
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    double f = frexp(x, &e);                 /* x = f * 2^e, 0.5 <= |f| < 1 */
    double scaled = ldexp(f, bits);          /* exact: |scaled| in [2^(bits-1), 2^bits) */
    double r = nearbyint(scaled);            /* default rounding mode: to nearest, ties to even */
    return ldexp(r, e - bits);
}

void oracle_round_array(int dtype_bits, int64_t n, double *x)
{
    for (int64_t i = 0; i < n; ++i) x[i] = round_significand(x[i], dtype_bits);
}

static double *alloc_d(int64_t n)
{
    return (double *)malloc((size_t)(n > 0 ? n : 1) * sizeof(double));
}

/* ------------------------------------------------------------------------------------------ */
/* Sec. 3.3: rectangular identity and the identity projection.                                  */
/* ------------------------------------------------------------------------------------------ */

/* Eq. rect_identity_definition: I is c x C with I[i][j] = 1 iff i == j. */
void oracle_rect_identity(int64_t c, int64_t C, double *I)
{
    for (int64_t i = 0; i < c; ++i)
        for (int64_t j = 0; j < C; ++j) I[i * C + j] = (i == j) ? 1.0 : 0.0;
}

/* Eq. Pid_definition: y = x . I_{c x C} for x in R^{L x c}; y in R^{L x C}. */
int oracle_pid(int64_t L, int64_t c, int64_t C, const double *x, double *y)
{
    double *I = alloc_d(c * C);
    if (!I) return -1;
    oracle_rect_identity(c, C, I);
    mm_nn(L, C, c, x, I, y);
    free(I);
    return 0;
}

/* Gradient through y = x . I_{c x C}: dx = dy . I_{c x C}^T (dx in R^{L x c}). */
static int pid_backward(int64_t L, int64_t c, int64_t C, const double *dy, double *dx)
{
    double *I = alloc_d(c * C);
    if (!I) return -1;
    oracle_rect_identity(c, C, I);
    mm_nt(L, c, C, dy, I, dx); /* I stored c x C == (C x c)^T rows: Z = dy . I^T */
    free(I);
    return 0;
}

static void apply_act(int act, int64_t n, const double *x, double *y)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) y[i] = oracle_act(act, x[i]);
}

/* ------------------------------------------------------------------------------------------ */
/* Send side (encoder at the end of block l, Sec. 3.2).                                         */
/*   S = X . I_{d x r};  P = F . We1;  A = phi(P);  E = A . We2;  B = S + E.                     */
/* X: T x d, F: T x d, We1: d x m, We2: m x r -> B: T x r, P (optional, may be NULL): T x m.     */
/* ------------------------------------------------------------------------------------------ */
int oracle_encode_fwd(int64_t T, int64_t d, int64_t r, int64_t m, int act,
                      const double *X, const double *F, const double *We1, const double *We2,
                      double *B, double *P_out)
{
    double *S = alloc_d(T * r), *P = alloc_d(T * m), *A = alloc_d(T * m), *E = alloc_d(T * r);
    int rc = (S && P && A && E) ? 0 : -1;
    if (rc == 0) rc = oracle_pid(T, d, r, X, S);
    if (rc == 0) {
        mm_nn(T, m, d, F, We1, P);
        apply_act(act, T * m, P, A);
        mm_nn(T, r, m, A, We2, E);
        for (int64_t i = 0; i < T * r; ++i) B[i] = S[i] + E[i];
        if (P_out) memcpy(P_out, P, (size_t)(T * m) * sizeof(double));
    }
    free(S); free(P); free(A); free(E);
    return rc;
}

/* ------------------------------------------------------------------------------------------ */
/* Receive side (decoder at the start of block l+1, Sec. 3.2).                                  */
/*   Q = B . Wd1;  G = phi(Q);  D = G . Wd2;  Y = merge ? B . I_{r x d} + D : D.                 */
/* B: T x r, Wd1: r x m, Wd2: m x d -> Y: T x d.                                                 */
/* ------------------------------------------------------------------------------------------ */
int oracle_decode_fwd(int64_t T, int64_t d, int64_t r, int64_t m, int act, int merge,
                      const double *B, const double *Wd1, const double *Wd2, double *Y)
{
    double *Q = alloc_d(T * m), *G = alloc_d(T * m), *D = alloc_d(T * d);
    double *R = merge ? alloc_d(T * d) : NULL;
    int rc = (Q && G && D && (!merge || R)) ? 0 : -1;
    if (rc == 0) {
        mm_nn(T, m, r, B, Wd1, Q);
        apply_act(act, T * m, Q, G);
        mm_nn(T, d, m, G, Wd2, D);
        if (merge) rc = oracle_pid(T, r, d, B, R);
    }
    if (rc == 0) {
        for (int64_t i = 0; i < T * d; ++i) Y[i] = merge ? R[i] + D[i] : D[i];
    }
    free(Q); free(G); free(D); free(R);
    return rc;
}

/* ------------------------------------------------------------------------------------------ */
/* Decoder backward for the upstream gradient dY of Y (chain rule of oracle_decode_fwd):        */
/*   dWd2 = G^T . dY;  dG = dY . Wd2^T;  dQ = dG * phi'(Q);  dWd1 = B^T . dQ;                    */
/*   dB = dQ . Wd1^T + merge * dY . I_{r x d}^T.                                                 */
/* dY: T x d, B: T x r -> dB: T x r, dWd1: r x m, dWd2: m x d.                                    */
/* ------------------------------------------------------------------------------------------ */
int oracle_decode_bwd(int64_t T, int64_t d, int64_t r, int64_t m, int act, int merge,
                      const double *dY, const double *B, const double *Wd1, const double *Wd2,
                      double *dB, double *dWd1, double *dWd2)
{
    double *Q = alloc_d(T * m), *G = alloc_d(T * m), *dG = alloc_d(T * m), *dQ = alloc_d(T * m);
    double *dBskip = alloc_d(T * r);
    int rc = (Q && G && dG && dQ && dBskip) ? 0 : -1;
    if (rc == 0) {
        mm_nn(T, m, r, B, Wd1, Q);               /* forward recomputed */
        apply_act(act, T * m, Q, G);
        mm_tn(m, d, T, G, dY, dWd2);             /* dWd2 = G^T . dY        */
        mm_nt(T, m, d, dY, Wd2, dG);             /* dG   = dY . Wd2^T      */
        for (int64_t i = 0; i < T * m; ++i) dQ[i] = dG[i] * oracle_dact(act, Q[i]);
        mm_tn(r, m, T, B, dQ, dWd1);             /* dWd1 = B^T . dQ        */
        mm_nt(T, r, m, dQ, Wd1, dB);             /* dB   = dQ . Wd1^T      */
        if (merge) {
            rc = pid_backward(T, r, d, dY, dBskip); /* dY . I_{r x d}^T     */
            if (rc == 0)
                for (int64_t i = 0; i < T * r; ++i) dB[i] += dBskip[i];
        }
    }
    free(Q); free(G); free(dG); free(dQ); free(dBskip);
    return rc;
}

/* ------------------------------------------------------------------------------------------ */
/* Encoder backward for the upstream gradient dB of B (chain rule of oracle_encode_fwd):        */
/*   dWe2 = A^T . dB;  dA = dB . We2^T;  dP = dA * phi'(P);  dWe1 = F^T . dP;  dF = dP . We1^T;  */
/*   dX = dB . I_{d x r}^T  (the full T x d gradient of X: dB in the first r columns, 0 after).  */
/* dB: T x r, F: T x d -> dF: T x d, dX: T x d (may be NULL), dWe1: d x m, dWe2: m x r.           */
/* ------------------------------------------------------------------------------------------ */
int oracle_encode_bwd(int64_t T, int64_t d, int64_t r, int64_t m, int act,
                      const double *dB, const double *F, const double *We1, const double *We2,
                      double *dF, double *dX, double *dWe1, double *dWe2)
{
    double *P = alloc_d(T * m), *A = alloc_d(T * m), *dA = alloc_d(T * m), *dP = alloc_d(T * m);
    int rc = (P && A && dA && dP) ? 0 : -1;
    if (rc == 0) {
        mm_nn(T, m, d, F, We1, P);               /* forward recomputed */
        apply_act(act, T * m, P, A);
        mm_tn(m, r, T, A, dB, dWe2);             /* dWe2 = A^T . dB        */
        mm_nt(T, m, r, dB, We2, dA);             /* dA   = dB . We2^T      */
        for (int64_t i = 0; i < T * m; ++i) dP[i] = dA[i] * oracle_dact(act, P[i]);
        mm_tn(d, m, T, F, dP, dWe1);             /* dWe1 = F^T . dP        */
        mm_nt(T, d, m, dP, We1, dF);             /* dF   = dP . We1^T      */
        if (dX) rc = pid_backward(T, d, r, dB, dX); /* dB . I_{d x r}^T     */
    }
    free(P); free(A); free(dA); free(dP);
    return rc;
}

/* ------------------------------------------------------------------------------------------ */
/* One linear layer per side (the single-matrix special case of the Sec. 3.2 encoder and       */
/* decoder; no nonlinearity):                                                                   */
/*   send:     B = X . I_{d x r} + F . We          We: d x r                                    */
/*   receive:  Y = merge ? B . I_{r x d} + B . Wd : B . Wd          Wd: r x d                   */
/*   backward: dB = B-gradient of sum(dY * Y) = merge * dY . I_{r x d}^T + dY . Wd^T;           */
/*             dWd = B^T . dY;  dF = dB . We^T;  dWe = F^T . dB;  dX = dB . I_{d x r}^T.          */
/* ------------------------------------------------------------------------------------------ */
int oracle_linear_encode_fwd(int64_t T, int64_t d, int64_t r, const double *X, const double *F,
                             const double *We, double *B)
{
    double *S = alloc_d(T * r), *L = alloc_d(T * r);
    int rc = (S && L) ? 0 : -1;
    if (rc == 0) rc = oracle_pid(T, d, r, X, S);
    if (rc == 0) {
        mm_nn(T, r, d, F, We, L);                /* L = F . We             */
        for (int64_t i = 0; i < T * r; ++i) B[i] = S[i] + L[i];
    }
    free(S); free(L);
    return rc;
}

int oracle_linear_decode_fwd(int64_t T, int64_t d, int64_t r, int merge, const double *B,
                             const double *Wd, double *Y)
{
    double *L = alloc_d(T * d), *Pad = merge ? alloc_d(T * d) : NULL;
    int rc = (L && (!merge || Pad)) ? 0 : -1;
    if (rc == 0) {
        mm_nn(T, d, r, B, Wd, L);                /* L = B . Wd             */
        if (merge) rc = oracle_pid(T, r, d, B, Pad);
    }
    if (rc == 0)
        for (int64_t i = 0; i < T * d; ++i) Y[i] = merge ? Pad[i] + L[i] : L[i];
    free(L); free(Pad);
    return rc;
}

int oracle_linear_decode_bwd(int64_t T, int64_t d, int64_t r, int merge, const double *dY,
                             const double *B, const double *Wd, double *dB, double *dWd)
{
    double *dBskip = alloc_d(T * r);
    int rc = dBskip ? 0 : -1;
    if (rc == 0) {
        mm_tn(r, d, T, B, dY, dWd);              /* dWd = B^T . dY          */
        mm_nt(T, r, d, dY, Wd, dB);              /* dB  = dY . Wd^T         */
        if (merge == 1) {                        /* + dY . I_{r x d}^T      */
            rc = pid_backward(T, r, d, dY, dBskip);
            if (rc == 0)
                for (int64_t i = 0; i < T * r; ++i) dB[i] += dBskip[i];
        }
    }
    free(dBskip);
    return rc;
}

int oracle_linear_encode_bwd(int64_t T, int64_t d, int64_t r, const double *dB, const double *F,
                             const double *We, double *dF, double *dX, double *dWe)
{
    mm_tn(d, r, T, F, dB, dWe);                  /* dWe = F^T . dB          */
    mm_nt(T, d, r, dB, We, dF);                  /* dF  = dB . We^T         */
    return dX ? pid_backward(T, d, r, dB, dX) : 0;
}
