/*
 * cola_oracle.c -- plain, slow, fp64 CPU oracle for the CoLA auto-encoder layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  The CUDA
 * product path never links, loads or calls it, and it shares no code, header,
 * table or helper with the CUDA path.
 *
 * What it computes (CoLA, arXiv 2502.10940):
 *   forward, Sec. 3.2 Eq. (main-fwd):  h = B sigma(A x),  A in R^{r x d_in},
 *     B in R^{d_out x r}.  Stored token-major (row t = token t):
 *       Z[t,i] = sum_k X[t,k] A[i,k]           (the rank-r activation A x)
 *       H[t,i] = sigma(Z[t,i])
 *       Y[t,o] = sum_i H[t,i] B[o,i]
 *   backward, Sec. 3.4 ("2x rule": grad_x = W^T grad_h, grad_W = grad_h x^T,
 *     applied to each of the two products, chain rule through sigma):
 *       dH[t,i] = sum_o dY[t,o] B[o,i]
 *       dZ[t,i] = dH[t,i] * sigma'(Z[t,i])
 *       dB[o,i] = sum_t dY[t,o] H[t,i]
 *       dA[i,k] = sum_t dZ[t,i] X[t,k]
 *       dX[t,k] = sum_i dZ[t,i] A[i,k]
 *   CoLA-M (Sec. 4.2, App. C) saves only the low-rank activation; the
 *   backward then recomputes H = sigma(Z) from the saved Z.
 *
 * Every sum runs in natural index order in fp64.  sigma in {identity, SiLU
 * (Swish, beta = 1), GELU (erf form)}; the paper names GeLU and Swish
 * (Sec. 5.2) without fixing their form.
 *
 * round_store != 0 rounds the stored low-rank tensors Z, H and dZ to the
 * bf16 grid (round to nearest, ties to even) at the point where they are
 * stored, with H = sigma(bf16(Z)) and dZ = bf16(dH * sigma'(bf16(Z))).  With
 * round_store == 0 everything stays in fp64.
 *
 * Inputs of the full routines are double arrays; inputs of the sampled
 * routines (meant for large shapes) are bf16 bit patterns (uint16) that are
 * widened exactly to double.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { ORC_SIGMA_IDENTITY = 0, ORC_SIGMA_SILU = 1, ORC_SIGMA_GELU = 2 };
enum { ORC_MODE_COLA = 0, ORC_MODE_COLA_M = 1 };

/* ---- activation and its derivative (from their mathematical definitions) ---- */

double oracle_sigma(int kind, double z)
{
    switch (kind) {
    case ORC_SIGMA_SILU: /* z * logistic(z) */
        return z / (1.0 + exp(-z));
    case ORC_SIGMA_GELU: /* z * Phi(z), Phi the standard normal CDF, via erfc
                            (no cancellation in the left tail) */
        return 0.5 * z * erfc(-z / sqrt(2.0));
    default:
        return z;
    }
}

double oracle_dsigma(int kind, double z)
{
    switch (kind) {
    case ORC_SIGMA_SILU: {
        /* d/dz [z s(z)] = s + z s (1 - s),  s = 1 / (1 + e^{-z}) */
        double s = 1.0 / (1.0 + exp(-z));
        return s * (1.0 + z * (1.0 - s));
    }
    case ORC_SIGMA_GELU: {
        /* d/dz [z Phi(z)] = Phi(z) + z phi(z) */
        double Phi = 0.5 * erfc(-z / sqrt(2.0));
        double phi = exp(-0.5 * z * z) / sqrt(2.0 * M_PI);
        return Phi + z * phi;
    }
    default:
        return 1.0;
    }
}

/* Round a double to the nearest bf16 value (8 significant bits, binary32
 * exponent range), ties to even, written from the format's definition. */
double oracle_round_bf16(double x)
{
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    frexp(x, &e);              /* |x| in [2^(e-1), 2^e) */
    int ex = e - 1;
    if (ex < -126) ex = -126;  /* bf16 subnormals share one quantum */
    double q = ldexp(1.0, ex - 7);
    double y = nearbyint(x / q) * q; /* default rounding mode: ties to even */
    if (fabs(y) > 3.3895313892515355e38) y = copysign(INFINITY, x);
    return y;
}

static double widen_bf16(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double st(int round_store, double v) { return round_store ? oracle_round_bf16(v) : v; }

void oracle_sigma_vec(int kind, const double* z, double* out, long m)
{
    for (long j = 0; j < m; ++j) out[j] = oracle_sigma(kind, z[j]);
}

void oracle_dsigma_vec(int kind, const double* z, double* out, long m)
{
    for (long j = 0; j < m; ++j) out[j] = oracle_dsigma(kind, z[j]);
}

void oracle_round_bf16_vec(const double* x, double* out, long m)
{
    for (long j = 0; j < m; ++j) out[j] = oracle_round_bf16(x[j]);
}

/* ---- full forward: Eq. (main-fwd) ---- */
void oracle_fwd(long n, long d_in, long d_out, long r, int sigma, int round_store,
                const double* X, const double* A, const double* B,
                double* Z, double* H, double* Y)
{
#pragma omp parallel for schedule(static)
    for (long t = 0; t < n; ++t) {
        for (long i = 0; i < r; ++i) {
            double s = 0.0;
            for (long k = 0; k < d_in; ++k) s += X[t * d_in + k] * A[i * d_in + k];
            s = st(round_store, s);
            Z[t * r + i] = s;
            H[t * r + i] = st(round_store, oracle_sigma(sigma, s));
        }
        for (long o = 0; o < d_out; ++o) {
            double s = 0.0;
            for (long i = 0; i < r; ++i) s += H[t * r + i] * B[o * r + i];
            Y[t * d_out + o] = s;
        }
    }
}

/* ---- full backward: Sec. 3.4 two-GEMM rule applied to both products ----
 * Zs: the saved Z.  Hs: the saved H (CoLA); ignored and recomputed as
 * sigma(Zs) under CoLA-M.  dZ (out, [n x r]) is the gradient at Z. */
void oracle_bwd(long n, long d_in, long d_out, long r, int sigma, int mode, int round_store,
                const double* X, const double* A, const double* B, const double* dY,
                const double* Zs, const double* Hs,
                double* dX, double* dA, double* dB, double* dZ)
{
    double* Hb = (double*)malloc(sizeof(double) * (size_t)(n * r));
    if (mode == ORC_MODE_COLA_M || Hs == NULL) {
        for (long j = 0; j < n * r; ++j) Hb[j] = st(round_store, oracle_sigma(sigma, Zs[j]));
    } else {
        memcpy(Hb, Hs, sizeof(double) * (size_t)(n * r));
    }

#pragma omp parallel for schedule(static)
    for (long t = 0; t < n; ++t) {
        for (long i = 0; i < r; ++i) {
            double dh = 0.0;
            for (long o = 0; o < d_out; ++o) dh += dY[t * d_out + o] * B[o * r + i];
            dZ[t * r + i] = st(round_store, dh * oracle_dsigma(sigma, Zs[t * r + i]));
        }
    }

    /* dB[o,:] accumulates over t in natural order */
#pragma omp parallel for schedule(static)
    for (long o = 0; o < d_out; ++o) {
        double* row = dB + o * r;
        for (long i = 0; i < r; ++i) row[i] = 0.0;
        for (long t = 0; t < n; ++t) {
            double a = dY[t * d_out + o];
            for (long i = 0; i < r; ++i) row[i] += a * Hb[t * r + i];
        }
    }

#pragma omp parallel for schedule(static)
    for (long i = 0; i < r; ++i) {
        double* row = dA + i * d_in;
        for (long k = 0; k < d_in; ++k) row[k] = 0.0;
        for (long t = 0; t < n; ++t) {
            double a = dZ[t * r + i];
            for (long k = 0; k < d_in; ++k) row[k] += a * X[t * d_in + k];
        }
    }

#pragma omp parallel for schedule(static)
    for (long t = 0; t < n; ++t) {
        for (long k = 0; k < d_in; ++k) {
            double s = 0.0;
            for (long i = 0; i < r; ++i) s += dZ[t * r + i] * A[i * d_in + k];
            dX[t * d_in + k] = s;
        }
    }
    free(Hb);
}

/* ---- CoLA-M block-level recompute (Sec. 4.2, App. C) ----
 * In the backward, CoLA-M rebuilds a layer output from the saved low-rank
 * activation instead of keeping it: H = sigma(Z) elementwise, then
 * Y[t,o] = sum_i H[t,i] B[o,i], the forward's second product. */
void oracle_recompute_up(long n, long d_out, long r, int sigma, const double* Z, const double* B, double* Y)
{
    double* H = (double*)malloc(sizeof(double) * (size_t)(n * r));
    for (long j = 0; j < n * r; ++j) H[j] = oracle_sigma(sigma, Z[j]);
#pragma omp parallel for schedule(static)
    for (long t = 0; t < n; ++t) {
        for (long o = 0; o < d_out; ++o) {
            double s = 0.0;
            for (long i = 0; i < r; ++i) s += H[t * r + i] * B[o * r + i];
            Y[t * d_out + o] = s;
        }
    }
    free(H);
}

/* ---- gated MLP (Fig. 4; Sec. 3.2; App. E) ----
 * LLaMA's MLP multiplies its gate and up projections element-wise before the
 * down projection; CoLA replaces both projections by auto-encoder layers and
 * keeps the product (and no full-rank activation on the gate branch):
 *   M = Y_gate (.) Y_up,   and for L = sum dM (.) M:
 *   dY_gate = dM (.) Y_up,  dY_up = dM (.) Y_gate. */
void oracle_gate_up_product(long m, const double* Yg, const double* Yu, double* M)
{
    for (long j = 0; j < m; ++j) M[j] = Yg[j] * Yu[j];
}

void oracle_gate_up_backward(long m, const double* dM, const double* Yg, const double* Yu, double* dYg, double* dYu)
{
    for (long j = 0; j < m; ++j) {
        dYg[j] = dM[j] * Yu[j];
        dYu[j] = dM[j] * Yg[j];
    }
}

/* ---- sampled routines on bf16 inputs (large shapes) ----
 * X[t,k] at X[t*ld_x + k]; dY[t,o] at dY[t*ld_y + o]; A [r x d_in] and
 * B [d_out x r] dense.  Each routine computes only the requested outputs,
 * each one exactly as the full routines define it. */

static double zval(long d_in, const uint16_t* X, long ld_x, const uint16_t* A, long t, long i)
{
    double s = 0.0;
    for (long k = 0; k < d_in; ++k) s += widen_bf16(X[t * ld_x + k]) * widen_bf16(A[i * d_in + k]);
    return s;
}

static double dhval(long d_out, long r, const uint16_t* dY, long ld_y, const uint16_t* B, long t, long i)
{
    double s = 0.0;
    for (long o = 0; o < d_out; ++o) s += widen_bf16(dY[t * ld_y + o]) * widen_bf16(B[o * r + i]);
    return s;
}

/* Token rows of Z, H, Y (forward) and dZ, dX (backward) for the listed tokens.
 * Outputs: Z,H,dZ [nrows x r]; Y [nrows x d_out]; dX [nrows x d_in].
 * dY may be NULL (then dZ, dX are not written). */
void oracle_rows_bf16(long d_in, long d_out, long r, int sigma, int round_store,
                      const uint16_t* X, long ld_x, const uint16_t* A, const uint16_t* B,
                      const uint16_t* dY, long ld_y, long nrows, const long* rows,
                      double* Z, double* H, double* Y, double* dZ, double* dX)
{
#pragma omp parallel for schedule(dynamic)
    for (long j = 0; j < nrows; ++j) {
        long t = rows[j];
        for (long i = 0; i < r; ++i) {
            double z = st(round_store, zval(d_in, X, ld_x, A, t, i));
            Z[j * r + i] = z;
            H[j * r + i] = st(round_store, oracle_sigma(sigma, z));
        }
        for (long o = 0; o < d_out; ++o) {
            double s = 0.0;
            for (long i = 0; i < r; ++i) s += H[j * r + i] * widen_bf16(B[o * r + i]);
            Y[j * d_out + o] = s;
        }
        if (dY) {
            for (long i = 0; i < r; ++i) {
                double dh = dhval(d_out, r, dY, ld_y, B, t, i);
                dZ[j * r + i] = st(round_store, dh * oracle_dsigma(sigma, Z[j * r + i]));
            }
            for (long k = 0; k < d_in; ++k) {
                double s = 0.0;
                for (long i = 0; i < r; ++i) s += dZ[j * r + i] * widen_bf16(A[i * d_in + k]);
                dX[j * d_in + k] = s;
            }
        }
    }
}

/* Entries dA[ii[e], kk[e]] = sum_t dZ[t,ii[e]] X[t,kk[e]], over all n tokens. */
void oracle_dA_entries_bf16(long n, long d_in, long d_out, long r, int sigma, int round_store,
                            const uint16_t* X, long ld_x, const uint16_t* A, const uint16_t* B,
                            const uint16_t* dY, long ld_y, long nent, const long* ii,
                            const long* kk, double* out)
{
#pragma omp parallel for schedule(dynamic)
    for (long e = 0; e < nent; ++e) {
        long i = ii[e], k = kk[e];
        double s = 0.0;
        for (long t = 0; t < n; ++t) {
            double z = st(round_store, zval(d_in, X, ld_x, A, t, i));
            double dz = st(round_store, dhval(d_out, r, dY, ld_y, B, t, i) * oracle_dsigma(sigma, z));
            s += dz * widen_bf16(X[t * ld_x + k]);
        }
        out[e] = s;
    }
}

/* Entries dB[oo[e], ii[e]] = sum_t dY[t,oo[e]] H[t,ii[e]], over all n tokens. */
void oracle_dB_entries_bf16(long n, long d_in, long r, int sigma, int round_store,
                            const uint16_t* X, long ld_x, const uint16_t* A,
                            const uint16_t* dY, long ld_y, long nent, const long* oo,
                            const long* ii, double* out)
{
    (void)r;
#pragma omp parallel for schedule(dynamic)
    for (long e = 0; e < nent; ++e) {
        long o = oo[e], i = ii[e];
        double s = 0.0;
        for (long t = 0; t < n; ++t) {
            double z = st(round_store, zval(d_in, X, ld_x, A, t, i));
            double h = st(round_store, oracle_sigma(sigma, z));
            s += widen_bf16(dY[t * ld_y + o]) * h;
        }
        out[e] = s;
    }
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}
