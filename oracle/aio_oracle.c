/*
 * aio_oracle.c -- fp64 CPU oracle for the decode-step linear layers.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference leg of bench.py may load or call this library.
 * It shares no code with the CUDA path (no headers, no helpers, no tables).
 *
 * What it computes (the plain definition, one output at a time):
 *
 *   The paper's premise is that each decoded token streams every weight of
 *   every linear layer from HBM (Sec. 2.1; Sec. 3.1).  A decode-step linear
 *   layer maps token rows x[m, :] to y[m, n] = sum_k x[m, k] * W[n, k]
 *   (nn.Linear convention, y = x W^T), for M = 1 token (plain decoding) or
 *   M > 1 rows (prompt-lookup verification, Sec. 4.2).
 *
 *   W8A16 storage-only quantization (Sec. 2.4; Sec. 6.2) keeps int8 codes q
 *   and dequantizes them before the multiply.  Reading used here: one bf16
 *   scale per output channel n, symmetric codes, zero-point 0, and the exact
 *   product s[n] * q[n, k] (never rounded to 16 bits):
 *       y[m, n] = sum_k x[m, k] * (s[n] * q[n, k])
 *
 *   Every value is widened to double; the sum runs in ascending k with one
 *   double accumulator per output.  bf16 is decoded by placing its 16 bits in
 *   the upper half of an IEEE-754 binary32 word (bf16 is the upper half of
 *   binary32 by definition) and widening that float to double.
 *
 * Parallelism: OpenMP over output channels n only; each output's sum order is
 * fixed, so results do not depend on the thread count.
 *
 * The chained decoder step (the steps on either side of the linear layers):
 * the paper names its models (Sec. 4.2) but prints no block structure.  The
 * reading used here is a pre-norm decoder block whose shapes match the
 * projections: RMSNorm -> QKV -> attention -> O (+ residual) -> RMSNorm ->
 * gate+up -> SwiGLU -> down (+ residual), and a final RMSNorm before lm_head.
 * Attention over a context of one position (the token being decoded) gives
 * each head's value vector, so O reads the V third of the QKV output.  Every
 * buffer between steps has the precision the CUDA path stores: the residual
 * stream h and every y are fp32, every projection input x is bf16 (rounded to
 * nearest even from the exact value).  The arithmetic of each step is done in
 * double, from those stored values:
 *   rmsnorm:  h' = fp32(h + r);  x = bf16(h'[k] * g[k] / sqrt(mean(h'^2) + eps))
 *   swiglu:   x = bf16(silu(y[k]) * y[I + k]),  silu(t) = t / (1 + exp(-t))
 *   slice:    x = bf16(y[off + k])
 *
 * Decode attention over a KV cache (the long-context half of the paper's routing, Sec. 3.3,
 * Sec. 5.1: standard contexts up to 2K tokens, long ones up to 32K).  For each head h and new
 * token m of M (positions L - M + m of a cache holding L positions), with d-dimensional heads:
 *   s_j = q[m, h] . k[h, j] / sqrt(d)  for j <= L - M + m   (causal among the new tokens)
 *   out[m, h] = sum_j softmax(s)_j v[h, j]
 * in double, from fp32 q and bf16 cache entries.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#include <stddef.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Planted-mistake hook for the mutation tests (tests/test_oracle_mutants.py):
 * a nonzero AIO_ORACLE_MUTANT compiles a deliberately wrong oracle so the
 * tests can prove that the pins catch it.  The shipped build defines nothing. */
#ifndef AIO_ORACLE_MUTANT
#define AIO_ORACLE_MUTANT 0
#endif

double aio_oracle_bf16_to_double(uint16_t h) {
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

int aio_oracle_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* y[m*N + n] = sum_k bf16(x[m*K + k]) * bf16(W[n*K + k]) */
void aio_oracle_linear_bf16(const uint16_t* x, const uint16_t* W, int64_t M, int64_t K, int64_t N, double* y) {
#pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        const uint16_t* w = W + n * K;
        for (int64_t m = 0; m < M; ++m) {
            const uint16_t* xm = x + m * K;
            double acc = 0.0;
#if AIO_ORACLE_MUTANT == 1   /* dropped term: skips the last k */
            for (int64_t k = 0; k < K - 1; ++k)
#else
            for (int64_t k = 0; k < K; ++k)
#endif
            {
#if AIO_ORACLE_MUTANT == 2   /* transposed operand: W read as [K, N] */
                double wv = aio_oracle_bf16_to_double(W[k * N + n]);
                (void)w;
#else
                double wv = aio_oracle_bf16_to_double(w[k]);
#endif
                acc += aio_oracle_bf16_to_double(xm[k]) * wv;
            }
#if AIO_ORACLE_MUTANT == 3   /* wrong sign */
            acc = -acc;
#endif
            y[m * N + n] = acc;
        }
    }
}

/* y[m*N + n] = sum_k bf16(x[m*K + k]) * (bf16(s[n]) * q[n*K + k]) */
void aio_oracle_linear_i8(const uint16_t* x, const int8_t* q, const uint16_t* s, int64_t M, int64_t K, int64_t N,
                          double* y) {
#pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        const int8_t* qn = q + n * K;
#if AIO_ORACLE_MUTANT == 4   /* wrong scale index */
        double sn = aio_oracle_bf16_to_double(s[(n + 1) % N]);
#else
        double sn = aio_oracle_bf16_to_double(s[n]);
#endif
        for (int64_t m = 0; m < M; ++m) {
            const uint16_t* xm = x + m * K;
            double acc = 0.0;
            for (int64_t k = 0; k < K; ++k) {
#if AIO_ORACLE_MUTANT == 5   /* dequant rounded to bf16 before the product (the reading the oracle rejects) */
                double d = sn * (double)qn[k];
                float df = (float)d;
                uint32_t u;
                memcpy(&u, &df, 4);
                u += 0x7FFFu + ((u >> 16) & 1u);
                u &= 0xFFFF0000u;
                memcpy(&df, &u, 4);
                double wv = (double)df;
#elif AIO_ORACLE_MUTANT == 6   /* sign of the code lost */
                double wv = sn * (double)(qn[k] < 0 ? -qn[k] : qn[k]);
#else
                double wv = sn * (double)qn[k];
#endif
                acc += aio_oracle_bf16_to_double(xm[k]) * wv;
            }
            y[m * N + n] = acc;
        }
    }
}

/* Dequantized weights Wd[n*K + k] = bf16(s[n]) * q[n*K + k] in double (exact). */
void aio_oracle_dequant_i8(const int8_t* q, const uint16_t* s, int64_t N, int64_t K, double* Wd) {
#pragma omp parallel for schedule(static)
    for (int64_t n = 0; n < N; ++n) {
        double sn = aio_oracle_bf16_to_double(s[n]);
        for (int64_t k = 0; k < K; ++k) Wd[n * K + k] = sn * (double)q[n * K + k];
    }
}

/* ---------------------------------------------------------------- the chained decoder step */

/* bf16 bit pattern of the double v, rounded to nearest, ties to even (no intermediate float
 * rounding): v is rounded to a multiple of the bf16 quantum at its binade, 2^(e-8) for
 * v = f 2^e with f in [0.5, 1), and never below 2^-133 (bf16 subnormals).  The rounded value has
 * at most 8 significant bits, so converting it to float is exact. */
uint16_t aio_oracle_double_to_bf16(double v) {
    if (v != v) return 0x7FC0u;
    if (v == 0.0) return signbit(v) ? 0x8000u : 0x0000u;
    if (isinf(v)) return v < 0 ? 0xFF80u : 0x7F80u;
    int e;
    frexp(v, &e);
    int qe = e - 8;
    if (qe < -133) qe = -133;
#if AIO_ORACLE_MUTANT == 7   /* rounds toward zero instead of to nearest even */
    double r = ldexp(trunc(ldexp(v, -qe)), qe);
#else
    double r = ldexp(nearbyint(ldexp(v, -qe)), qe);   /* default rounding mode: nearest, ties to even */
#endif
    if (fabs(r) > 3.3895313892515355e38) return r < 0 ? 0xFF80u : 0x7F80u;   /* above the largest bf16 */
    float f = (float)r;
    uint32_t u;
    memcpy(&u, &f, 4);
    return (uint16_t)(u >> 16);
}

double aio_oracle_silu(double t) {
#if AIO_ORACLE_MUTANT == 8   /* wrong sign in the logistic */
    return t / (1.0 + exp(t));
#else
    return t / (1.0 + exp(-t));
#endif
}

/* Residual add and RMSNorm of M token rows of width K.  r may be NULL (no add); h_out may be NULL
 * (not stored).  h_out[m, k] = fp32(h_in + r), then x[m, k] = bf16(h_out * gamma[k] * inv_rms)
 * with inv_rms = 1 / sqrt(sum_k h_out^2 / K + eps), the sum in ascending k. */
void aio_oracle_rmsnorm(const float* h_in, const float* r, const uint16_t* gamma, int64_t M, int64_t K, double eps,
                        float* h_out, uint16_t* x) {
    for (int64_t m = 0; m < M; ++m) {
        double ss = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            float h = r ? (float)(h_in[m * K + k] + r[m * K + k]) : h_in[m * K + k];
            if (h_out) h_out[m * K + k] = h;
            ss += (double)h * (double)h;
        }
#if AIO_ORACLE_MUTANT == 9   /* mean over K - 1 */
        double inv = 1.0 / sqrt(ss / (double)(K - 1) + eps);
#else
        double inv = 1.0 / sqrt(ss / (double)K + eps);
#endif
        for (int64_t k = 0; k < K; ++k) {
            float h = r ? (float)(h_in[m * K + k] + r[m * K + k]) : h_in[m * K + k];
            x[m * K + k] = aio_oracle_double_to_bf16((double)h * aio_oracle_bf16_to_double(gamma[k]) * inv);
        }
    }
}

/* SwiGLU of the concatenated gate+up output: y is [M, stride] fp32 with the gate in columns
 * [0, I) and the up projection in [I, 2I); x[m, k] = bf16(silu(gate) * up), k < I. */
void aio_oracle_swiglu(const float* y, int64_t M, int64_t I, int64_t stride, uint16_t* x) {
    for (int64_t m = 0; m < M; ++m)
        for (int64_t k = 0; k < I; ++k) {
#if AIO_ORACLE_MUTANT == 10   /* gate and up swapped */
            double g = y[m * stride + I + k], u = y[m * stride + k];
#else
            double g = y[m * stride + k], u = y[m * stride + I + k];
#endif
            x[m * I + k] = aio_oracle_double_to_bf16(aio_oracle_silu(g) * u);
        }
}

/* Columns [off, off + K) of y [M, stride] as bf16: x[m, k] = bf16(y[m, off + k]). */
void aio_oracle_slice(const float* y, int64_t M, int64_t K, int64_t stride, int64_t off, uint16_t* x) {
    for (int64_t m = 0; m < M; ++m)
        for (int64_t k = 0; k < K; ++k) x[m * K + k] = aio_oracle_double_to_bf16((double)y[m * stride + off + k]);
}

/* ---------------------------------------------------------------- decode attention */

/* q [M, q_stride] fp32 (head h at columns [h d, h d + d)); k, v bf16 [n_heads][L_max][d];
 * out [M, n_heads d] double. */
void aio_oracle_attention(const float* q, int64_t q_stride, const uint16_t* k, const uint16_t* v, int64_t n_heads,
                          int64_t d, int64_t L_max, int64_t L, int64_t M, double* out) {
#pragma omp parallel for schedule(static) collapse(2)
    for (int64_t m = 0; m < M; ++m)
        for (int64_t h = 0; h < n_heads; ++h) {
#if AIO_ORACLE_MUTANT == 12   /* causal limit off by one: sees the next new token */
            int64_t last = L - M + m + 1 < L ? L - M + m + 1 : L - 1;
#else
            int64_t last = L - M + m;
#endif
#if AIO_ORACLE_MUTANT == 11   /* no 1/sqrt(d) scale */
            double scale = 1.0;
#else
            double scale = 1.0 / sqrt((double)d);
#endif
            const float* qm = q + m * q_stride + h * d;
            double mx = -INFINITY;
            for (int64_t j = 0; j <= last; ++j) {
                const uint16_t* kj = k + (h * L_max + j) * d;
                double s = 0.0;
                for (int64_t e = 0; e < d; ++e) s += (double)qm[e] * aio_oracle_bf16_to_double(kj[e]);
                s *= scale;
                if (s > mx) mx = s;
            }
            double* o = out + m * n_heads * d + h * d;
            for (int64_t e = 0; e < d; ++e) o[e] = 0.0;
            double sum = 0.0;
            for (int64_t j = 0; j <= last; ++j) {
                const uint16_t* kj = k + (h * L_max + j) * d;
                const uint16_t* vj = v + (h * L_max + j) * d;
                double s = 0.0;
                for (int64_t e = 0; e < d; ++e) s += (double)qm[e] * aio_oracle_bf16_to_double(kj[e]);
                double p = exp(s * scale - mx);
                sum += p;
                for (int64_t e = 0; e < d; ++e) o[e] += p * aio_oracle_bf16_to_double(vj[e]);
            }
#if AIO_ORACLE_MUTANT == 13   /* not normalised */
            (void)sum;
#else
            for (int64_t e = 0; e < d; ++e) o[e] /= sum;
#endif
        }
}
