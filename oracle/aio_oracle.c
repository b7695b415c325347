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
 */
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
