/*
 * CPU oracle of the integer LayerNorm (Sec. 2.1, Eqs. 1-4; the integer
 * kernel of Sec. 2.2).  TEST INFRASTRUCTURE ONLY: see ipo_norm.h.
 *
 * LayerNorm(x)_i = gamma_i (x_i - mean) / sqrt(var + eps) + beta_i over the
 * d channels of one frame, on integers of the input grid: the centred values
 * are kept exactly as d (q_i - mean), the standard deviation is an integer
 * square root of their mean square, the division by it is one reciprocal
 * per row, and gamma, beta and the output grid fold into one dyadic
 * multiplier and offset per channel.
 */
#include "ipo_norm.h"

#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define IPO_OK 0
#define IPO_ERR_NULL (-1)
#define IPO_ERR_SHAPE (-2)
#define IPO_ERR_PARAM (-3)

/* floor(x / 2^n), 0 <= n <= 62, independent of the sign behaviour of >>. */
static int64_t norm_floor_pow2(int64_t x, int n) {
    int64_t dd = (int64_t)1 << n;
    if (x >= 0) return x / dd;
    return -((-x + dd - 1) / dd);
}

static int64_t norm_round_shift(int64_t x, int n) {
    return norm_floor_pow2(x + ((int64_t)1 << (n - 1)), n);
}

/* Newton's iteration on integers, started above the root: r_{k+1} =
 * floor((r_k + floor(n / r_k)) / 2) decreases while r_k > floor(sqrt(n)). */
int64_t ipo_isqrt(int64_t n) {
    if (n <= 0) return 0;
    int64_t r = (int64_t)1 << 31;          /* > sqrt(2^62) */
    for (;;) {
        int64_t next = (r + n / r) / 2;
        if (next >= r) return r;
        r = next;
    }
}

int ipo_layernorm_i8(const int8_t *x, long long rows, int d, int64_t eps_c, const int32_t *M,
                     const int64_t *B, const int32_t *E, int8_t *y) {
    if (rows < 0 || d < 2 || d > 4096) return IPO_ERR_SHAPE;
    if (rows == 0) return IPO_OK;
    if (!x || !M || !B || !E || !y) return IPO_ERR_NULL;
    if (eps_c < 0 || eps_c > ((int64_t)1 << 40)) return IPO_ERR_PARAM;
    for (int i = 0; i < d; ++i)
        if (E[i] < 31 || E[i] > 62 || B[i] >= ((int64_t)1 << 60) || B[i] <= -((int64_t)1 << 60))
            return IPO_ERR_PARAM;
#pragma omp parallel for schedule(static)
    for (long long r = 0; r < rows; ++r) {
        const int8_t *q = x + (size_t)r * d;
        int8_t *out = y + (size_t)r * d;
        int64_t sum = 0;
        for (int i = 0; i < d; ++i) sum += q[i];
        int64_t v = 0;
        for (int i = 0; i < d; ++i) {
            int64_t c = (int64_t)d * q[i] - sum;
            v += c * c;
        }
        int64_t sigma = ipo_isqrt(v / d + eps_c);
        if (sigma < 1) sigma = 1;
        int64_t f = ((int64_t)1 << 31) / sigma;
        for (int i = 0; i < d; ++i) {
            int64_t c = (int64_t)d * q[i] - sum;
            int64_t n = norm_round_shift(c * f, 16);
            int64_t t = norm_round_shift((int64_t)M[i] * n + B[i], E[i]);
            if (t > 127) t = 127;
            if (t < -127) t = -127;
            out[i] = (int8_t)t;
        }
    }
    return IPO_OK;
}
