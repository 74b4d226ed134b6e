/*
 * CPU oracle of the integer linear layer (I-Parakeet, Sec. 2.2).  TEST
 * INFRASTRUCTURE ONLY: see ipo_linear.h.
 *
 * Plain scalar int64 code in the order the paper states it:
 *   Eq. 6  every tensor on a symmetric grid, q = round(clip(x) / S)
 *          (int8: [-127, 127]); weights with one scale per output channel
 *   Eq. 7  q_y = round(2^-n m q_W q_x): the integer product accumulates
 *          exactly (INT32 on the device), then one integer multiplication
 *          by m and one rounding right shift by n = 31 + s onto the int8
 *          grid of y.  A bias, where the layer has one, is an integer on
 *          the accumulator's grid S_W S_x and is added before the shift.
 *   Eqs. 12-13  Swish sw(x) = x sigma(x) = x (1 + tanh(x / 2)) / 2 with
 *          tanh(u) ~ sgn(u) [a (min(|u|, c) - c)^2 + 1], (a, c) the minimax
 *          fit (a* = -0.1240, c* = 2.4632), evaluated on integers of the
 *          input grid; the constants come from consts.swish_params.
 */
#include "ipo_linear.h"

#include <stddef.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define IPO_OK 0
#define IPO_ERR_NULL (-1)
#define IPO_ERR_SHAPE (-2)
#define IPO_ERR_PARAM (-3)

/* floor(x / 2^n), 0 <= n <= 62, independent of the sign behaviour of >>. */
static int64_t lin_floor_pow2(int64_t x, int n) {
    int64_t d = (int64_t)1 << n;
    if (x >= 0) return x / d;
    return -((-x + d - 1) / d);
}

/* Offset of channel c of frame (b, t) in an activation tensor. */
static size_t act_index(int layout, int b, int t, int c, int B, int T, int C, int G) {
    if (layout == IPO_ROWS) return ((size_t)b * T + t) * (size_t)C + (size_t)c;
    int per = C / G;              /* channels of one group */
    int g = c / per, cc = c % per;
    int heads = per / 128;
    return ((((size_t)g * B + b) * heads + (size_t)(cc / 128)) * T + t) * 128 + (size_t)(cc % 128);
}

int ipo_linear_i8(const int8_t *x, int x_layout, const int8_t *w, const int32_t *bias,
                  const int32_t *m, const int32_t *s, int B, int T, int K, int N, int G,
                  int8_t *y, int y_layout) {
    /* K <= 2^16 and |bias| < 2^30 keep |acc| < 2^31 and |m acc| < 2^62. */
    if (B < 0 || T < 1 || K < 1 || K > 65536 || N < 1 || G < 1) return IPO_ERR_SHAPE;
    if (x_layout != IPO_ROWS && x_layout != IPO_HEADS) return IPO_ERR_PARAM;
    if (y_layout != IPO_ROWS && y_layout != IPO_HEADS) return IPO_ERR_PARAM;
    if (x_layout == IPO_HEADS && K % 128 != 0) return IPO_ERR_SHAPE;
    if (y_layout == IPO_HEADS && N % (128 * G) != 0) return IPO_ERR_SHAPE;
    if (y_layout == IPO_ROWS && G != 1) return IPO_ERR_SHAPE;
    if (B == 0) return IPO_OK;
    if (!x || !w || !m || !s || !y) return IPO_ERR_NULL;
    for (int n = 0; n < N; ++n) {
        if (m[n] < 0 || s[n] < 0 || s[n] > 31) return IPO_ERR_PARAM;
        if (bias && (bias[n] >= (1 << 30) || bias[n] <= -(1 << 30))) return IPO_ERR_PARAM;
    }

    long long frames = (long long)B * T;
    int err = IPO_OK;
#pragma omp parallel
    {
        int64_t *xr = (int64_t *)malloc(sizeof(int64_t) * (size_t)K);
        if (!xr) {
#pragma omp atomic write
            err = IPO_ERR_PARAM;
        }
#pragma omp for schedule(static)
    for (long long f = 0; f < frames; ++f) {
        if (!xr) continue;
        int b = (int)(f / T), t = (int)(f % T);
        /* the input row of frame (b, t) */
        for (int k = 0; k < K; ++k) xr[k] = x[act_index(x_layout, b, t, k, B, T, K, 1)];
        for (int n = 0; n < N; ++n) {
            int64_t acc = bias ? (int64_t)bias[n] : 0;
            const int8_t *wn = w + (size_t)n * K;
            for (int k = 0; k < K; ++k) acc += xr[k] * (int64_t)wn[k];
            int e = 31 + s[n];
            int64_t v = lin_floor_pow2((int64_t)m[n] * acc + ((int64_t)1 << (e - 1)), e);
            if (v > 127) v = 127;
            if (v < -127) v = -127;
            y[act_index(y_layout, b, t, n, B, T, N, G)] = (int8_t)v;
        }
    }
        free(xr);
    }
    return err;
}

int ipo_swish_i8(const int8_t *z, long long n, const ipo_swish_params *p, int8_t *y) {
    if (n < 0) return IPO_ERR_SHAPE;
    if (n == 0) return IPO_OK;
    if (!z || !p || !y) return IPO_ERR_NULL;
    if (p->q_c < 1 || p->q_c >= (1 << 15) || p->q_one < 1 || p->q_one >= (1 << 23) ||
        (int64_t)p->q_one < (int64_t)p->q_c * p->q_c || p->m < 0 || p->s < 0 || p->s > 31)
        return IPO_ERR_PARAM;
    int e = 31 + p->s;
    for (long long i = 0; i < n; ++i) {
        int64_t q = z[i];
        int64_t a = q < 0 ? -q : q;                    /* |u| on the grid S_z / 2 */
        int64_t dclip = (a < p->q_c ? a : p->q_c) - p->q_c;
        int64_t L = (int64_t)p->q_one - dclip * dclip; /* |tanh|, grid S_t */
        int64_t sg = q > 0 ? 1 : (q < 0 ? -1 : 0);
        int64_t t = (int64_t)p->q_one + sg * L;        /* 1 + tanh */
        int64_t v = lin_floor_pow2((int64_t)p->m * (q * t) + ((int64_t)1 << (e - 1)), e);
        if (v > 127) v = 127;
        if (v < -127) v = -127;
        y[i] = (int8_t)v;
    }
    return IPO_OK;
}
