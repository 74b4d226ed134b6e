/*
 * CPU oracle of the remaining integer parts of the Conformer block (Sec.
 * 2.1 Eqs. 1-5, Sec. 2.2, Sec. 3.2, Sec. 3.3).  TEST INFRASTRUCTURE ONLY:
 * see ipo_block.h.  Plain scalar int64 code (int128 where a product needs
 * more than 63 bits).
 */
#include "ipo_block.h"

#include <stddef.h>

#define IPO_OK 0
#define IPO_ERR_NULL (-1)
#define IPO_ERR_SHAPE (-2)
#define IPO_ERR_PARAM (-3)

/* floor(x / 2^n), 0 <= n <= 62, independent of the sign behaviour of >>. */
static int64_t blk_floor_pow2(int64_t x, int n) {
    int64_t d = (int64_t)1 << n;
    if (x >= 0) return x / d;
    return -((-x + d - 1) / d);
}

static int64_t blk_clamp(int64_t v, int64_t lim) {
    return v > lim ? lim : (v < -lim ? -lim : v);
}

int ipo_residual_i8(const int8_t *x, const int8_t *y, long long n, int32_t m_x, int32_t m_y,
                    int32_t s, int8_t *z) {
    if (n < 0) return IPO_ERR_SHAPE;
    if (n == 0) return IPO_OK;
    if (!x || !y || !z) return IPO_ERR_NULL;
    if (m_x < 0 || m_y < 0 || s < 0 || s > 31) return IPO_ERR_PARAM;
    int e = 31 + s;
    for (long long i = 0; i < n; ++i) {
        int64_t v = (int64_t)m_x * x[i] + (int64_t)m_y * y[i];
        z[i] = (int8_t)blk_clamp(blk_floor_pow2(v + ((int64_t)1 << (e - 1)), e), 127);
    }
    return IPO_OK;
}

int ipo_glu_i8(const int8_t *ab, long long rows, int C, const ipo_swish_params *p, int8_t *y) {
    if (rows < 0 || C < 1) return IPO_ERR_SHAPE;
    if (rows == 0) return IPO_OK;
    if (!ab || !p || !y) return IPO_ERR_NULL;
    if (p->q_c < 1 || p->q_c >= (1 << 15) || p->q_one < 1 || p->q_one >= (1 << 23) ||
        (int64_t)p->q_one < (int64_t)p->q_c * p->q_c || p->m < 0 || p->s < 0 || p->s > 31)
        return IPO_ERR_PARAM;
    int e = 31 + p->s;
    for (long long r = 0; r < rows; ++r) {
        for (int c = 0; c < C; ++c) {
            int64_t a = ab[(size_t)r * 2 * C + c];
            int64_t b = ab[(size_t)r * 2 * C + C + c];
            int64_t mag = b < 0 ? -b : b;
            int64_t dclip = (mag < p->q_c ? mag : p->q_c) - p->q_c;
            int64_t L = (int64_t)p->q_one - dclip * dclip;           /* |tanh(b/2)| */
            int64_t sg = b > 0 ? 1 : (b < 0 ? -1 : 0);
            int64_t t = (int64_t)p->q_one + sg * L;                   /* 1 + tanh */
            int64_t v = (int64_t)p->m * (a * t) + ((int64_t)1 << (e - 1));
            y[(size_t)r * C + c] = (int8_t)blk_clamp(blk_floor_pow2(v, e), 127);
        }
    }
    return IPO_OK;
}

int ipo_dwconv_i16(const int8_t *x, int B, int T, int C, const int8_t *w, int K,
                   const int32_t *bias, const int32_t *m, const int32_t *s, int16_t *y) {
    if (B < 0 || T < 1 || C < 1 || K < 1 || K % 2 == 0 || K > 63) return IPO_ERR_SHAPE;
    if (B == 0) return IPO_OK;
    if (!x || !w || !bias || !m || !s || !y) return IPO_ERR_NULL;
    for (int c = 0; c < C; ++c)
        if (m[c] < 0 || s[c] < 0 || s[c] > 31 || bias[c] >= (1 << 30) || bias[c] <= -(1 << 30))
            return IPO_ERR_PARAM;
    int half = K / 2;
    for (int b = 0; b < B; ++b)
        for (int t = 0; t < T; ++t)
            for (int c = 0; c < C; ++c) {
                int64_t acc = bias[c];
                for (int k = 0; k < K; ++k) {
                    int tt = t + k - half;
                    if (tt < 0 || tt >= T) continue;               /* zero padding */
                    acc += (int64_t)w[(size_t)c * K + k] * x[((size_t)b * T + tt) * C + c];
                }
                int e = 31 + s[c];
                int64_t v = blk_floor_pow2((int64_t)m[c] * acc + ((int64_t)1 << (e - 1)), e);
                y[((size_t)b * T + t) * C + c] = (int16_t)blk_clamp(v, 32767);
            }
    return IPO_OK;
}

int ipo_swish_i16(const int16_t *z, long long n, const ipo_swish16_params *p, int8_t *y) {
    if (n < 0) return IPO_ERR_SHAPE;
    if (n == 0) return IPO_OK;
    if (!z || !p || !y) return IPO_ERR_NULL;
    if (p->q_c < 1 || p->q_c >= (1 << 16) || p->q_one < 1 || p->q_one >= ((int64_t)1 << 31) ||
        p->q_one < (int64_t)p->q_c * p->q_c || p->m < 0 || p->s < 0 || p->s > 31)
        return IPO_ERR_PARAM;
    int e = 31 + p->s;
    for (long long i = 0; i < n; ++i) {
        int64_t q = z[i];
        int64_t mag = q < 0 ? -q : q;
        int64_t dclip = (mag < p->q_c ? mag : p->q_c) - p->q_c;
        int64_t L = p->q_one - dclip * dclip;
        int64_t sg = q > 0 ? 1 : (q < 0 ? -1 : 0);
        int64_t t = p->q_one + sg * L;
        __int128 v = (__int128)p->m * (__int128)(q * t) + ((__int128)1 << (e - 1));
        /* floor(v / 2^e) without relying on the sign behaviour of >> */
        __int128 d = (__int128)1 << e;
        __int128 r = v >= 0 ? v / d : -((-v + d - 1) / d);
        y[i] = (int8_t)blk_clamp((int64_t)(r > 1000 ? 1000 : (r < -1000 ? -1000 : r)), 127);
    }
    return IPO_OK;
}
