/*
 * CPU oracle of the remaining integer parts of the I-Parakeet Conformer
 * block (Sec. 2.1 Eqs. 1-5, Sec. 2.2, Sec. 3.2, Sec. 3.3): residual
 * additions, the gated linear unit, the depthwise convolution with folded
 * BatchNorm on an INT16 output, and the Swish of that INT16 output.
 *
 * TEST INFRASTRUCTURE ONLY: called by tests/, __graft_entry__.smoke() and
 * the CPU legs of bench.py; it shares no code with the GPU library.
 */
#ifndef IPO_BLOCK_H
#define IPO_BLOCK_H

#include <stdint.h>

#include "ipo_linear.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Residual addition z = x + alpha y of two int8 tensors on grids S_x, S_y
 * onto S_z (Eqs. 1-4; alpha = 1/2 for the feed-forward branches), one
 * shared shift as in Eq. 11:
 *   z = clamp(round(2^-(31+s) (m_x x + m_y y)), -127, 127)
 * m_x, m_y in [0, 2^31), s in [0, 31]. */
int ipo_residual_i8(const int8_t *x, const int8_t *y, long long n, int32_t m_x, int32_t m_y,
                    int32_t s, int8_t *z);

/* Gated linear unit of Eq. 5, GLU(a, b) = a sigma(b) with sigma(b) = (1 +
 * tanh(b/2)) / 2 and the minimax tanh of Eq. 13, on int8 a (grid S_a) and
 * b (grid S_b), rows of 2C values [a_0..a_{C-1}, b_0..b_{C-1}]:
 *   D = min(|b|, q_c) - q_c;  t = q_one + sgn(b) (q_one - D^2)
 *   y = clamp(round(2^-(31+s) m a t), -127, 127)
 * with q_c, q_one from S_b and m 2^-(31+s) = S_a S_t / (2 S_y).  The Swish
 * is the case a = b (ipo_swish_i8).  y: [rows][C]. */
int ipo_glu_i8(const int8_t *ab, long long rows, int C, const ipo_swish_params *p, int8_t *y);

/* Depthwise convolution over time, kernel K (odd) centred with zero padding
 * at both ends of each utterance, BatchNorm folded into w and bias (Sec.
 * 2.2), requantised per channel onto the INT16 grid (Sec. 3.3):
 *   acc[b,t,c] = sum_k w[c][k] x[b][t + k - K/2][c] + bias[c]
 *   y[b,t,c]   = clamp(round(2^-(31+s[c]) m[c] acc), -32767, 32767)
 * x: int8 [B][T][C]; w: int8 [C][K]; bias int32 [C] (|bias| < 2^30);
 * y: int16 [B][T][C]. */
int ipo_dwconv_i16(const int8_t *x, int B, int T, int C, const int8_t *w, int K,
                   const int32_t *bias, const int32_t *m, const int32_t *s, int16_t *y);

/* Integer constants of the Swish for an INT16 input on grid S_z:
 * q_c = round(2 c* / S_z) in [1, 2^16), q_one = round(1 / S_t) in [1, 2^31)
 * with S_t = |a*| (S_z/2)^2 and q_one >= q_c^2, m 2^-(31+s) = S_z S_t /
 * (2 S_y). */
typedef struct {
    int32_t q_c;
    int64_t q_one;
    int32_t m, s;
} ipo_swish16_params;

/* Swish of n INT16 values onto int8 (the same steps as ipo_swish_i8; the
 * product m z t needs up to 78 bits and is formed exactly). */
int ipo_swish_i16(const int16_t *z, long long n, const ipo_swish16_params *p, int8_t *y);

#ifdef __cplusplus
}
#endif
#endif /* IPO_BLOCK_H */
