/*
 * CPU oracle of the integer LayerNorm used before every sub-module of the
 * I-Parakeet Conformer block (Sec. 2.1, Eqs. 1-4; Sec. 2.2 takes the
 * integer kernel from I-BERT).
 *
 * TEST INFRASTRUCTURE ONLY: called by tests/, __graft_entry__.smoke() and
 * the CPU legs of bench.py; it shares no code with the GPU library.
 */
#ifndef IPO_NORM_H
#define IPO_NORM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* floor(sqrt(n)) for 0 <= n < 2^62. */
int64_t ipo_isqrt(int64_t n);

/* Integer LayerNorm of `rows` rows of d int8 values q (grid S_x), for each
 * row (all integer, exact):
 *   c_i   = d q_i - sum_j q_j                     d (q_i - mean)
 *   sigma = isqrt(floor(sum_i c_i^2 / d) + eps_c)  d std(q), at least 1
 *   f     = floor(2^31 / sigma)
 *   n_i   = round(c_i f / 2^16)                   (q_i - mean) / std on 2^-15
 *   y_i   = clamp(round((M_i n_i + B_i) / 2^E_i), -127, 127)
 * round(v / 2^e) = floor((v + 2^(e-1)) / 2^e).  M (int32), B (int64), E
 * (int32 in [31, 62]) carry gamma, beta and the output grid per channel
 * (consts.layernorm_constants); eps_c >= 0 is epsilon on the grid of c^2.
 * d in [2, 4096] (|c| < 2^20, sum c^2 < 2^52); |B_i| < 2^60.  Returns 0 or a negative error. */
int ipo_layernorm_i8(const int8_t *x, long long rows, int d, int64_t eps_c, const int32_t *M,
                     const int64_t *B, const int32_t *E, int8_t *y);

#ifdef __cplusplus
}
#endif
#endif /* IPO_NORM_H */
