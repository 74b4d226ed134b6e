/*
 * CPU oracle of the integer linear layer of I-Parakeet (Sec. 2.2, Eqs. 6-7).
 *
 * TEST INFRASTRUCTURE ONLY: called by tests/, __graft_entry__.smoke() and
 * the CPU-baseline leg of bench.py; never by the GPU library, with which it
 * shares no code.
 */
#ifndef IPO_LINEAR_H
#define IPO_LINEAR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Tensor layouts of the activations (d = 128 channels per head):
 *   IPO_ROWS   [B][T][C]                 row-major, C channels per frame
 *   IPO_HEADS  [G][B][C/G/128][T][128]   head-split: channel c of group
 *              g = c / (C/G) sits in head (c mod C/G) / 128 at d = c mod 128
 * G (groups) is 1 except for a head-split output that stacks several
 * projections (Q, K, V as G = 3 tensors [B][H][T][128]). */
#define IPO_ROWS 0
#define IPO_HEADS 1

/* Eqs. 6-7 for every frame (b, t) and output channel n:
 *   acc     = sum_k x[b,t,k] w[n,k] + bias[n]                (exact)
 *   y[b,t,n] = clamp(round(2^-(31 + s[n]) m[n] acc), -127, 127)
 * round(v 2^-e) = floor((v + 2^(e-1)) / 2^e).  w: [N][K] row-major, one
 * row per output channel (per-channel weight scales give per-channel m, s);
 * bias: [N] or NULL (no bias); m: [N] in [0, 2^31); s: [N] in [0, 31].
 * Shapes: B >= 0, T >= 1, K >= 1, N >= 1; an IPO_HEADS input needs K a
 * multiple of 128, an IPO_HEADS output N a multiple of 128 G; an IPO_ROWS
 * output needs G = 1.  Returns IPO_OK or a negative IPO_ERR_*. */
int ipo_linear_i8(const int8_t *x, int x_layout, const int8_t *w, const int32_t *bias,
                  const int32_t *m, const int32_t *s, int B, int T, int K, int N, int G,
                  int8_t *y, int y_layout);

/* Integer constants of the minimax Swish (Sec. 3.2, Eqs. 12-13) for an
 * int8 input on grid S_z and an int8 output on grid S_y:
 *   q_c   = round(2 c* / S_z)                 clip point of |z| (|u| >= c*)
 *   q_one = round(1 / (|a*| (S_z / 2)^2))     the constant 1 on the grid
 *                                             S_t = |a*| (S_z / 2)^2
 *   m, s  : m 2^-(31+s) = S_z S_t / (2 S_y)   output requantisation */
typedef struct {
    int32_t q_c, q_one, m, s;
} ipo_swish_params;

/* Integer Swish of n int8 values (Eqs. 12-13, a* < 0):
 *   D = min(|z|, q_c) - q_c;  L = q_one - D^2      (|tanh| on the grid S_t)
 *   t = q_one + sgn(z) L                           (1 + tanh(z S_z / 2))
 *   y = clamp(round(2^-(31+s) m z t), -127, 127)   (z (1 + tanh) / 2)
 * Needs 1 <= q_c < 2^15, 1 <= q_one < 2^23, q_one >= q_c^2, m in [0, 2^31),
 * s in [0, 31]. */
int ipo_swish_i8(const int8_t *z, long long n, const ipo_swish_params *p, int8_t *y);

#ifdef __cplusplus
}
#endif
#endif /* IPO_LINEAR_H */
