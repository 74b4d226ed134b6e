/*
 * CPU oracle of the integer-only relative-positional multi-head
 * self-attention (I-Parakeet, Sec. 3.1, Eqs. 8-11; softmax per I-BERT).
 *
 * TEST INFRASTRUCTURE ONLY.  This library is the slow, obviously correct
 * int64 statement of what the GPU path must compute.  Only the tests, the
 * smoke check and the CPU-baseline leg of the benchmark load it; the GPU
 * library shares no code, header, table or constant with it.
 *
 * All pointers are host pointers to C-contiguous arrays.  Functions return 0
 * on success and a negative code when an argument is unusable.
 */
#ifndef IPO_MHSA_H
#define IPO_MHSA_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Integer constants of I-BERT's exponential for one score grid S_s:
 * q_ln2 = floor(ln2 / S_s), q_b = floor(b / S_s), q_c = floor(c / (a S_s^2)). */
typedef struct {
    int32_t q_ln2;
    int32_t q_b;
    int32_t q_c;
} ipo_isoftmax_params;

#define IPO_OK 0
#define IPO_ERR_NULL (-1)
#define IPO_ERR_SHAPE (-2)
#define IPO_ERR_PARAM (-3)

/* Whole layer.  q,k,v,out: [B,H,T,dh]; p: [H,2T-1,dh]; u,vb: [H,dh];
 * multipliers = {m_c, m_p, m_o}; shifts = {s_s, s_o} (right shift 31+s);
 * lengths: [B] valid lengths (clamped to [0,T]) or NULL for all T. */
int ipo_relpos_mhsa_i8(const int8_t *q, const int8_t *k, const int8_t *v,
                       const int8_t *p, const int8_t *u, const int8_t *vb,
                       const int32_t *multipliers, const int32_t *shifts,
                       const ipo_isoftmax_params *sm, const int32_t *lengths,
                       int B, int H, int T, int dh, int8_t *out);

/* Content branch of Eq. 8, A^c = (Q + 1u^T) K^T, as int32 [B,H,T,T]. */
int ipo_content_scores_i32(const int8_t *q, const int8_t *k, const int8_t *u,
                           int B, int H, int T, int dh, int32_t *out);

/* Position branch of Eq. 8 after the relative shift,
 * Phi((Q + 1v^T) P^T)[i][j], as int32 [B,H,T,T]. */
int ipo_position_scores_i32(const int8_t *q, const int8_t *p, const int8_t *vb,
                            int B, int H, int T, int dh, int32_t *out);

/* Fused integer scores of Eq. 11, clamped to the int8 grid, [B,H,T,T]
 * (no key mask applied). */
int ipo_fused_scores_i8(const int8_t *q, const int8_t *k, const int8_t *p,
                        const int8_t *u, const int8_t *vb, int32_t m_c,
                        int32_t m_p, int32_t s_s, int B, int H, int T, int dh,
                        int8_t *out);

/* I-BERT integer exponential of one non-positive integer d on grid S_s. */
int64_t ipo_iexp(int32_t d, const ipo_isoftmax_params *sm);

/* Integer softmax of `rows` rows of n int8 scores.  Row r uses its first
 * valid[r] entries (clamped to [0,n]); the rest of the row, and whole rows
 * with no valid entry, get probability 0.  Output u8 on the grid 2^-8. */
int ipo_isoftmax_u8(const int8_t *scores, const int32_t *valid, int rows,
                    int n, const ipo_isoftmax_params *sm, uint8_t *out);

/* Number of OpenMP threads used by ipo_relpos_mhsa_i8 (<= 0: library
 * default).  Returns the count in effect. */
int ipo_set_threads(int n);

#ifdef __cplusplus
}
#endif
#endif
