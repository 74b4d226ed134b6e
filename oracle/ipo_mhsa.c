/*
 * CPU oracle of the integer-only relative-positional MHSA (I-Parakeet,
 * Sec. 3.1).  TEST INFRASTRUCTURE ONLY: see ipo_mhsa.h.
 *
 * Plain scalar int64 code, written in the order the method states it:
 *   Eq. 8   content  qc[i][j] = sum_d (Q[i][d] + u[d]) K[j][d]
 *           position qp[i][j] = Phi((Q + 1v^T) P^T)[i][j]
 *                    with Phi the static index map r = j - i + T - 1
 *                    (P row r <-> relative distance T-1-r)
 *   Eq. 11  qs = round(2^-n (m_c qc + m_p qp)), n = 31 + s_s, onto the
 *           symmetric int8 grid [-127, 127] (Eq. 6)
 *   softmax I-BERT integer softmax over the valid keys (keys j >= len are
 *           excluded), output on the grid 2^-8
 *   Eq. 9   O = A V, requantised by Eq. 7 with n = 31 + s_o onto [-127, 127]
 * Rows i >= len output 0.  round(x 2^-n) is floor((x + 2^(n-1)) / 2^n).
 */
#include "ipo_mhsa.h"

#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static int g_threads = 0;

int ipo_set_threads(int n) {
#ifdef _OPENMP
    g_threads = n > 0 ? n : 0;
    return g_threads > 0 ? g_threads : omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}

/* floor(x / 2^n) for 0 <= n <= 62, without relying on the sign behaviour of
 * the C right shift. */
static int64_t floor_div_pow2(int64_t x, int n) {
    int64_t d = (int64_t)1 << n;
    if (x >= 0) return x / d;
    return -((-x + d - 1) / d);
}

/* round(x 2^-n), ties toward +infinity: floor((x + 2^(n-1)) / 2^n). */
static int64_t round_shift(int64_t x, int n) {
    return floor_div_pow2(x + ((int64_t)1 << (n - 1)), n);
}

static int64_t clamp_i8(int64_t x) {
    if (x > 127) return 127;
    if (x < -127) return -127;
    return x;
}

/* Domain of the softmax constants: q_ln2 >= 1, q_b >= 0, q_c >= 0, the
 * polynomial at p = 0 (the row maximum) at least 2, and the polynomial below
 * 2^31 on the whole interval (-q_ln2, 0] (a parabola: check both ends). */
static int check_params(const ipo_isoftmax_params *sm) {
    if (!sm) return IPO_ERR_NULL;
    if (sm->q_ln2 < 1 || sm->q_b < 0 || sm->q_c < 0) return IPO_ERR_PARAM;
    int64_t t0 = sm->q_b, t1 = (int64_t)sm->q_b - sm->q_ln2 + 1;
    int64_t l0 = t0 * t0 + sm->q_c, l1 = t1 * t1 + sm->q_c;
    if (l0 < 2) return IPO_ERR_PARAM;
    if (l0 >= ((int64_t)1 << 31) || l1 >= ((int64_t)1 << 31)) return IPO_ERR_PARAM;
    return IPO_OK;
}

/* --- Eq. 8, content branch, one score ---------------------------------- */
static int64_t content_score(const int8_t *qi, const int8_t *kj, const int8_t *u,
                             int dh) {
    int64_t acc = 0;
    for (int d = 0; d < dh; ++d)
        acc += ((int64_t)qi[d] + (int64_t)u[d]) * (int64_t)kj[d];
    return acc;
}

/* --- Eq. 8, position branch after Phi, one score ----------------------- */
static int64_t position_score(const int8_t *qi, const int8_t *ph, const int8_t *vb,
                              int i, int j, int T, int dh) {
    int r = j - i + T - 1; /* Phi: relative row of key j for query i */
    const int8_t *pr = ph + (size_t)r * dh;
    int64_t acc = 0;
    for (int d = 0; d < dh; ++d)
        acc += ((int64_t)qi[d] + (int64_t)vb[d]) * (int64_t)pr[d];
    return acc;
}

/* --- Eq. 11 ------------------------------------------------------------ */
static int64_t fused_score(int64_t qc, int64_t qp, int32_t m_c, int32_t m_p,
                           int32_t s_s) {
    int64_t x = (int64_t)m_c * qc + (int64_t)m_p * qp;
    return clamp_i8(round_shift(x, 31 + s_s));
}

/* --- I-BERT integer exponential ---------------------------------------
 * d <= 0 on grid S.  z = floor(-d / q_ln2), p = d + z q_ln2 in
 * (-q_ln2, 0], L = (p + q_b)^2 + q_c approximates exp(p S) / (a S^2), and
 * the result is L shifted right by z (0 once z reaches 63). */
int64_t ipo_iexp(int32_t d, const ipo_isoftmax_params *sm) {
    int64_t nd = -(int64_t)d;
    int64_t z = nd / sm->q_ln2;
    int64_t p = (int64_t)d + z * sm->q_ln2;
    int64_t t = p + sm->q_b;
    int64_t L = t * t + sm->q_c;
    if (z >= 63) return 0;
    return L >> z; /* L >= 0 */
}

/* --- I-BERT integer softmax over the first nvalid of n scores -----------
 * mx = max, e_j = iexp(s_j - mx), S = sum e_j, f = floor(2^32 / S),
 * a_j = min(255, floor(e_j f / 2^24)). */
static void isoftmax_row(const int8_t *s, int nvalid, int n,
                         const ipo_isoftmax_params *sm, int64_t *e, uint8_t *a) {
    for (int j = 0; j < n; ++j) a[j] = 0;
    if (nvalid <= 0) return;
    int32_t mx = s[0];
    for (int j = 1; j < nvalid; ++j)
        if (s[j] > mx) mx = s[j];
    int64_t sum = 0;
    for (int j = 0; j < nvalid; ++j) {
        e[j] = ipo_iexp((int32_t)s[j] - mx, sm);
        sum += e[j];
    }
    if (sum <= 0) return;
    int64_t f = ((int64_t)1 << 32) / sum;
    for (int j = 0; j < nvalid; ++j) {
        int64_t y = (e[j] * f) >> 24; /* e_j <= sum, so e_j f <= 2^32 */
        a[j] = (uint8_t)(y > 255 ? 255 : y);
    }
}

int ipo_isoftmax_u8(const int8_t *scores, const int32_t *valid, int rows, int n,
                    const ipo_isoftmax_params *sm, uint8_t *out) {
    if (!scores || !valid || !out) return IPO_ERR_NULL;
    if (rows < 0 || n < 1) return IPO_ERR_SHAPE;
    int rc = check_params(sm);
    if (rc) return rc;
    int64_t *e = (int64_t *)malloc(sizeof(int64_t) * (size_t)n);
    if (!e) return IPO_ERR_SHAPE;
    for (int r = 0; r < rows; ++r) {
        int nv = valid[r] < 0 ? 0 : (valid[r] > n ? n : valid[r]);
        isoftmax_row(scores + (size_t)r * n, nv, n, sm, e, out + (size_t)r * n);
    }
    free(e);
    return IPO_OK;
}

static int check_shape(int B, int H, int T, int dh) {
    if (B < 0 || H < 0 || T < 1 || dh < 1) return IPO_ERR_SHAPE;
    return IPO_OK;
}

int ipo_content_scores_i32(const int8_t *q, const int8_t *k, const int8_t *u,
                           int B, int H, int T, int dh, int32_t *out) {
    if (!q || !k || !u || !out) return IPO_ERR_NULL;
    int rc = check_shape(B, H, T, dh);
    if (rc) return rc;
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            size_t bh = (size_t)b * H + h;
            const int8_t *qh = q + bh * T * dh, *kh = k + bh * T * dh;
            for (int i = 0; i < T; ++i)
                for (int j = 0; j < T; ++j)
                    out[(bh * T + i) * T + j] = (int32_t)content_score(
                        qh + (size_t)i * dh, kh + (size_t)j * dh, u + (size_t)h * dh, dh);
        }
    return IPO_OK;
}

int ipo_position_scores_i32(const int8_t *q, const int8_t *p, const int8_t *vb,
                            int B, int H, int T, int dh, int32_t *out) {
    if (!q || !p || !vb || !out) return IPO_ERR_NULL;
    int rc = check_shape(B, H, T, dh);
    if (rc) return rc;
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            size_t bh = (size_t)b * H + h;
            const int8_t *qh = q + bh * T * dh;
            const int8_t *ph = p + (size_t)h * (2 * (size_t)T - 1) * dh;
            for (int i = 0; i < T; ++i)
                for (int j = 0; j < T; ++j)
                    out[(bh * T + i) * T + j] = (int32_t)position_score(
                        qh + (size_t)i * dh, ph, vb + (size_t)h * dh, i, j, T, dh);
        }
    return IPO_OK;
}

int ipo_fused_scores_i8(const int8_t *q, const int8_t *k, const int8_t *p,
                        const int8_t *u, const int8_t *vb, int32_t m_c,
                        int32_t m_p, int32_t s_s, int B, int H, int T, int dh,
                        int8_t *out) {
    if (!q || !k || !p || !u || !vb || !out) return IPO_ERR_NULL;
    int rc = check_shape(B, H, T, dh);
    if (rc) return rc;
    if (m_c < 0 || m_p < 0 || s_s < 0 || s_s > 31) return IPO_ERR_PARAM;
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            size_t bh = (size_t)b * H + h;
            const int8_t *qh = q + bh * T * dh, *kh = k + bh * T * dh;
            const int8_t *ph = p + (size_t)h * (2 * (size_t)T - 1) * dh;
            for (int i = 0; i < T; ++i)
                for (int j = 0; j < T; ++j) {
                    const int8_t *qi = qh + (size_t)i * dh;
                    int64_t qc = content_score(qi, kh + (size_t)j * dh, u + (size_t)h * dh, dh);
                    int64_t qp = position_score(qi, ph, vb + (size_t)h * dh, i, j, T, dh);
                    out[(bh * T + i) * T + j] = (int8_t)fused_score(qc, qp, m_c, m_p, s_s);
                }
        }
    return IPO_OK;
}

/* One (b, h) head of the whole layer. */
static void head(const int8_t *qh, const int8_t *kh, const int8_t *vh,
                 const int8_t *ph, const int8_t *u, const int8_t *vb,
                 const int32_t *mult, const int32_t *shifts,
                 const ipo_isoftmax_params *sm, int len, int T, int dh,
                 int8_t *oh, int8_t *srow, int64_t *e, uint8_t *a) {
    for (int i = 0; i < T; ++i) {
        int8_t *oi = oh + (size_t)i * dh;
        if (i >= len) { /* padded query row */
            memset(oi, 0, (size_t)dh);
            continue;
        }
        const int8_t *qi = qh + (size_t)i * dh;
        for (int j = 0; j < len; ++j) {
            int64_t qc = content_score(qi, kh + (size_t)j * dh, u, dh);
            int64_t qp = position_score(qi, ph, vb, i, j, T, dh);
            srow[j] = (int8_t)fused_score(qc, qp, mult[0], mult[1], shifts[0]);
        }
        isoftmax_row(srow, len, len, sm, e, a);
        for (int d = 0; d < dh; ++d) {
            int64_t acc = 0;
            for (int j = 0; j < len; ++j)
                acc += (int64_t)a[j] * (int64_t)vh[(size_t)j * dh + d];
            oi[d] = (int8_t)clamp_i8(round_shift((int64_t)mult[2] * acc, 31 + shifts[1]));
        }
    }
}

int ipo_relpos_mhsa_i8(const int8_t *q, const int8_t *k, const int8_t *v,
                       const int8_t *p, const int8_t *u, const int8_t *vb,
                       const int32_t *multipliers, const int32_t *shifts,
                       const ipo_isoftmax_params *sm, const int32_t *lengths,
                       int B, int H, int T, int dh, int8_t *out) {
    if (!q || !k || !v || !p || !u || !vb || !multipliers || !shifts || !out)
        return IPO_ERR_NULL;
    int rc = check_shape(B, H, T, dh);
    if (rc) return rc;
    rc = check_params(sm);
    if (rc) return rc;
    for (int c = 0; c < 3; ++c)
        if (multipliers[c] < 0) return IPO_ERR_PARAM;
    for (int c = 0; c < 2; ++c)
        if (shifts[c] < 0 || shifts[c] > 31) return IPO_ERR_PARAM;
    long nbh = (long)B * H;
    int err = 0;
#ifdef _OPENMP
    int nt = g_threads > 0 ? g_threads : omp_get_max_threads();
#pragma omp parallel num_threads(nt) reduction(| : err)
#endif
    {
        int8_t *srow = (int8_t *)malloc((size_t)T);
        int64_t *e = (int64_t *)malloc(sizeof(int64_t) * (size_t)T);
        uint8_t *a = (uint8_t *)malloc((size_t)T);
        if (!srow || !e || !a) err = 1;
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
        for (long bh = 0; bh < nbh; ++bh) {
            if (!srow || !e || !a) continue;
            int b = (int)(bh / H), h = (int)(bh % H);
            int len = lengths ? lengths[b] : T;
            if (len < 0) len = 0;
            if (len > T) len = T;
            size_t off = (size_t)bh * T * dh;
            head(q + off, k + off, v + off, p + (size_t)h * (2 * (size_t)T - 1) * dh,
                 u + (size_t)h * dh, vb + (size_t)h * dh, multipliers, shifts, sm,
                 len, T, dh, out + off, srow, e, a);
        }
        free(srow);
        free(e);
        free(a);
    }
    return err ? IPO_ERR_SHAPE : IPO_OK;
}
