/*
 * ip_mhsa.h - C ABI of the integer-only relative-positional multi-head
 * self-attention of I-Parakeet (Sec. 3.1) on one GB300 GPU (sm_103a).
 *
 * Per (batch b, head h), with T frames, head width dh = 128 and R = 2T-1
 * relative positions, the library computes
 *
 *   content   qc[i][j] = sum_d (Q[i][d] + u[d]) K[j][d]                (Eq. 8)
 *   position  qp[i][j] = sum_d (Q[i][d] + v[d]) P[j - i + T - 1][d]    (Eq. 8,
 *             the relative shift Phi applied as an index map; P row r holds
 *             relative distance T-1-r)
 *   fused     qs = clamp(round(2^-(31+s_s) (m_c qc + m_p qp)), -127, 127)
 *                                                             (Eqs. 10-11, 6)
 *   softmax   I-BERT integer softmax over the valid keys j < len_b:
 *             mx = max_j qs, e_j = iexp(qs_j - mx), f = floor(2^32 / sum e),
 *             a_j = min(255, floor(e_j f / 2^24))  (probabilities on 2^-8)
 *             iexp(d): z = floor(-d / q_ln2), p = d + z q_ln2,
 *                      floor(((p + q_b)^2 + q_c) / 2^z)
 *   output    O[i][d] = clamp(round(2^-(31+s_o) m_o sum_j a_j V[j][d]),
 *                             -127, 127)                      (Eq. 9, Eq. 7)
 *
 * and writes O; query rows i >= len_b are written as 0.  round(x 2^-n) is
 * floor((x + 2^(n-1)) / 2^n) (ties toward +infinity).  Every step runs in
 * integer arithmetic on the GPU; the offline helpers at the end turn real
 * scales into the integer constants on the host, as the paper precomputes
 * its multipliers offline (Sec. 2.2, under Eq. 7).
 *
 * Layouts: all arrays C-contiguous, int8 unless stated.
 *   q, k, v, out : [B][H][T][dh]      p : [H][2T-1][dh]      u, v_bias : [H][dh]
 * Ownership: every buffer belongs to the caller; the library allocates no
 * memory.  Device entry points are asynchronous on `stream`; inputs are not
 * modified.  The attention calls keep the TMA descriptors of the last 32
 * (pointer, shape) pairs they saw; a descriptor holds nothing but the
 * address and the shape, so one stays valid for any buffer at that address.  Return value: IP_OK (0) or a negative IP_ERR_* code
 * (ip_strerror gives its text); the library never aborts the process.
 */
#ifndef IP_MHSA_H
#define IP_MHSA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st *ip_stream_t; /* a cudaStream_t; NULL = legacy default stream */

/* Integer constants of I-BERT's exponential on the fused-score grid S_s:
 * q_ln2 = floor(ln2 / S_s), q_b = floor(1.353 / S_s),
 * q_c = floor(0.344 / (0.3585 S_s^2)).  Domain: q_ln2 >= 1, q_b >= 0,
 * q_c >= 0, q_b^2 + q_c >= 2, and (p + q_b)^2 + q_c < 2^31 for all p in
 * (-q_ln2, 0]. */
typedef struct {
    int32_t q_ln2;
    int32_t q_b;
    int32_t q_c;
} ip_isoftmax_params;

#define IP_OK 0
#define IP_ERR_NULL (-1)        /* a required pointer is NULL */
#define IP_ERR_SHAPE (-2)       /* B, H, T out of range (see IP_MAX_*) */
#define IP_ERR_ALIGN (-3)       /* a pointer is not 16-byte aligned (workspace: 256) */
#define IP_ERR_UNSUPPORTED (-4) /* dh != 128 */
#define IP_ERR_CUDA (-5)        /* a CUDA runtime call failed */
#define IP_ERR_TIMEOUT (-6)     /* a kernel gave up waiting on a barrier */
#define IP_ERR_PARAM (-7)       /* a multiplier, shift or softmax constant is out of its domain */
#define IP_ERR_WORKSPACE (-8)   /* workspace smaller than ip_relpos_mhsa_workspace_bytes */

#define IP_DH 128
#define IP_MAX_T 2048   /* frames; the int8 scores of a 64-row tile stay on chip or in L2 */
#define IP_MAX_B 65535
#define IP_MAX_H 65535
/* B H ceil(T / 64) (the 64-row query tiles of a call) must stay below this:
 * the kernel's work items (up to four per tile) are numbered with 31 bits. */
#define IP_MAX_TILES (1ll << 29)

/* Bytes of device workspace a call needs: the device-side status word of
 * the calls that use it.  The caller zero-fills the workspace once before
 * its first use; ip_relpos_mhsa_status reads and clears it.  The workspace
 * also holds the work-item counters of the attention kernel (its CTAs claim
 * query tiles from them), which every call returns to zero when it ends;
 * calls that share a workspace must not overlap on the GPU.
 * For T > 384 the size also counts a region for the int8 scores of every
 * resident CTA of the current device (4 warps x 16 rows x T, rounded up to
 * 64 keys, per CTA): a call given that much keeps the scores between the
 * softmax passes there (in L2) and fits two CTAs per SM; a call given only
 * the first 256 bytes keeps them in shared memory, one CTA per SM, with the
 * same result.  The region needs no zero fill.  0 if the shape is invalid. */
size_t ip_relpos_mhsa_workspace_bytes(int B, int H, int T, int dh);

/* The whole layer on the GPU.
 *   q, k, v, p, u, v_bias, out : device pointers, 16-byte aligned.
 *   multipliers : HOST array {m_c, m_p, m_o}, each in [0, 2^31).
 *   shifts      : HOST array {s_s, s_o}, each in [0, 31]; the right shift
 *                 of Eq. 11 is 31 + s_s, that of the output 31 + s_o.
 *   sm          : HOST pointer to the softmax constants.
 *   lengths     : DEVICE array [B] of valid lengths (values clamped to
 *                 [0, T]), or NULL for all T.
 *   workspace   : device memory of workspace_bytes >= the size above,
 *                 256-byte aligned, owned by the caller; one call at a time
 *                 per workspace.  NULL: the workspace registered with
 *                 ip_set_workspace (IP_ERR_NULL if there is none, or
 *                 IP_ERR_WORKSPACE if it is smaller than the call needs).
 * The call validates its arguments on the host and then enqueues one
 * kernel on `stream` (a persistent grid of one CTA per resident slot that
 * walks the 64-row query tiles of all (b, h)).  B == 0 or H == 0 is an empty problem: the call
 * returns IP_OK without touching any pointer.  A kernel-side barrier timeout is reported later by
 * ip_relpos_mhsa_status. */
int ip_relpos_mhsa_i8(const int8_t *q, const int8_t *k, const int8_t *v,
                      const int8_t *p, const int8_t *u, const int8_t *v_bias,
                      const int32_t *multipliers, const int32_t *shifts,
                      const ip_isoftmax_params *sm, const int32_t *lengths,
                      int B, int H, int T, int dh, int8_t *out,
                      void *workspace, size_t workspace_bytes, ip_stream_t stream);

/* Synchronises `stream`, reports the device-side status of the calls that
 * used `workspace` since the previous status call (IP_OK, IP_ERR_TIMEOUT,
 * or IP_ERR_CUDA) and clears it.  workspace = NULL: the one registered with
 * ip_set_workspace (IP_ERR_NULL if there is none). */
int ip_relpos_mhsa_status(const void *workspace, ip_stream_t stream);

/* Registers a default workspace for the attention calls of this process
 * that pass a NULL workspace: device memory of `bytes` (at least
 * ip_relpos_mhsa_workspace_bytes), 256-byte aligned, zero-filled once by the
 * caller and owned by it until it is replaced or released.  ptr = NULL
 * releases the registration.  Since calls that share a workspace must not
 * overlap on the GPU, the default suits callers that issue their attention
 * calls on one stream.  IP_ERR_ALIGN for a misaligned ptr,
 * IP_ERR_WORKSPACE if bytes is too small. */
int ip_set_workspace(void *ptr, size_t bytes);

/* Bytes of device staging memory ip_relpos_mhsa_i8_host needs (inputs,
 * output, lengths and workspace), 0 if the shape is invalid. */
size_t ip_relpos_mhsa_host_arena_bytes(int B, int H, int T, int dh);

/* The whole layer from HOST buffers: copies the inputs (and lengths, a HOST
 * array or NULL) into `arena` (device memory of arena_bytes >= the size
 * above, 256-byte aligned, owned by the caller), runs ip_relpos_mhsa_i8,
 * copies the result into the HOST buffer `out` and synchronises `stream`.
 * Page-locked host buffers make the copies asynchronous DMA. */
int ip_relpos_mhsa_i8_host(const int8_t *q, const int8_t *k, const int8_t *v,
                           const int8_t *p, const int8_t *u, const int8_t *v_bias,
                           const int32_t *multipliers, const int32_t *shifts,
                           const ip_isoftmax_params *sm, const int32_t *lengths,
                           int B, int H, int T, int dh, int8_t *out,
                           void *arena, size_t arena_bytes, ip_stream_t stream);

/* The whole layer without any allocation by anyone: the same computation
 * and result as ip_relpos_mhsa_i8, for callers that cannot allocate device
 * memory, such as a plugin whose host framework owns the whole device pool
 * and hands it only input and output buffers, or a latency-critical
 * streaming path where a device allocation (which may synchronise the
 * device) is not allowed.  The paper has no counterpart of this entry point.
 *
 * The caller passes inputs and outputs as for ip_relpos_mhsa_i8 (device
 * pointers, 16-byte aligned; lengths a device array or NULL).  The scratch
 * the kernel needs - the device status word that ip_relpos_mhsa_i8 keeps in
 * the caller's workspace - lives instead in a file-scope device array of
 * IP_NOALLOC_SCRATCH_BYTES bytes inside the library, held by every GPU that
 * loads the library until the process exits.  A call whose scratch need
 * exceeds that size is rejected with IP_ERR_WORKSPACE (every shape the
 * library accepts needs IP_NOALLOC_SCRATCH_BYTES at most).  The call makes
 * no allocation: no cudaMalloc, cudaFree or allocating library routine.
 *
 * The first call on a device looks up the device address of the array
 * (cudaGetSymbolAddress, with that device current) and caches it for the
 * life of the process; make that first call before any stream capture.  A
 * device reset (cudaDeviceReset) after that first call is not supported:
 * the cached address would belong to the destroyed context.  Every call shares the array and
 * clears its status word in stream order before launching; calls that
 * overlap on the GPU (concurrent streams) race on it.  Kernel-side barrier
 * timeouts are recorded there; ip_relpos_mhsa_noalloc_status reads them.
 * Returns IP_OK or an IP_ERR_* code as ip_relpos_mhsa_i8. */
#define IP_NOALLOC_SCRATCH_BYTES 256
int ip_relpos_mhsa_i8_noalloc(const int8_t *q, const int8_t *k, const int8_t *v,
                              const int8_t *p, const int8_t *u, const int8_t *v_bias,
                              const int32_t *multipliers, const int32_t *shifts,
                              const ip_isoftmax_params *sm, const int32_t *lengths,
                              int B, int H, int T, int dh, int8_t *out, ip_stream_t stream);

/* Device-side status of the ip_relpos_mhsa_i8_noalloc calls made on the
 * current device since the last call of this function or of the entry
 * point itself (each call clears the word before its kernel): synchronises
 * `stream`, returns IP_OK, IP_ERR_TIMEOUT (a bounded barrier wait ran out)
 * or IP_ERR_PARAM (a device-side constant out of its domain), and clears
 * the word.  Read it after the call whose result is in question, on the
 * call's stream, before the next call.  Allocates nothing; IP_OK if the
 * entry point was never called on this device. */
int ip_relpos_mhsa_noalloc_status(ip_stream_t stream);

/* ---- integer linear layer (Sec. 2.2, Eqs. 6-7) ------------------------
 *
 * The projections around the attention: Q, K, V (and P) from the
 * normalised frames, and the output projection of the heads.  Weights carry
 * one scale per output channel, so Eq. 7's multiplier is per channel.
 *
 * Activation layouts (int8, C channels per frame, d = 128 per head):
 *   IP_LAYOUT_ROWS   [B][T][C] row-major
 *   IP_LAYOUT_HEADS  [G][B][C/G/128][T][128]: channel c of group g = c / (C/G)
 *                    sits in head (c mod C/G) / 128 at d = c mod 128.  G = 1 is
 *                    the attention's [B][H][T][128]; G = 3 writes Q, K and V
 *                    of one stacked projection as three such tensors. */
#define IP_LAYOUT_ROWS 0
#define IP_LAYOUT_HEADS 1
#define IP_LINEAR_MAX_K 32768          /* keeps the int32 accumulator exact */
#define IP_LINEAR_MAX_N 65536
#define IP_LINEAR_MAX_FRAMES 134217728  /* B T, 2^27 */

/* For every frame (b, t) and output channel n (Eq. 7):
 *   acc       = sum_k x[b,t,k] w[n,k] + bias[n]                   (int32)
 *   y[b,t,n]  = clamp(round(2^-(31 + s[n]) m[n] acc), -127, 127)
 * round(v 2^-e) = floor((v + 2^(e-1)) / 2^e).
 * x: device int8, x_layout with C = K (IP_LAYOUT_HEADS reads K/128 heads).
 * w: device int8 [N][K] row-major (one row per output channel).
 * bias: device int32 [N] with |bias| < 2^30, or NULL; m: device int32 [N]
 *   in [0, 2^31); s: device int32 [N] in [0, 31] (a value outside is
 *   clamped into its domain and reported as IP_ERR_PARAM by
 *   ip_relpos_mhsa_status).
 * y: device int8, y_layout with C = N and G groups (G = 1 for ROWS).
 * Shapes: B in [0, IP_MAX_B], T >= 1, B T <= IP_LINEAR_MAX_FRAMES, K a
 *   multiple of 128 in [128, IP_LINEAR_MAX_K], N a multiple of 128 (of 128 G
 *   for a HEADS output) up to IP_LINEAR_MAX_N.
 * x, w, y 16-byte aligned; bias, m, s 4-byte aligned; workspace as for
 *   ip_relpos_mhsa_i8 (>= 256 bytes, 256-aligned, zero-filled once; its
 *   status word is read and cleared by ip_relpos_mhsa_status).
 * Inputs are not modified; launch is asynchronous on `stream`; B == 0
 * returns IP_OK without touching any pointer.  Returns IP_OK or IP_ERR_*. */
int ip_linear_i8(const int8_t *x, int x_layout, const int8_t *w, const int32_t *bias,
                 const int32_t *m, const int32_t *s, int B, int T, int K, int N, int G,
                 int8_t *y, int y_layout, void *workspace, size_t workspace_bytes,
                 ip_stream_t stream);

/* ---- minimax integer Swish (Sec. 3.2, Eqs. 12-13) ----------------------
 *
 * Swish sw(x) = x (1 + tanh(x/2)) / 2 with tanh(u) ~ sgn(u) [a (min(|u|, c)
 * - c)^2 + 1] and the paper's minimax fit (a, c) below, on int8 inputs z of
 * grid S_z and int8 outputs of grid S_y:
 *   D = min(|z|, q_c) - q_c;  L = q_one - D^2;  t = q_one + sgn(z) L
 *   y = clamp(round(2^-(31+s) m z t), -127, 127)
 * q_c = round(2c / S_z) is the clip point of |z|, q_one = round(1 / S_t)
 * the 1 of the polynomial on its grid S_t = |a| (S_z/2)^2, and m 2^-(31+s)
 * is S_z S_t / (2 S_y).  Domain: 1 <= q_c < 2^15, 1 <= q_one < 2^23,
 * q_one >= q_c^2, m in [0, 2^31), s in [0, 31]. */
#define IP_SWISH_A (-0.1240)
#define IP_SWISH_C 2.4632

typedef struct {
    int32_t q_c, q_one, m, s;
} ip_swish_params;

/* The feed-forward layer's first projection with the Swish fused into its
 * epilogue: z = ip_linear_i8's output (row-major, G = 1; m, s put z on the
 * grid S_z), then y = Swish(z) on S_y.  Arguments as ip_linear_i8 (x and y
 * IP_LAYOUT_ROWS); sw: host, validated (IP_ERR_PARAM outside its domain). */
int ip_linear_swish_i8(const int8_t *x, const int8_t *w, const int32_t *bias, const int32_t *m,
                       const int32_t *s, const ip_swish_params *sw, int B, int T, int K, int N,
                       int8_t *y, void *workspace, size_t workspace_bytes, ip_stream_t stream);

/* Swish constants for the grids S_z (input) and S_y (output), host only. */
int ip_swish_params_from_scales(double S_z, double S_y, ip_swish_params *out);

/* ---- integer LayerNorm (Sec. 2.1, Eqs. 1-4; integer kernel of Sec. 2.2) --
 *
 * For each row of d int8 values q (grid S_x), all in integers:
 *   c_i   = d q_i - sum_j q_j                          d (q_i - mean)
 *   sigma = max(1, isqrt(floor(sum_i c_i^2 / d) + eps_c))
 *   f     = floor(2^31 / sigma)
 *   n_i   = round(c_i f / 2^16)                        (q_i - mean) / std on 2^-15
 *   y_i   = clamp(round((M_i n_i + B_i) / 2^E_i), -127, 127)
 * round(v / 2^e) = floor((v + 2^(e-1)) / 2^e).  M, B, E per channel carry
 * gamma, beta and the output grid S_y (ip_layernorm_constants); eps_c is the
 * epsilon of the variance on the grid of c^2 / d. */
#define IP_NORM_MAX_ROWS (1ll << 40)

/* x, y: device int8 [rows][d] row-major (16-byte aligned); d in {512, 1024,
 * 1536, 2048} (others: IP_ERR_UNSUPPORTED); M: device int32 [d]; B: device
 * int64 [d] with |B| < 2^60; E: device int32 [d] in [31, 62] (a value out of
 * its domain is clamped and reported as IP_ERR_PARAM by
 * ip_relpos_mhsa_status); eps_c in [0, 2^40]; workspace as for
 * ip_relpos_mhsa_i8.  rows == 0 returns IP_OK without touching any pointer.
 * Launch asynchronous on `stream`.  Returns IP_OK or IP_ERR_*. */
int ip_layernorm_i8(const int8_t *x, long long rows, int d, long long eps_c, const int32_t *M,
                    const long long *B, const int32_t *E, int8_t *y, void *workspace,
                    size_t workspace_bytes, ip_stream_t stream);

/* Offline constants of the LayerNorm (host, float64): gamma, beta [d] real,
 * input grid S_x, output grid S_y, epsilon eps.  Per channel, (|M_i|, E_i -
 * 31) is the dyadic of |gamma_i| 2^-15 / S_y with the sign of gamma_i on M_i
 * (gamma_i = 0: M_i = 0, E_i = 31), B_i = round(beta_i / S_y 2^E_i), and
 * eps_c = round(eps d^2 / S_x^2).  Outputs: eps_c, M, B, E [d]. */
int ip_layernorm_constants(double S_x, const double *gamma, const double *beta, int d,
                           double S_y, double eps, long long *eps_c, int32_t *M, long long *B,
                           int32_t *E);

/* ---- rest of the Conformer block (Sec. 2.1 Eqs. 1-5, Sec. 3.3) ---------- */

/* Residual addition of two int8 tensors of n elements on grids S_x, S_y onto
 * S_z (Eqs. 1-4; the feed-forward branches enter with alpha = 1/2):
 *   z = clamp(round(2^-(31+s) (m_x x + m_y y)), -127, 127)
 * (m_x, m_y, s) from ip_residual_params (one shared shift, as Eq. 11).
 * x, y, z: device, 16-byte aligned; m_x, m_y in [0, 2^31), s in [0, 31].
 * n == 0 returns IP_OK without touching any pointer.  Asynchronous on
 * `stream`.  Returns IP_OK or IP_ERR_*. */
int ip_residual_i8(const int8_t *x, const int8_t *y, long long n, int32_t m_x, int32_t m_y,
                   int32_t s, int8_t *z, ip_stream_t stream);

/* (m_x, m_y, s) of z = x + alpha y onto S_z (host, float64). */
int ip_residual_params(double S_x, double S_y, double S_z, double alpha, int32_t *m_x,
                       int32_t *m_y, int32_t *s);

/* The ConvBlock's first pointwise convolution with the gated linear unit of
 * Eq. 5 fused: the projection x W^T onto the int8 grids of a and b (m, s per
 * row of w), then GLU(a, b) = a sigma(b), sigma(b) = (1 + tanh(b/2)) / 2 with
 * the minimax tanh:
 *   D = min(|b|, q_c) - q_c;  t = q_one + sgn(b) (q_one - D^2)
 *   y = clamp(round(2^-(31+s) m a t), -127, 127)
 * w: device int8 [N][K] with the rows of a and b interleaved (row 2c is a_c,
 * row 2c + 1 is b_c; N even, output channels N/2); bias, m, s per row as
 * ip_linear_i8; glu: host constants (ip_glu_params), q_c and q_one from S_b.
 * x: [B][T][K] row-major; y: [B][T][N/2] row-major.  Other arguments and
 * errors as ip_linear_i8. */
int ip_linear_glu_i8(const int8_t *x, const int8_t *w, const int32_t *bias, const int32_t *m,
                     const int32_t *s, const ip_swish_params *glu, int B, int T, int K, int N,
                     int8_t *y, void *workspace, size_t workspace_bytes, ip_stream_t stream);

/* A linear layer with the residual addition of its output fused (the
 * output projection, the second feed-forward projections and the second
 * pointwise convolution of the block, Eqs. 1-4): y = clamp(round(2^-(31+s_r)
 * (m_x res + m_y z)), -127, 127) with z the requantised int8 output of
 * ip_linear_i8 on (x, w, bias, m, s).  Bit-identical to ip_linear_i8 then
 * ip_residual_i8(res, z, m_x, m_y, s_r).  res: device int8 [B][T][N]
 * row-major, 16-byte aligned; it may be y itself (in place: each element
 * is read by the thread that then writes it), but a partial overlap with y
 * is rejected with IP_ERR_PARAM; m_x, m_y in [0, 2^31), s_r in [0, 31]
 * (else IP_ERR_PARAM).  x: [B][T][K] row-major; y: [B][T][N]
 * row-major.  Other arguments and errors as ip_linear_i8. */
int ip_linear_residual_i8(const int8_t *x, const int8_t *w, const int32_t *bias,
                          const int32_t *m, const int32_t *s, const int8_t *res, int32_t m_x,
                          int32_t m_y, int32_t s_r, int B, int T, int K, int N, int8_t *y,
                          void *workspace, size_t workspace_bytes, ip_stream_t stream);

/* GLU constants for the grids S_a, S_b of the two halves and S_y of the
 * output (host, float64): q_c = round(2c / S_b), q_one = round(1 / S_t),
 * S_t = |a| (S_b/2)^2, m 2^-(31+s) = S_a S_t / (2 S_y). */
int ip_glu_params(double S_a, double S_b, double S_y, ip_swish_params *out);

/* Swish constants for an INT16 input (the BatchNorm output, Sec. 3.3):
 * q_c in [1, 2^16), q_one in [1, 2^31) with q_one >= q_c^2, m, s. */
typedef struct {
    int32_t q_c;
    long long q_one;
    int32_t m, s;
} ip_swish16_params;

/* Depthwise convolution over time with BatchNorm folded into w and bias
 * (Sec. 2.2), onto the INT16 grid (Sec. 3.3), then the minimax Swish onto
 * int8 (the INT16 tensor never reaches memory):
 *   acc = sum_k w[c][k] x[b][t + k - K/2][c] + bias[c]   (zero padding)
 *   z   = clamp(round(2^-(31+s[c]) m[c] acc), -32767, 32767)
 *   y   = Swish(z) with the steps of ip_linear_swish_i8 on z's grid; the
 *         product m z t (up to 78 bits) is formed exactly.
 * x, y: device int8 [B][T][C] row-major; w: device int8 [C][K], K odd in
 * [1, 15]; bias, m, s: device int32 [C] (|bias| < 2^30, m >= 0, s in
 * [0, 31]; out-of-domain values are clamped and reported as IP_ERR_PARAM by
 * ip_relpos_mhsa_status); sw: host (IP_ERR_PARAM outside its domain).
 * Workspace as ip_relpos_mhsa_i8.  Returns IP_OK or IP_ERR_*. */
int ip_dwconv_swish_i8(const int8_t *x, int B, int T, int C, const int8_t *w, int K,
                       const int32_t *bias, const int32_t *m, const int32_t *s,
                       const ip_swish16_params *sw, int8_t *y, void *workspace,
                       size_t workspace_bytes, ip_stream_t stream);

/* Swish constants of an INT16 input grid S_z and int8 output grid S_y. */
int ip_swish16_params_from_scales(double S_z, double S_y, ip_swish16_params *out);

/* ip_relpos_mhsa_i8 with a choice of output layout: out_layout =
 * IP_LAYOUT_HEADS writes [B][H][T][dh] (as ip_relpos_mhsa_i8), IP_LAYOUT_ROWS
 * writes [B][T][H][dh], i.e. [B][T][H dh] row-major, the frames' rows that
 * the output projection (ip_linear_i8 with a row-major input) reads.  Other
 * values: IP_ERR_PARAM.  Everything else as ip_relpos_mhsa_i8. */
int ip_relpos_mhsa_i8_ex(const int8_t *q, const int8_t *k, const int8_t *v, const int8_t *p,
                         const int8_t *u, const int8_t *v_bias, const int32_t *multipliers,
                         const int32_t *shifts, const ip_isoftmax_params *sm,
                         const int32_t *lengths, int B, int H, int T, int dh, int8_t *out,
                         int out_layout, void *workspace, size_t workspace_bytes,
                         ip_stream_t stream);

/* ip_relpos_mhsa_i8_host without the final wait: enqueues the uploads, the
 * kernel and the download on `stream` and returns.  The output in `out` (and
 * the inputs' host buffers, which stay in use until the uploads are done) is
 * valid once the stream has synchronised; ip_relpos_mhsa_host_status then
 * reports device-side errors.  Calls on different streams with different
 * arenas overlap one call's copies with another's kernel.  Pinned host
 * buffers make the copies asynchronous. */
int ip_relpos_mhsa_i8_host_async(const int8_t *q, const int8_t *k, const int8_t *v,
                                 const int8_t *p, const int8_t *u, const int8_t *v_bias,
                                 const int32_t *multipliers, const int32_t *shifts,
                                 const ip_isoftmax_params *sm, const int32_t *lengths, int B,
                                 int H, int T, int dh, int8_t *out, void *arena,
                                 size_t arena_bytes, ip_stream_t stream);

/* Status of the last ip_relpos_mhsa_i8_host_async call that used `arena`
 * (same shape arguments): synchronises `stream`, returns IP_OK,
 * IP_ERR_TIMEOUT or IP_ERR_PARAM, and clears the status word. */
int ip_relpos_mhsa_host_status(const void *arena, int B, int H, int T, int dh,
                               ip_stream_t stream);

/* Text of an IP_* code. */
const char *ip_strerror(int code);

/* Test hook: bound, in SM clock cycles, of every barrier wait inside the
 * kernels launched afterwards by this process (0 = give up at the first
 * wait that is not already satisfied; negative = the default of about two
 * seconds).  A wait that runs out records IP_ERR_TIMEOUT for
 * ip_relpos_mhsa_status; the kernel lets its own copies in flight land and
 * returns. */
int ip_debug_set_timeout_cycles(long long cycles);

/* Test hook: when on, the kernels launched afterwards by this process first
 * make every consumer warp wait on a barrier that nothing arrives on, so
 * that the bounded wait runs out and the error path (IP_ERR_TIMEOUT, copies
 * in flight drained, early return) is exercised without faulting or hanging
 * the GPU.  Off by default. */
int ip_debug_set_stall_injection(int on);

/* Test hook: how the kernels launched afterwards by this process do the
 * tiles of 64 query rows.  Negative (the default): as planned, i.e. when the
 * last round of work items over the resident CTAs would be at most a
 * quarter full, its tiles are done as four quarters of 16 rows, when at most
 * half full as two halves of 32 rows, whose warps split the keys of every
 * chunk and combine their row maxima, exponential sums and attn.V partial
 * sums.  0: no tile is split.  1: every tile in halves.  2 (or more): every
 * tile in quarters.  The outputs are the same bit for bit in every mode. */
int ip_debug_set_split_mode(int mode);

/* Test hook: nonzero makes the attention kernel take its general softmax
 * arithmetic everywhere: 64-bit partial row sums even where the host has
 * shown that 32-bit partial sums cannot wrap (exp(0) x 16 ceil(T/64) <
 * 2^32), and the probability as min(floor(e f / 2^24), 255) from the full
 * 64-bit product even where every row sum exceeds 2^8 (exp(0) > 2^8, so
 * f < 2^24 and one multiply-high gives it); 0 restores the choice.  Both
 * paths compute the same integers, so the outputs are the same bit for
 * bit. */
int ip_debug_set_wide_sums(int on);

/* Diagnostic: enqueues a throughput probe of the integer warp MMA
 * (mma.sync m16n8k32 s8 x s8 -> s32, eight independent accumulators per
 * warp, `iters` rounds) on `stream`; sink is a device int array of
 * blocks * 256 entries.  Returns the number of integer ops the launch
 * performs (one multiply-add = 2), or -1 on error.  Timing it with events
 * gives the measured INT8 peak of this GPU. */
long long ip_probe_int8_mma(int blocks, int iters, int *sink, ip_stream_t stream);

/* Diagnostic: the two integer pipes at once.  In each block of 256 threads
 * the first mma_warps (0..8) warps run four integer-MMA chains for `iters`
 * rounds and the other warps eight dp4a chains for 4 iters rounds of four;
 * sink as above.  Returns the integer ops of the launch (both kinds), or -1
 * on error.  mma_warps = 0 gives the dp4a rate alone; a launch time close
 * to that of the MMA warps alone shows the two pipes working concurrently. */
long long ip_probe_int8_mix(int blocks, int iters, int mma_warps, int *sink, ip_stream_t stream);

/* ---- offline constants (host only, float64, run once per layer) -------- */

/* m, s with m 2^-(31+s) nearest to ratio, m in [2^30, 2^31) unless s is
 * clipped at 31.  ratio must be in (0, 1 - 2^-32). */
int ip_dyadic_multiplier(double ratio, int32_t *m, int32_t *s);

/* Eq. 11 multipliers of the two score branches on one shared shift s,
 * taken from the larger ratio. */
int ip_dyadic_pair(double r_c, double r_p, int32_t *m_c, int32_t *m_p, int32_t *s);

/* I-BERT exponential constants on the score grid S_s (see the struct). */
int ip_isoftmax_params_from_scale(double S_s, ip_isoftmax_params *out);

/* Every integer constant of one attention layer from its real scales
 * (offline, float64, as the paper precomputes its multipliers, Sec. 2.2
 * under Eq. 7), ready for ip_relpos_mhsa_i8:
 *   Eq. 11: the branch ratios r_c = S_Q S_K / (S_s sqrt(dh)) and
 *     r_p = S_Q S_P / (S_s sqrt(dh)) (u and v live on Q's grid, so the
 *     content and position branches carry S_Q S_K and S_Q S_P) as one
 *     dyadic pair on a shared shift (ip_dyadic_pair): multipliers[0..1] =
 *     {m_c, m_p}, shifts[0] = s_s;
 *   Eq. 7 after Eq. 9: the probabilities sit on the grid 2^-8, so the
 *     output ratio is r_o = 2^-8 S_V / S_O: multipliers[2] = m_o,
 *     shifts[1] = s_o (ip_dyadic_multiplier);
 *   the I-BERT exponential constants on S_s (ip_isoftmax_params_from_scale).
 * S_Q, S_K, S_P, S_V: the int8 grids of Q (and u, v), K, P and V; S_s: the
 * fused score's int8 grid; S_O: the output's; dh: head size (the scale of
 * Eq. 8 is 1/sqrt(dh)).  multipliers (3), shifts (2), softmax: host memory
 * owned by the caller.  Returns IP_OK; IP_ERR_NULL for a NULL output;
 * IP_ERR_PARAM when a scale is not positive and finite, dh < 1, or a ratio
 * cannot be encoded (the outputs are then left untouched). */
int ip_relpos_layer_constants(double S_Q, double S_K, double S_P, double S_V, double S_s,
                              double S_O, int dh, int32_t *multipliers, int32_t *shifts,
                              ip_isoftmax_params *softmax);

/* Per-output-channel constants of Eq. 7 for ip_linear_i8 and its variants
 * (offline, float64): weights carry one scale per output channel (Sec. 2.2),
 * so channel n < N requantises with m[n] 2^-(31+s[n]), the dyadic nearest
 * to S_x S_w[n] / S_y[n] (ip_dyadic_multiplier).  S_x: the input's grid;
 * S_w, S_y: host arrays of N weight and output grids (repeat one output grid
 * for a per-tensor output); m, s: host int32 arrays of N owned by the
 * caller.  Returns IP_OK; IP_ERR_NULL for a NULL array; IP_ERR_PARAM when
 * N < 1, a scale is not positive and finite or a ratio cannot be encoded
 * (m and s are then left untouched). */
int ip_linear_constants(double S_x, const double *S_w, const double *S_y, int N, int32_t *m,
                        int32_t *s);

#ifdef __cplusplus
}
#endif
#endif /* IP_MHSA_H */
