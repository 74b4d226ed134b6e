// Device code of the integer LayerNorm (I-Parakeet, Sec. 2.1, Eqs. 1-4, with
// the integer kernel of Sec. 2.2) for sm_103a.  Integer arithmetic only: no
// floating-point type, no division by a run-time value (d is a compile-time
// multiple of 512; the square root and the reciprocal are Newton iterations
// with multiplications only, each settled exactly by a final comparison).
//
// One warp per batch of four rows of d channels, batches dealt warp-major
// over a grid of one CTA per SM, so that every warp takes two or more
// batches and loads the next one's rows during the current pass B.  Per row: the sum and the sum of squares of the
// int8 values (dp4a, warp reduction), floor(sum c^2 / d) = d sum q^2 -
// (sum q)^2 exactly for the centred values c_i = d q_i - sum, sigma =
// isqrt(that + eps_c) (at least 1), f = floor(2^31 / sigma), and per element
// n = round(c f / 2^16), y = clamp(round((M_i n + B_i) / 2^E_i), -127, 127).
// With d = C 2^9, n is one 32-bit multiply-add and a shift of the int8
// value q itself: n = floor((q F + G) / 2^7) with F = C f and
// G = floor((2^15 - sum f) / 2^9), evaluated modulo 2^32 (see pass_a).
// Lane l takes the 16-byte segments l, l + 32, ... of the row (coalesced)
// and keeps them in registers between the two passes; the per-channel
// constants (B, M, E) of its channels sit in shared memory in lane-major
// order, one 16-byte record per channel, each read once per batch of rows.
#pragma once

#include <stdint.h>

#include "ip_ptx.cuh"

namespace ipn {

using namespace ipk;

constexpr int THREADS = 256;              // 8 warps, one batch of rows each
constexpr int NB = 4;                     // rows per warp batch
constexpr int ERR_PARAM = 16;             // a per-channel constant out of its domain

struct NormParams {
    const int8_t *x;
    int8_t *y;
    long long rows;
    long long eps_c;
    const int32_t *M;
    const long long *B;
    const int32_t *E;
    int *err;
};

// floor(sqrt(n)) for 0 <= n < 2^42 by Newton's iteration on 1 / sqrt, with
// multiplications only.  An even shift normalises n to m = n 4^k in [2^40,
// 2^42), M = m / 2^42 in [1/4, 1).  y approximates 2^30 / sqrt(M): it starts
// from the chord of that function over [1/4, 1/2) or [1/2, 1) (y0 = a - b q
// with q = M 2^10; relative error under 3 %), and each step y <- y (3 - M
// y^2) / 2, in fixed point (t = M y^2 2^60 by a 64 x 64 high product, y' =
// y (3 2^60 - t) / 2^61), squares the error: after three steps it is below
// 2^-28 with the truncations.  sqrt(m) is then m y / 2^51, and its integer
// part shifted right by k lies within one of floor(sqrt(n)); two
// comparisons each way settle it.
__device__ __forceinline__ unsigned long long isqrt_u42(unsigned long long n) {
    if (n == 0) return 0;
    const int k = (__clzll(static_cast<long long>(n)) - 22) >> 1;
    const unsigned long long m = n << (2 * k);
    const unsigned long long q = m >> 32;   // M 2^10, in [256, 1024)
    // chord of 2^30 / sqrt(q / 2^10) through q = 256, 512 and q = 512, 1024
    unsigned long long y = q < 512 ? 2776467046ull - 2456966ull * q : 1963258675ull - 868669ull * q;
#pragma unroll
    for (int it = 0; it < 3; ++it) {
        const unsigned long long t = __umul64hi(m << 22, y * y);
        y = __umul64hi(y << 32, 3ull * (1ull << 60) - t) >> 29;
    }
    unsigned long long s = (__umul64hi(m << 22, y << 10) >> 19) >> k;
    s -= s * s > n ? 1ull : 0ull;
    s -= s * s > n ? 1ull : 0ull;
    s += (s + 1) * (s + 1) <= n ? 1ull : 0ull;
    s += (s + 1) * (s + 1) <= n ? 1ull : 0ull;
    return s;
}

// floor(2^31 / s) for 1 <= s < 2^22 by Newton's iteration on the
// reciprocal of the normalised divisor, with multiplications only.  With L
// the bit length of s, x = s 2^(22-L) lies in [2^21, 2^22), X = x / 2^22 in
// [1/2, 1), and floor(2^31 / s) = floor(floor(2^52 / x) / 2^(L-1)).  r
// approximates 2^52 / x: the start 2^30 (48 - 32 X) / 17 has relative error
// at most 1/17, and each step r += r (2^52 - x r) / 2^52 squares it (three
// steps: below 2^-29 with the truncations).  q = r / 2^(L-1) is then within
// one of the quotient, and the remainder 2^31 - q s settles it.
__device__ __forceinline__ uint32_t recip_2pow31(unsigned long long s64) {
    const long long s = static_cast<long long>(s64);
    const int L = 64 - __clzll(s);
    const long long x = s << (22 - L);
    long long r = (51539607552ll - 8192ll * x) / 17;   // 2^30 (48 - 32 X) / 17
#pragma unroll
    for (int it = 0; it < 3; ++it) {
        const long long e = (1ll << 52) - x * r;       // |e| < 2^48
        r += (r * (e >> 21)) >> 31;
    }
    long long q = r >> (L - 1);
    long long rem = (1ll << 31) - q * s;
    if (rem < 0) { --q; rem += s; }
    if (rem < 0) { --q; rem += s; }
    if (rem >= s) { ++q; rem -= s; }
    if (rem >= s) { ++q; }
    return static_cast<uint32_t>(q);
}

// C = d / 512 segments of 16 channels per lane.  A warp takes NB rows at a
// time and keeps their int8 values in registers: it reduces them, lane r
// computes the square root and the reciprocal of row r (one chain of those
// scalar steps serves NB rows), then it normalises the rows from registers,
// each channel record read from shared memory once for the NB rows.  The
// segment loop stays rolled so that the code fits the instruction cache.
// Pass A of one batch of NB rows (rows past the end read as zero): the rows
// into registers, sum and sum of squares of each row (dp4a, warp
// reduction); lane r then computes floor(sum c^2 / d) = d sum q^2 -
// (sum q)^2 of row r (exact, c = d q - sum), sigma and f = floor(2^31 /
// sigma), which every lane receives for every row.
template <int C>
struct Batch {
    uint4 xv[NB][C];
    uint32_t F[NB], G[NB];   // n = floor((q F + G) / 2^7) for row r (see pass_a)
};

template <int C>
__device__ __forceinline__ void load_rows(const NormParams &prm, long long row0, int nrows, int lane,
                                          uint4 (&xv)[NB][C]) {
    constexpr int D = 512 * C;
#pragma unroll
    for (int r = 0; r < NB; ++r) {
        const int8_t *xr = prm.x + (row0 + (r < nrows ? r : 0)) * D;
#pragma unroll
        for (int j = 0; j < C; ++j)
            xv[r][j] = r < nrows ? __ldcs(reinterpret_cast<const uint4 *>(xr + j * 512 + lane * 16))
                                 : make_uint4(0u, 0u, 0u, 0u);
    }
}

template <int C>
__device__ __forceinline__ void pass_a_stats(const NormParams &prm, int lane, Batch<C> &bt) {
    constexpr int D = 512 * C;
    int sq[NB], sum[NB];
#pragma unroll
    for (int r = 0; r < NB; ++r) {
        sum[r] = 0;
        sq[r] = 0;
#pragma unroll
        for (int j = 0; j < C; ++j) {
            const uint32_t w[4] = {bt.xv[r][j].x, bt.xv[r][j].y, bt.xv[r][j].z, bt.xv[r][j].w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                sum[r] = __dp4a(static_cast<int>(w[i]), 0x01010101, sum[r]);
                sq[r] = __dp4a(static_cast<int>(w[i]), static_cast<int>(w[i]), sq[r]);
            }
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
#pragma unroll
        for (int r = 0; r < NB; ++r) {
            sum[r] += __shfl_xor_sync(0xffffffffu, sum[r], o);
            sq[r] += __shfl_xor_sync(0xffffffffu, sq[r], o);
        }
    long long ms = 0;
#pragma unroll
    for (int r = 0; r < NB; ++r)
        if (lane == r) ms = static_cast<long long>(D) * sq[r] - static_cast<long long>(sum[r]) * sum[r];
    unsigned long long sigma = isqrt_u42(static_cast<unsigned long long>(ms + prm.eps_c));
    sigma = sigma < 1 ? 1 : sigma;
    // f = floor(2^31 / sigma), held as a signed 32-bit value: f = 2^31 only
    // for sigma = 1, where sum c^2 < 4 d gives |c| < 2^7 and round(c (2^31 -
    // 1) / 2^16) = round(c 2^31 / 2^16), so 2^31 - 1 stands in exactly
    uint32_t f_own = recip_2pow31(sigma);
    f_own = f_own > 0x7fffffffu ? 0x7fffffffu : f_own;
    // n = floor(u / 2^16) with u = c f + 2^15 and c = D q - sum, D = C 2^9:
    // u = (q C f + G) 2^9 + l with G = floor((2^15 - sum f) / 2^9) and
    // 0 <= l < 2^9, so n = floor((q C f + G) / 2^7) (the fraction l / 2^9
    // never carries an integer quotient over).  With s = sqrt(sum c^2 / d +
    // eps_c), sigma >= s / 2 when s >= 1 (and every c is 0 when s < 1), and
    // |c| <= sqrt(d) s, so |c| f <= 2^32 sqrt(d) and |q C f + G| < 2^29:
    // the 32-bit multiply-add modulo 2^32 gives it exactly.
#pragma unroll
    for (int r = 0; r < NB; ++r) {
        const uint32_t f = __shfl_sync(0xffffffffu, f_own, r);
        bt.F[r] = static_cast<uint32_t>(C) * f;
        const long long g = ((1ll << 15) - static_cast<long long>(sum[r]) * static_cast<long long>(f)) >> 9;
        bt.G[r] = static_cast<uint32_t>(g);
    }
}

// Pass B of one batch: normalise and requantise the rows from registers;
// each channel record serves the NB rows.  The segment loop stays rolled so
// that the code fits the instruction cache.
template <int C, bool HI>
__device__ __forceinline__ void pass_b(const NormParams &prm, const uint4 *cst, long long row0,
                                       int nrows, int lane, const Batch<C> &bt) {
    constexpr int D = 512 * C;
#pragma unroll 1
    for (int j = 0; j < C; ++j) {
        uint4 xj[NB];
#pragma unroll
        for (int r = 0; r < NB; ++r) xj[r] = bt.xv[r][0];
#pragma unroll
        for (int jj = 1; jj < C; ++jj)
            if (j == jj) {
#pragma unroll
                for (int r = 0; r < NB; ++r) xj[r] = bt.xv[r][jj];
            }
        uint32_t o[NB][4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          // bytes 3 and 2 first, packed as soon as both are there
          int t[NB][4];
          uint32_t hi2[NB];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int ee = 3 - k;
            const int e = 4 * i + ee;
            const uint4 rec = cst[(j * 16 + e) * 32 + lane];
            const long long b = static_cast<long long>((static_cast<unsigned long long>(rec.y) << 32) | rec.x);
#pragma unroll
            for (int r = 0; r < NB; ++r) {
                const uint32_t w[4] = {xj[r].x, xj[r].y, xj[r].z, xj[r].w};
                const uint32_t q = static_cast<uint32_t>(sbyte(w[i], ee));
                const int n = static_cast<int>(q * bt.F[r] + bt.G[r]) >> 7;   // |n| < 2^23
                // floor(v / 2^E), |v| < 2^62: with every E >= 32 the high word
                // shifted by E - 32 (the record holds E - 32), else
                // floor(v / 2^31) (a 32-bit value) shifted by E - 31
                const long long v = static_cast<long long>(static_cast<int>(rec.z)) * n + b;
                int h;
                if (HI)
                    h = static_cast<int>(static_cast<uint32_t>(static_cast<unsigned long long>(v) >> 32));
                else
                    h = static_cast<int>(__funnelshift_r(static_cast<uint32_t>(v),
                                                         static_cast<uint32_t>(v >> 32), 31));
                t[r][ee] = max(h >> static_cast<int>(rec.w), -127);   // 127 by the saturating pack
                if (ee == 2) hi2[r] = pack_sat2(t[r][3], t[r][2], 0u);
                if (ee == 0) o[r][i] = pack_sat2(t[r][1], t[r][0], hi2[r]);
            }
          }
        }
#pragma unroll
        for (int r = 0; r < NB; ++r)
            if (r < nrows)
                __stcs(reinterpret_cast<uint4 *>(prm.y + (row0 + r) * D + j * 512 + lane * 16),
                       make_uint4(o[r][0], o[r][1], o[r][2], o[r][3]));
    }
}

template <int C>
__device__ __forceinline__ void pass_a(const NormParams &prm, long long row0, int nrows, int lane,
                                       Batch<C> &bt) {
    load_rows<C>(prm, row0, nrows, lane, bt.xv);
    pass_a_stats<C>(prm, lane, bt);
}

// The batches of one warp after the first one's pass A: the next batch's
// rows are loaded before the current batch's pass B, so their latency
// hides behind it.
template <int C, bool HI>
__device__ __forceinline__ void run_batches(const NormParams &prm, const uint4 *cst, long long grp,
                                            long long warps, long long groups, int lane,
                                            Batch<C> &bt) {
    for (;;) {
        const long long row0 = grp * NB;
        const int nrows = prm.rows - row0 < NB ? static_cast<int>(prm.rows - row0) : NB;
        const long long nxt = grp + warps;
        uint4 xn[NB][C];
        if (nxt < groups) {
            const long long nrow0 = nxt * NB;
            load_rows<C>(prm, nrow0, prm.rows - nrow0 < NB ? static_cast<int>(prm.rows - nrow0) : NB,
                         lane, xn);
        }
        pass_b<C, HI>(prm, cst, row0, nrows, lane, bt);
        if (nxt >= groups) break;
        grp = nxt;
#pragma unroll
        for (int r = 0; r < NB; ++r)
#pragma unroll
            for (int j = 0; j < C; ++j) bt.xv[r][j] = xn[r][j];
        pass_a_stats<C>(prm, lane, bt);
    }
}

// C = d / 512 segments of 16 channels per lane.  A warp takes NB rows at a
// time and keeps their int8 values in registers: pass A reduces them (lane
// r computes the square root and the reciprocal of row r, one chain of
// those scalar steps for NB rows), pass B normalises them.  The first
// batch's pass A runs before the channel records are built, so its loads
// overlap that set-up.
template <int C>
__global__ void __launch_bounds__(THREADS, 1)
    layernorm_i8_kernel(const NormParams prm) {
    constexpr int D = 512 * C;
    extern __shared__ uint8_t smem_raw[];
    uint4 *cst = reinterpret_cast<uint4 *>(smem_raw);   // [C * 16][32] records
    const int lane = threadIdx.x & 31;
    // Batches are dealt warp-major (warp w of CTA c takes batch w G + c, then
    // that plus 8 G, ...), so that with fewer batches than warps every CTA,
    // and every SM, keeps about the same number of busy warps.
    const long long warps = static_cast<long long>(gridDim.x) * (THREADS / 32);
    const long long groups = (prm.rows + NB - 1) / NB;
    long long grp = static_cast<long long>(threadIdx.x >> 5) * gridDim.x + blockIdx.x;

    Batch<C> bt;
    const bool first = grp < groups;
    pdl_launch_dependents();
    pdl_wait();   // the grid before this one on the stream: complete, memory visible
    if (first) {
        const long long row0 = grp * NB;
        pass_a<C>(prm, row0, prm.rows - row0 < NB ? static_cast<int>(prm.rows - row0) : NB, lane, bt);
    }

    // per-channel records {B' lo, B' hi, M, E - 31} with B' = B + 2^(E-1)
    // (the rounding term folded in): channel j 512 + l 16 + e of lane l goes
    // to record (j 16 + e) 32 + l.  When every E is at least 32 the records
    // hold E - 32 and pass B shifts the high word of M n + B'.
    bool bad = false, hi = true;
    for (int k = threadIdx.x; k < D; k += THREADS) {
        const int j = k >> 9, l = (k >> 4) & 31, e = k & 15;
        long long b = prm.B[k];
        int m = prm.M[k], ex = prm.E[k];
        if (ex < 31 || ex > 62 || b >= (1ll << 60) || b <= -(1ll << 60)) {
            bad = true;
            ex = ex < 31 ? 31 : (ex > 62 ? 62 : ex);
            b = 0;
        }
        b += 1ll << (ex - 1);
        hi = hi && ex >= 32;
        cst[(j * 16 + e) * 32 + l] =
            make_uint4(static_cast<uint32_t>(b), static_cast<uint32_t>(static_cast<unsigned long long>(b) >> 32),
                       static_cast<uint32_t>(m), static_cast<uint32_t>(ex - 31));
    }
    if (bad) atomicOr(prm.err, ERR_PARAM);
    const bool all_hi = __syncthreads_and(hi) != 0;
    if (all_hi) {
        for (int k = threadIdx.x; k < D; k += THREADS) {
            const int j = k >> 9, l = (k >> 4) & 31, e = k & 15;
            cst[(j * 16 + e) * 32 + l].w -= 1u;
        }
        __syncthreads();
    }
    if (!first) return;
    if (all_hi)
        run_batches<C, true>(prm, cst, grp, warps, groups, lane, bt);
    else
        run_batches<C, false>(prm, cst, grp, warps, groups, lane, bt);
}

}  // namespace ipn
