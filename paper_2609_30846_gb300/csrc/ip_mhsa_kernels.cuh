// Device code of the integer-only relative-positional MHSA (I-Parakeet,
// Sec. 3.1) for sm_103a.  Integer arithmetic only: no floating-point type
// appears in this file, and no division by a run-time value (the two
// divisions the method needs are done by binary long division).
//
// sm_103a has no integer tcgen05 MMA kind, so the three contractions use the
// integer warp MMA (mma.sync m16n8k32, s8 x s8 and u8 x s8 -> s32, which
// runs on the tensor pipe), fed from shared-memory tiles that the tensor
// memory accelerator (TMA) stages with the 128-byte swizzle.
//
// The CTAs are persistent (one per resident slot) and take work items in
// turn: a whole 64-row tile of one (b, h), or, for the tail of the work, a
// 32-row half of one.  Four consumer warps of 16 rows and two producer
// warps: the copy warp issues the TMA loads through a two-stage ring that
// runs on across items (the next item's first chunks are in flight while
// the current one finishes), and the bias warp computes the bias vectors
// K u and P v of each staged score-pass chunk (the exact rank-1 split of
// (Q + 1u^T)K^T and (Q + 1v^T)P^T, since Q + u does not fit an int8
// operand).  The attn.V pass reads the V tile as TMA stages it: transposed
// ldmatrix loads and byte selects build the MMA operand.
// The consumers, per item:
//   pass 1  for each chunk of 64 keys: the content MMAs Q K^T, the MMAs of
//           the position band Q P_band^T for the next chunk (issued before
//           this chunk's epilogue so that the tensor pipe stays busy; the 16
//           band columns it shares with this chunk are carried over), the
//           relative shift as an index remap through shared memory, the
//           fused requantisation of Eq. 11 and the key mask; int8 scores
//           stay in shared memory, row maxima in registers;
//   pass 2  integer exponentials (a 256-entry table, one copy per row
//           group to spread the banks) and row sums;
//   pass 3  probabilities on the grid 2^-8 as the u8 operand of the A.V
//           MMA, then the output requantisation and 4-byte stores.
#pragma once

#include <cuda.h>
#include <stdint.h>

#include "ip_ptx.cuh"

namespace ipk {

constexpr int DH = 128;
constexpr int MROWS = 64;                 // query rows per CTA
constexpr int NCWARPS = 4;                // consumer warps, 16 rows each
constexpr int NPWARPS = 2;                // producer warps: the copy warp and the bias warp
constexpr int NTHREADS = (NCWARPS + NPWARPS) * 32;
constexpr int NK = 64;                    // keys per chunk
constexpr int NSTAGE = 2;
constexpr int BAND_ROWS = 128;            // P rows staged per chunk (NK + MROWS - 1, padded)
constexpr int K_TILE_BYTES = NK * DH;     // K (pass 1) or V (pass 3) tile
constexpr int P_TILE_BYTES = BAND_ROWS * DH;   // P band (pass 1) or transposed V (pass 3)
constexpr int KU_OFF = K_TILE_BYTES + P_TILE_BYTES;   // int32 K u of the chunk's keys
constexpr int PV_OFF = KU_OFF + NK * 4;                // int32 P v of the band rows
constexpr int STAGE_BYTES = 25600;        // PV_OFF + BAND_ROWS * 4, rounded to 1024
constexpr int BAND_TILES = 10;            // n8 tiles of one warp's band: 16 + NK - 1 -> 80
constexpr int CARRY_TILES = BAND_TILES - NK / 8;   // band tiles shared by consecutive chunks
constexpr int REMAP_STRIDE = 88;          // int32 words per band row in the remap buffer
constexpr int REMAP_BYTES = 16 * REMAP_STRIDE * 4;
constexpr int LUT_ENTRIES = 256;
constexpr int LUT_COPIES = 4;             // row groups g and g + 4 share one
constexpr int CHUNK_SCORE_BYTES = 16 * NK;   // one warp's int8 scores of one chunk
constexpr int Q_TILE_BYTES = MROWS * DH;  // the Q rows of the current item

static_assert(PV_OFF + BAND_ROWS * 4 <= STAGE_BYTES, "stage layout");
static_assert(STAGE_BYTES % 1024 == 0, "the 128-byte swizzle needs 1024-byte aligned tiles");
static_assert(CARRY_TILES == 2 && (BAND_TILES - CARRY_TILES) % 4 == 0, "band tiling");

struct SmemLayout {
    int stages, qtile, scores, remap, lut, bars, total;
};

// Offsets from a 1024-byte aligned base.  With global_scores the consumer
// warps keep their int8 scores in the caller's workspace instead (ScoreBuf).
__host__ __device__ inline SmemLayout smem_layout(int nchunk_max, bool global_scores = false) {
    SmemLayout L;
    L.stages = 0;
    L.qtile = NSTAGE * STAGE_BYTES;   // 1024-byte aligned (128-byte swizzle); Ring::qtile
    L.scores = L.qtile + Q_TILE_BYTES;
    L.remap = L.scores + (global_scores ? 0 : NCWARPS * nchunk_max * CHUNK_SCORE_BYTES);
    L.lut = L.remap + NCWARPS * REMAP_BYTES;
    L.bars = L.lut + LUT_ENTRIES * LUT_COPIES * 4;
    L.total = L.bars + 128;
    return L;
}

struct FusedParams {
    const int8_t *u;          // [H][DH]
    const int8_t *vb;         // [H][DH]
    int8_t *out;
    const int32_t *lengths;   // [B] or nullptr
    int *err;                 // device error word
    int B, H, T, nchunk_max;
    int32_t m_c, m_p, m_o;
    int32_t sh_s, sh_o;       // total right shifts, 31 + s
    int32_t q_ln2, q_b, q_c;
    unsigned long long ln2_magic;   // udiv_magic constant of q_ln2
    long long timeout_cycles; // bound of every barrier wait
    int stall_injection;      // test hook: consumers first wait on a barrier nobody arrives on
    int sum32;                // exp(0) x 16 nchunk_max < 2^32: 32-bit partial sums in pass 2
    int f24;                  // exp(0) > 2^8: every row sum exceeds 2^8, so f = 2^32 / sum < 2^24
    // Work items, claimed in order by the persistent CTAs: items [0, nwhole)
    // are whole 64-row tiles in (b, h, tile) order, items [nwhole, nitems)
    // the 2^split_log2 parts (32-row halves or 16-row quarters) of the tiles
    // from nwhole on.
    unsigned int *sched;      // workspace words: [0] next item, [16] CTAs done claiming
    int ntiles;                        // 64-row tiles per (b, h)
    unsigned long long tiles_magic;    // udiv_magic constant of ntiles
    unsigned long long heads_magic;    // udiv_magic constant of H
    uint32_t nwhole, nitems;           // nitems < 2^31
    int split_log2;                    // 1: halves, 2: quarters
    int out_rows;             // output [B][T][H][DH] instead of [B][H][T][DH]
    uint8_t *gscores;         // global mode: score slices, NCWARPS per CTA, nchunk_max KB each
};

// Where a consumer warp keeps the int8 scores of its 16 rows between the
// three passes (CHUNK_SCORE_BYTES per key chunk, each thread's bytes at the
// same offsets in both places): its slice of shared memory, or, for long
// sequences whose slices would leave room for one CTA per SM only, a slice
// of the caller's workspace in global memory (written and read back by the
// same thread, cached in L2).
struct ScoreBuf {
    uint32_t s;    // shared-memory address of the slice
    uint8_t *g;    // global address of the slice
};

template <bool GS>
__device__ __forceinline__ void sc_st128(const ScoreBuf &b, uint32_t off, uint32_t x, uint32_t y,
                                         uint32_t z, uint32_t w) {
    if constexpr (GS) stg128_cg(b.g + off, x, y, z, w);
    else sts128(b.s + off, x, y, z, w);
}

template <bool GS>
__device__ __forceinline__ uint4 sc_ld128(const ScoreBuf &b, uint32_t off) {
    if constexpr (GS) return ldg128_cg(b.g + off);
    else return lds128(b.s + off);
}

template <bool GS>
__device__ __forceinline__ void sc_st64(const ScoreBuf &b, uint32_t off, int x, int y) {
    if constexpr (GS) stg64_cg(b.g + off, x, y);
    else sts64(b.s + off, x, y);
}

template <bool GS>
__device__ __forceinline__ int2 sc_ld64(const ScoreBuf &b, uint32_t off) {
    if constexpr (GS) return ldg64_cg(b.g + off);
    else return lds64(b.s + off);
}

// Offset of output row `row` of (b, h).
__device__ __forceinline__ size_t out_offset(const FusedParams &p, int b, int h, int row) {
    return p.out_rows ? ((static_cast<size_t>(b) * p.T + row) * p.H + h) * DH
                      : ((static_cast<size_t>(b) * p.H + h) * p.T + row) * DH;
}

constexpr uint32_t NO_ITEM = 0xffffffffu;
constexpr int ERR_TIMEOUT_FULL = 1;
constexpr int ERR_TIMEOUT_EMPTY = 2;
constexpr int ERR_TIMEOUT_READY = 4;
constexpr int ERR_TIMEOUT_INJECTED = 8;
constexpr long long DRAIN_CYCLES = 2000000000ll;

// ---------------------------------------------------------------- helpers --

// Byte transpose of a 4x4 block: y_c = [x0.b_c, x1.b_c, x2.b_c, x3.b_c].
__device__ __forceinline__ void transpose4(uint32_t x0, uint32_t x1, uint32_t x2, uint32_t x3,
                                           uint32_t &y0, uint32_t &y1, uint32_t &y2,
                                           uint32_t &y3) {
    const uint32_t t0 = __byte_perm(x0, x1, 0x5140);
    const uint32_t t1 = __byte_perm(x0, x1, 0x7362);
    const uint32_t t2 = __byte_perm(x2, x3, 0x5140);
    const uint32_t t3 = __byte_perm(x2, x3, 0x7362);
    y0 = __byte_perm(t0, t2, 0x5410);
    y1 = __byte_perm(t0, t2, 0x7632);
    y2 = __byte_perm(t1, t3, 0x5410);
    y3 = __byte_perm(t1, t3, 0x7632);
}

// Packs the low bytes of four values: [a.b0, b.b0, c.b0, d.b0].
__device__ __forceinline__ uint32_t pack4(uint32_t a, uint32_t b, uint32_t c, uint32_t d) {
    return __byte_perm(__byte_perm(a, b, 0x0040), __byte_perm(c, d, 0x0040), 0x5410);
}

// Table indices of the four scores of a packed word (rows g, g, g + 8,
// g + 8): the row maximum minus the score, 0 .. 255 since the maximum is
// at least every score of its row (masked keys, -128, included).  With
// every byte offset by 128 no byte difference borrows from the next, so
// one 32-bit subtraction gives all four.  mx4h: the maxima of the word's
// rows, offset by 128, in the word's byte order.
__device__ __forceinline__ uint32_t exp_index4(uint32_t w, uint32_t mx4h) {
    return mx4h - (w ^ 0x80808080u);
}

__device__ __forceinline__ uint32_t max4h(int mx0, int mx1) {
    const uint32_t a = static_cast<uint32_t>(mx0 + 128) & 0xffu;
    const uint32_t b = static_cast<uint32_t>(mx1 + 128) & 0xffu;
    return a | (a << 8) | (b << 16) | (b << 24);
}

// Address of the exp table entry of byte e of an index word.
__device__ __forceinline__ uint32_t lut_at(uint32_t lut_g, uint32_t d4, int e) {
    return lut_g + ((d4 >> (8 * e)) & 0xffu) * (LUT_COPIES * 4);
}

// B fragments of the attn.V MMA for keys 32 ks .. 32 ks + 31 of the staged
// V tile (keys as rows, 128-byte swizzle) and the 16 values of d in chunk c,
// with no transposed copy of V: ldmatrix.trans on 16-bit elements hands
// thread (g, t) the byte pairs (d = 16c + 2g, 16c + 2g + 1) of keys 2t, 2t + 1
// (r0), 8 + 2t, 9 + 2t (r1) and the same + 16 (r2, r3); byte selects split
// them into the fragment of the even d (n-tile 2c) and of the odd d (n-tile
// 2c + 1).  The k order, keys 2t, 2t + 1, 8 + 2t, 9 + 2t then + 16, is the one
// of the probability operand (prob_operand).  N-tile 2c + p holds d =
// 16c + 2n + p in its column n.
__device__ __forceinline__ void vfrag(uint32_t vtile, int ks, int c, int lane, uint32_t &b0e,
                                      uint32_t &b1e, uint32_t &b0o, uint32_t &b1o) {
    const int key = 32 * ks + 8 * (lane >> 3) + (lane & 7);
    uint32_t r0, r1, r2, r3;
    ldsm_x4_trans(vtile + swz(key, c), r0, r1, r2, r3);
    b0e = __byte_perm(r0, r1, 0x6420);
    b1e = __byte_perm(r2, r3, 0x6420);
    b0o = __byte_perm(r0, r1, 0x7531);
    b1o = __byte_perm(r2, r3, 0x7531);
}

// floor(2^32 / s) for s >= 2 by restoring binary long division (the
// quotient is at most 2^31).  With 2^(L-1) <= s < 2^L the quotient is at
// most 2^(33-L), so the digits start at bit 33 - L.
__device__ __forceinline__ uint32_t div_2pow32(unsigned long long s) {
    if (s > (1ull << 32)) return 0u;
    unsigned long long rem = 1ull << 32;
    uint32_t quo = 0;
    const int top = __clzll(static_cast<long long>(s)) - 31;   // 33 - L
#pragma unroll 1
    for (int bit = top < 31 ? top : 31; bit >= 0; --bit) {
        const unsigned long long t = s << bit;
        if (t <= rem) {
            rem -= t;
            quo |= 1u << bit;
        }
    }
    return quo;
}

// I-BERT integer exponential of d = -nd (0 <= nd < 512): z = floor(nd /
// q_ln2) (exact multiply-high by the constant of q_ln2), p = -nd + z q_ln2,
// ((p + q_b)^2 + q_c) >> z.
__device__ __forceinline__ uint32_t iexp_neg(int nd, int q_ln2, int q_b, int q_c,
                                             unsigned long long ln2_magic) {
    const int z = static_cast<int>(udiv_magic(static_cast<uint32_t>(nd), ln2_magic));
    const long long p = -static_cast<long long>(nd) + static_cast<long long>(z) * q_ln2;
    const long long t = p + q_b;
    const long long L = t * t + q_c;
    if (z >= 63) return 0u;
    return static_cast<uint32_t>(L >> z);
}

// ---------------------------------------------------------- consumer parts --

// Position band of one warp: acc[nt] = Pv + Q P_band^T over 80 band columns
// (P rows rw0 .. rw0 + 79, staged at ptile rows 0 .. 79; pv = shared address
// of their P v).  Tiles go in groups of five so that the two MMAs into one
// accumulator are separated by four independent ones.
__device__ __forceinline__ void band_mma(int (&acc)[BAND_TILES][4], const uint32_t (&qa)[4][4],
                                         uint32_t ptile, uint32_t pv, int lane) {
    const int t4 = lane & 3;
#pragma unroll
    for (int nt = 0; nt < BAND_TILES; ++nt) {
        const int2 v = lds64(pv + (nt * 8 + 2 * t4) * 4);
        acc[nt][0] = v.x;
        acc[nt][1] = v.y;
        acc[nt][2] = v.x;
        acc[nt][3] = v.y;
    }
    const int lm_row = lane & 7, lm_mat = lane >> 3;
#pragma unroll
    for (int grp = 0; grp < BAND_TILES; grp += 5) {
#pragma unroll
        for (int kh = 0; kh < 2; ++kh) {
            uint32_t b[5][4];
#pragma unroll
            for (int i = 0; i < 5; ++i)
                ldsm_x4(ptile + swz((grp + i) * 8 + lm_row, kh * 4 + lm_mat), b[i][0], b[i][1],
                        b[i][2], b[i][3]);
#pragma unroll
            for (int i = 0; i < 5; ++i) mma_s8s8(acc[grp + i], qa[2 * kh], b[i][0], b[i][1]);
#pragma unroll
            for (int i = 0; i < 5; ++i) mma_s8s8(acc[grp + i], qa[2 * kh + 1], b[i][2], b[i][3]);
        }
    }
}

// Content scores of one warp: acc[nt] = Ku + Q K^T over the chunk's 64 keys
// (ku = shared address of the chunk's K u).
__device__ __forceinline__ void content_mma(int (&acc)[8][4], const uint32_t (&qa)[4][4],
                                            uint32_t ktile, uint32_t ku, int lane) {
    const int t4 = lane & 3;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
        const int2 v = lds64(ku + (nt * 8 + 2 * t4) * 4);
        acc[nt][0] = v.x;
        acc[nt][1] = v.y;
        acc[nt][2] = v.x;
        acc[nt][3] = v.y;
    }
    const int lm_row = lane & 7, lm_mat = lane >> 3;
#pragma unroll
    for (int grp = 0; grp < 8; grp += 4) {
#pragma unroll
        for (int kh = 0; kh < 2; ++kh) {
            uint32_t b[4][4];
#pragma unroll
            for (int i = 0; i < 4; ++i)
                ldsm_x4(ktile + swz((grp + i) * 8 + lm_row, kh * 4 + lm_mat), b[i][0], b[i][1],
                        b[i][2], b[i][3]);
#pragma unroll
            for (int i = 0; i < 4; ++i) mma_s8s8(acc[grp + i], qa[2 * kh], b[i][0], b[i][1]);
#pragma unroll
            for (int i = 0; i < 4; ++i) mma_s8s8(acc[grp + i], qa[2 * kh + 1], b[i][2], b[i][3]);
        }
    }
}

// Eq. 11 for one n8 tile of the content accumulator: the fused int8 scores
// of rows g, g+8 and keys 8nt + 2t, 8nt + 2t + 1 (Phi as the index remap
// jj - rho + 15 into the band), key mask, running row maxima; returns the
// four scores packed [g:2t, g:2t+1, g+8:2t, g+8:2t+1].
template <bool MASK>
__device__ __forceinline__ uint32_t score_tile(const int (&c)[4], int nt, uint32_t remap, int lane,
                                               long long m_c, long long m_p, long long half_s,
                                               int s_s, int kvalid, int &mx0, int &mx1) {
    const int g = lane >> 2, t4 = lane & 3;
    uint32_t v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const int rho = g + ((e >> 1) << 3);
        const int jj = nt * 8 + 2 * t4 + (e & 1);
        const int qp = static_cast<int>(lds32(remap + (rho * (REMAP_STRIDE - 1) + jj + 15) * 4));
        // |x| < 2^55, so x >> 31 fits 32 bits; >> (31 + s_s) = (x >> 31) >> s_s
        const long long x = m_c * c[e] + m_p * qp + half_s;
        const int y = static_cast<int>(__funnelshift_r(static_cast<uint32_t>(x),
                                                       static_cast<uint32_t>(x >> 32), 31));
        int sc = min(max(y >> s_s, -127), 127);
        if (MASK && jj >= kvalid) sc = -128;
        if (e < 2) mx0 = max(mx0, sc);
        else mx1 = max(mx1, sc);
        v[e] = static_cast<uint32_t>(sc);
    }
    return pack4(v[0], v[1], v[2], v[3]);
}

// Eq. 11 for a whole chunk (8 tiles) and the store of the packed scores.
template <bool MASK, bool GS>
__device__ __forceinline__ void score_epilogue(const int (&cacc)[8][4], uint32_t remap,
                                               const ScoreBuf &sb, uint32_t soff, int lane,
                                               long long m_c, long long m_p, long long half_s,
                                               int s_s, int kvalid, int &mx0, int &mx1) {
    uint32_t packed[8];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt)
        packed[nt] = score_tile<MASK>(cacc[nt], nt, remap, lane, m_c, m_p, half_s, s_s, kvalid,
                                      mx0, mx1);
    sc_st128<GS>(sb, soff + lane * 16, packed[0], packed[1], packed[2], packed[3]);
    sc_st128<GS>(sb, soff + 512 + lane * 16, packed[4], packed[5], packed[6], packed[7]);
}

// Sum of the integer exponentials of one stored half chunk (16 scores per
// thread: rows g and g+8, 8 keys each), in 64 bits.
template <bool MASK>
__device__ __forceinline__ void exp_sums(uint4 sv, uint32_t lut_g, uint32_t mx4h, int t4,
                                         int kbase, int kvalid, unsigned long long &s0,
                                         unsigned long long &s1) {
    const uint32_t wv[4] = {sv.x, sv.y, sv.z, sv.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t d4 = exp_index4(wv[q], mx4h);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            uint32_t ev = lds32(lut_at(lut_g, d4, e));
            if (MASK && kbase + q * 8 + 2 * t4 + (e & 1) >= kvalid) ev = 0u;
            if (e < 2) s0 += ev;
            else s1 += ev;
        }
    }
}

// The same in four 32-bit partial sums (a[0], a[1]: row g; a[2], a[3]: row
// g + 8), for calls whose exp(0) times the terms a thread adds per row
// stays below 2^32 (the host checks it), so no partial sum wraps.
template <bool MASK>
__device__ __forceinline__ void exp_sums32(uint4 sv, uint32_t lut_g, uint32_t mx4h, int t4,
                                           int kbase, int kvalid, uint32_t (&a)[4]) {
    const uint32_t wv[4] = {sv.x, sv.y, sv.z, sv.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const uint32_t d4 = exp_index4(wv[q], mx4h);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            uint32_t ev = lds32(lut_at(lut_g, d4, e));
            if (MASK && kbase + q * 8 + 2 * t4 + (e & 1) >= kvalid) ev = 0u;
            a[(e >> 1) * 2 + (q & 1)] += ev;
        }
    }
}

template <bool B> struct BoolTag {
    static constexpr bool value = B;
};

// Probabilities of one packed score word (rows g, g+8 x two keys) on the
// grid 2^-8: min(floor(ev f / 2^24), 255).  Masked keys (score -128) are
// zeroed by the caller.  F24: every row sum exceeds 2^8, so f < 2^24 and
// the callers pass f0, f1 times 2^8: the floor is then the high word of
// ev (f 2^8).  Otherwise, with ev f = hi 2^32 + lo, it is 255 when hi > 0,
// else lo >> 24 (at most 255).
template <bool F24>
__device__ __forceinline__ uint32_t prob_word(uint32_t wv, uint32_t lut_g, uint32_t mx4h,
                                              uint32_t f0, uint32_t f1) {
    const uint32_t d4 = exp_index4(wv, mx4h);
    uint32_t a[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const uint32_t f = e < 2 ? f0 : f1;
        const uint32_t ev = lds32(lut_at(lut_g, d4, e));
        if (F24)
            a[e] = min(__umulhi(ev, f), 255u);
        else
            a[e] = __umulhi(ev, f) != 0u ? 255u : (ev * f) >> 24;
    }
    return pack4(a[0], a[1], a[2], a[3]);
}

// Byte mask of a probability word of tile q of a 32-key step whose first
// key is kbase: keys kbase + 8q + 2t (bytes 0, 2) and + 1 (bytes 1, 3)
// are kept when below kvalid.
__device__ __forceinline__ uint32_t key_mask(int kbase, int q, int t4, int kvalid) {
    const int k0 = kbase + 8 * q + 2 * t4;
    return (k0 < kvalid ? 0x00ff00ffu : 0u) | (k0 + 1 < kvalid ? 0xff00ff00u : 0u);
}

// The u8 A operand of the A.V MMA from the four probability words of a
// 32-key step (k order: keys 2t, 2t+1, 8+2t, 9+2t, then the same + 16).
__device__ __forceinline__ void prob_operand(const uint32_t (&pw)[4], uint32_t (&af)[4]) {
    af[0] = __byte_perm(pw[0], pw[1], 0x5410);
    af[1] = __byte_perm(pw[0], pw[1], 0x7632);
    af[2] = __byte_perm(pw[2], pw[3], 0x5410);
    af[3] = __byte_perm(pw[2], pw[3], 0x7632);
}

// ------------------------------------------------------- split-tile parts --
// In a split tile the two warps of a row strip take the key halves
// [32 hk, 32 hk + 32) of every chunk.  Exchange area in each warp's remap
// buffer (after its score pass): row maxima, exponential sums, and the
// attn.V partial sums that the partner warp finishes.
constexpr int XMAX_OFF = 0;      // 32 lanes x 2 int32
constexpr int XSUM_OFF = 256;    // 32 lanes x 2 uint64
constexpr int XO_OFF = 768;      // 32 words x 32 lanes
static_assert(XO_OFF + 32 * 32 * 4 <= REMAP_BYTES, "exchange area");

// Band n-tiles nt0 .. nt0 + 5 and content n-tiles nt0 .. nt0 + 3 of one
// key half (nt0 = 4 hk): the band columns of keys 32 hk .. 32 hk + 31 of 16
// rows are 32 hk .. 32 hk + 46.
__device__ __forceinline__ void half_chunk_mma(int (&bacc)[6][4], int (&cacc)[4][4],
                                               const uint32_t (&qa)[4][4], uint32_t ptile,
                                               uint32_t pv, uint32_t ktile, uint32_t ku, int nt0,
                                               int lane) {
    const int t4 = lane & 3;
#pragma unroll
    for (int i = 0; i < 6; ++i) {
        const int2 v = lds64(pv + ((nt0 + i) * 8 + 2 * t4) * 4);
        bacc[i][0] = v.x;
        bacc[i][1] = v.y;
        bacc[i][2] = v.x;
        bacc[i][3] = v.y;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int2 v = lds64(ku + ((nt0 + i) * 8 + 2 * t4) * 4);
        cacc[i][0] = v.x;
        cacc[i][1] = v.y;
        cacc[i][2] = v.x;
        cacc[i][3] = v.y;
    }
    const int lm_row = lane & 7, lm_mat = lane >> 3;
#pragma unroll
    for (int kh = 0; kh < 2; ++kh) {
        uint32_t b[6][4], kb[4][4];
#pragma unroll
        for (int i = 0; i < 6; ++i)
            ldsm_x4(ptile + swz((nt0 + i) * 8 + lm_row, kh * 4 + lm_mat), b[i][0], b[i][1],
                    b[i][2], b[i][3]);
#pragma unroll
        for (int i = 0; i < 4; ++i)
            ldsm_x4(ktile + swz((nt0 + i) * 8 + lm_row, kh * 4 + lm_mat), kb[i][0], kb[i][1],
                    kb[i][2], kb[i][3]);
#pragma unroll
        for (int i = 0; i < 6; ++i) mma_s8s8(bacc[i], qa[2 * kh], b[i][0], b[i][1]);
#pragma unroll
        for (int i = 0; i < 4; ++i) mma_s8s8(cacc[i], qa[2 * kh], kb[i][0], kb[i][1]);
#pragma unroll
        for (int i = 0; i < 6; ++i) mma_s8s8(bacc[i], qa[2 * kh + 1], b[i][2], b[i][3]);
#pragma unroll
        for (int i = 0; i < 4; ++i) mma_s8s8(cacc[i], qa[2 * kh + 1], kb[i][2], kb[i][3]);
    }
}

// Sends the partial sums of the partner's output n-tiles (8 (1 - HK) ..
// + 7) to this warp's exchange area.
template <int HK>
__device__ __forceinline__ void send_partial(const int (&oacc)[16][4], uint32_t xo, int lane) {
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int e = 0; e < 4; ++e)
            sts32(xo + ((i * 4 + e) * 32 + lane) * 4, static_cast<uint32_t>(oacc[8 * (1 - HK) + i][e]));
}

// Adds the partner's partial sums of this warp's n-tiles 8 HK .. 8 HK + 7
// (d = 64 HK .. 64 HK + 63), requantises them (Eq. 7) and stores four bytes
// per row and d chunk: d = 16c + 4t .. 16c + 4t + 3 for c in 4 HK .. 4 HK + 3.
template <int HK>
__device__ __forceinline__ void finish_half(int (&oacc)[16][4], uint32_t pxo, int lane, int wrow0,
                                            int len, const FusedParams &prm, int b, int h,
                                            long long m_o, long long half_o) {
    const int T = prm.T, sh_o = prm.sh_o;
    const int g = lane >> 2, t4 = lane & 3;
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int e = 0; e < 4; ++e)
            oacc[8 * HK + i][e] += static_cast<int>(lds32(pxo + ((i * 4 + e) * 32 + lane) * 4));
#pragma unroll
    for (int rr = 0; rr < 2; ++rr) {
        const int row = wrow0 + g + 8 * rr;
        if (row >= T) continue;
        int8_t *dst = prm.out + out_offset(prm, b, h, row) + 4 * t4;
#pragma unroll
        for (int c = 4 * HK; c < 4 * HK + 4; ++c) {
            uint32_t w = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                // byte e: d = 16c + 4t + e = n-tile 2c + (e & 1), column 2t + (e >> 1)
                const long long x = m_o * oacc[2 * c + (e & 1)][2 * rr + (e >> 1)] + half_o;
                const int o = row < len ? clamp127(x >> sh_o) : 0;
                w |= (static_cast<uint32_t>(o) & 0xffu) << (8 * e);
            }
            *reinterpret_cast<uint32_t *>(dst + 16 * c) = w;
        }
    }
}

// ---------------------------------------------------------- producer parts --

// Dot product of one staged 128-byte row (128-byte swizzle) with a vector
// held as 32 packed words: the bias K u of a key or P v of a band row.
__device__ __forceinline__ void bias_row(uint32_t tile, uint32_t dst, const uint32_t (&w)[32],
                                         int row) {
    int acc = 0;
#pragma unroll
    for (int ch = 0; ch < 8; ++ch) {
        const uint4 x = lds128(tile + swz(row, ch));
        acc = __dp4a(static_cast<int>(x.x), static_cast<int>(w[4 * ch + 0]), acc);
        acc = __dp4a(static_cast<int>(x.y), static_cast<int>(w[4 * ch + 1]), acc);
        acc = __dp4a(static_cast<int>(x.z), static_cast<int>(w[4 * ch + 2]), acc);
        acc = __dp4a(static_cast<int>(x.w), static_cast<int>(w[4 * ch + 3]), acc);
    }
    sts32(dst + row * 4, static_cast<uint32_t>(acc));
}

// The bias warp's work on a staged score-pass chunk: K u of the 64 keys
// (rows l, l + 32) and P v of the 128 band rows (l, l + 32, l + 64, l + 96).
__device__ __forceinline__ void prep_bias(uint32_t ktile, uint32_t ptile, uint32_t ku, uint32_t pv,
                                          const uint32_t (&uw)[32], const uint32_t (&vw)[32],
                                          int lane) {
    bias_row(ktile, ku, uw, lane);
    bias_row(ktile, ku, uw, lane + 32);
#pragma unroll
    for (int r = 0; r < 4; ++r) bias_row(ptile, pv, vw, lane + 32 * r);
}

// ------------------------------------------------------------- work items --

// One work item: a whole 64-row tile of (b, h) (part < 0, nparts 1) or part
// `part` of nparts (2: 32-row halves, 4: 16-row quarters) of one.  Items are decoded without a division instruction (exact
// multiply-high by the constants of ntiles and H).
struct Item {
    int b, h, bh, i0, part, nparts, plog2, len, nchunks;
    bool pad;   // every row of the tile (half) is padding
};

__device__ __forceinline__ Item decode_item(const FusedParams &p, uint32_t item) {
    Item it;
    uint32_t lin = item;
    it.part = -1;
    it.nparts = 1;
    it.plog2 = 0;
    if (item >= p.nwhole) {
        const uint32_t t = item - p.nwhole;
        lin = p.nwhole + (t >> p.split_log2);
        it.part = static_cast<int>(t & ((1u << p.split_log2) - 1u));
        it.nparts = 1 << p.split_log2;
        it.plog2 = p.split_log2;
    }
    const uint32_t bh = udiv_magic(lin, p.tiles_magic);
    const int tile = static_cast<int>(lin - bh * static_cast<uint32_t>(p.ntiles));
    it.b = static_cast<int>(udiv_magic(bh, p.heads_magic));
    it.h = static_cast<int>(bh) - it.b * p.H;
    it.bh = static_cast<int>(bh);
    it.i0 = tile * MROWS;
    int len = p.T;
    if (p.lengths != nullptr) {
        len = p.lengths[it.b];
        len = len < 0 ? 0 : (len > p.T ? p.T : len);
    }
    it.len = len;
    it.nchunks = (len + NK - 1) / NK;
    it.pad = (it.part < 0 ? it.i0 : it.i0 + (MROWS >> it.plog2) * it.part) >= len;
    return it;
}

// Q fragments (A operand) of 16-row strip `strip` of the staged Q tile for
// the four 32-wide k steps (ldmatrix: matrices rows 0-7 / 8-15 x the two
// 16-byte halves of k step ks, the m16n8k32 A layout); rows >= T were
// filled with zeros by the copy.
__device__ __forceinline__ void load_q(uint32_t qtile, int strip, int lane, uint32_t (&qa)[4][4]) {
    const int m = lane >> 3;
    const int row = strip * 16 + ((m & 1) << 3) + (lane & 7);
#pragma unroll
    for (int ks = 0; ks < 4; ++ks)
        ldsm_x4(qtile + swz(row, 2 * ks + (m >> 1)), qa[ks][0], qa[ks][1], qa[ks][2], qa[ks][3]);
}

// Shared-memory stage ring: use u of the ring (all items of a CTA in order;
// an item takes nchunks score-pass uses, then nchunks attn.V uses) sits in
// stage u & 1 with barrier phase (u >> 1) & 1.  TMA lands (full), the bias
// warp prepares a score-pass chunk or passes an attn.V chunk on (ready),
// the consumers release it (empty), and the stage is refilled with use
// u + 2.  Every barrier completes one phase per use of its stage and every
// waiter waits on each phase in order, so a parity names one phase.
struct Ring {
    uint32_t stage_base, bar_base;   // the Q tile follows the stages
    __device__ __forceinline__ uint32_t stage(int u) const { return stage_base + (u & 1) * STAGE_BYTES; }
    __device__ __forceinline__ uint32_t full(int u) const { return bar_base + 8u * (u & 1); }
    __device__ __forceinline__ uint32_t ready(int u) const { return bar_base + 8u * (NSTAGE + (u & 1)); }
    __device__ __forceinline__ uint32_t empty(int u) const { return bar_base + 8u * (2 * NSTAGE + (u & 1)); }
    __device__ __forceinline__ static uint32_t parity(int u) { return (static_cast<uint32_t>(u) >> 1) & 1u; }
    // The Q tile of live item k: landed (qfull phase k), read by all
    // consumer warps (qempty phase k); refilled with item k + 1 after that.
    __device__ __forceinline__ uint32_t qtile() const { return stage_base + NSTAGE * STAGE_BYTES; }
    __device__ __forceinline__ uint32_t qfull() const { return bar_base + 8u * (3 * NSTAGE + 3); }
    __device__ __forceinline__ uint32_t qempty() const { return bar_base + 8u * (3 * NSTAGE + 4); }
    // Item number of the CTA's live item k (written by the copy warp before
    // it arrives on that item's barriers), or NO_ITEM after the last.
    __device__ __forceinline__ uint32_t slot(int k) const { return bar_base + 96u + 4u * (k & 3); }
    // The four consumer warps of a quarter item exchange maxima, sums and
    // partial sums (one phase per exchange step).
    __device__ __forceinline__ uint32_t quad() const { return bar_base + 120u; }
};

// ------------------------------------------------------ consumer: whole tile --
// Passes 1-3 and the output of one whole 64-row tile by one consumer warp
// (its 16-row strip), with ring uses u0 .. u0 + 2 nchunks - 1; the item's
// Q tile has landed.  Returns false after a barrier wait ran out.
template <bool GS>
__device__ __forceinline__ bool consume_whole(const FusedParams &prm, const Item &it, int u0,
                                              const Ring &R, uint32_t remap, const ScoreBuf &scores,
                                              uint32_t lut, int warp, int lane) {
    const int T = prm.T, len = it.len, nchunks = it.nchunks;
    const int g = lane >> 2, t4 = lane & 3;
    const int wrow0 = it.i0 + warp * 16;
    const long long m_c = prm.m_c, m_p = prm.m_p;
    const long long half_s = 1ll << (prm.sh_s - 1);
    const int s_s = prm.sh_s - 31;
    const int band_row0 = 48 - 16 * warp;      // this warp's first row in the staged band
    int mx0 = -128, mx1 = -128;                // running maxima of rows g and g + 8
    uint32_t qa[4][4];
    load_q(R.qtile(), warp, lane, qa);

    // ---- pass 1: scores.  A warp that issues an integer MMA waits until the
    // tensor pipe accepts it, so the band MMAs of chunk c+1 are issued in
    // groups with the epilogue of chunk c between them: the epilogue runs
    // while the pipe works through the band.
    int bacc[BAND_TILES][4];
    if (!warp_wait(R.ready(u0), Ring::parity(u0), prm.timeout_cycles)) {
        if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
        return false;
    }
    band_mma(bacc, qa, R.stage(u0) + K_TILE_BYTES + band_row0 * 128,
             R.stage(u0) + PV_OFF + band_row0 * 4, lane);
    const int lm_row = lane & 7, lm_mat = lane >> 3;
    uint32_t packed[8];   // int8 scores of the previous chunk, stored late
    for (int c = 0; c < nchunks; ++c) {
        const int u = u0 + c;
        // The content MMAs go first: they do not need the band, whose last
        // MMAs are still in the pipe, nor the previous chunk's scores, whose
        // stores would otherwise hold back their loads.
        int cacc[8][4];
        content_mma(cacc, qa, R.stage(u), R.stage(u) + KU_OFF, lane);
        if (c > 0) {
            const uint32_t oprev = (c - 1) * CHUNK_SCORE_BYTES;
            sc_st128<GS>(scores, oprev + lane * 16, packed[0], packed[1], packed[2], packed[3]);
            sc_st128<GS>(scores, oprev + 512 + lane * 16, packed[4], packed[5], packed[6],
                         packed[7]);
        }
        __syncwarp();
#pragma unroll
        for (int nt = 0; nt < BAND_TILES; ++nt) {
            sts64(remap + (g * REMAP_STRIDE + nt * 8 + 2 * t4) * 4, bacc[nt][0], bacc[nt][1]);
            sts64(remap + ((g + 8) * REMAP_STRIDE + nt * 8 + 2 * t4) * 4, bacc[nt][2], bacc[nt][3]);
        }
        release_stage(R.empty(u), lane);
        const uint32_t sdst = c * CHUNK_SCORE_BYTES;
        if (c + 1 < nchunks) {
            if (!warp_wait(R.ready(u + 1), Ring::parity(u + 1), prm.timeout_cycles)) {
                if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
                return false;
            }
            const uint32_t ptile = R.stage(u + 1) + K_TILE_BYTES + band_row0 * 128;
            const uint32_t pvs = R.stage(u + 1) + PV_OFF + band_row0 * 4;
            // The band of chunk c + 1 starts NK positions after that of chunk
            // c: its first CARRY_TILES tiles are the last ones of chunk c
            // (the same rows of Q against the same rows of P), kept in
            // registers; only the other NK columns are new MMAs.
#pragma unroll
            for (int nt = 0; nt < CARRY_TILES; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) bacc[nt][e] = bacc[NK / 8 + nt][e];
#pragma unroll
            for (int nt = CARRY_TILES; nt < BAND_TILES; ++nt) {
                const int2 v = lds64(pvs + (nt * 8 + 2 * t4) * 4);
                bacc[nt][0] = v.x;
                bacc[nt][1] = v.y;
                bacc[nt][2] = v.x;
                bacc[nt][3] = v.y;
            }
            __syncwarp();
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                const int kh = m >> 1, t0 = CARRY_TILES + (m & 1) * 4;
                uint32_t b[4][4];
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    ldsm_x4(ptile + swz((t0 + i) * 8 + lm_row, kh * 4 + lm_mat), b[i][0], b[i][1],
                            b[i][2], b[i][3]);
#pragma unroll
                for (int i = 0; i < 4; ++i) mma_s8s8(bacc[t0 + i], qa[2 * kh], b[i][0], b[i][1]);
                packed[2 * m] = score_tile<false>(cacc[2 * m], 2 * m, remap, lane, m_c, m_p, half_s,
                                                  s_s, NK, mx0, mx1);
#pragma unroll
                for (int i = 0; i < 4; ++i) mma_s8s8(bacc[t0 + i], qa[2 * kh + 1], b[i][2], b[i][3]);
                packed[2 * m + 1] = score_tile<false>(cacc[2 * m + 1], 2 * m + 1, remap, lane, m_c,
                                                      m_p, half_s, s_s, NK, mx0, mx1);
            }
        } else {
            __syncwarp();
            const int kvalid = len - c * NK;
            if (kvalid < NK)
                score_epilogue<true, GS>(cacc, remap, scores, sdst, lane, m_c, m_p, half_s, s_s,
                                         kvalid, mx0, mx1);
            else
                score_epilogue<false, GS>(cacc, remap, scores, sdst, lane, m_c, m_p, half_s, s_s,
                                          kvalid, mx0, mx1);
        }
    }

    release_stage(R.qempty(), lane);   // done with the Q tile

    // ---- row maxima across the quad
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));

    // ---- pass 2: sums of the integer exponentials
    const uint32_t lut_g = lut + 4 * (g & (LUT_COPIES - 1));
    const uint32_t mx4h = max4h(mx0, mx1);
    unsigned long long sum0 = 0, sum1 = 0;
    if constexpr (GS) {
        // scores from L2: each chunk's two words are requested one chunk ahead
        uint4 nx0 = sc_ld128<GS>(scores, lane * 16), nx1 = sc_ld128<GS>(scores, 512 + lane * 16);
        for (int c = 0; c < nchunks; ++c) {
            const int kvalid = len - c * NK;
            const uint4 sv0 = nx0, sv1 = nx1;
            if (c + 1 < nchunks) {
                nx0 = sc_ld128<GS>(scores, (c + 1) * CHUNK_SCORE_BYTES + lane * 16);
                nx1 = sc_ld128<GS>(scores, (c + 1) * CHUNK_SCORE_BYTES + 512 + lane * 16);
            }
            if (kvalid < NK) {
                exp_sums<true>(sv0, lut_g, mx4h, t4, 0, kvalid, sum0, sum1);
                exp_sums<true>(sv1, lut_g, mx4h, t4, 32, kvalid, sum0, sum1);
            } else {
                exp_sums<false>(sv0, lut_g, mx4h, t4, 0, kvalid, sum0, sum1);
                exp_sums<false>(sv1, lut_g, mx4h, t4, 32, kvalid, sum0, sum1);
            }
        }
    } else if (prm.sum32) {
        uint32_t a[4] = {0u, 0u, 0u, 0u};
        for (int c = 0; c < nchunks; ++c) {
            const int kvalid = len - c * NK;
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
                const uint4 sv = sc_ld128<GS>(scores, c * CHUNK_SCORE_BYTES + hf * 512 + lane * 16);
                if (kvalid < NK)
                    exp_sums32<true>(sv, lut_g, mx4h, t4, 32 * hf, kvalid, a);
                else
                    exp_sums32<false>(sv, lut_g, mx4h, t4, 32 * hf, kvalid, a);
            }
        }
        sum0 = static_cast<unsigned long long>(a[0]) + a[1];
        sum1 = static_cast<unsigned long long>(a[2]) + a[3];
    } else {
        for (int c = 0; c < nchunks; ++c) {
            const int kvalid = len - c * NK;
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
                const uint4 sv = sc_ld128<GS>(scores, c * CHUNK_SCORE_BYTES + hf * 512 + lane * 16);
                if (kvalid < NK)
                    exp_sums<true>(sv, lut_g, mx4h, t4, 32 * hf, kvalid, sum0, sum1);
                else
                    exp_sums<false>(sv, lut_g, mx4h, t4, 32 * hf, kvalid, sum0, sum1);
            }
        }
    }
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 1);
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 2);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 1);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 2);
    const uint32_t f0 = div_2pow32(sum0);
    const uint32_t f1 = div_2pow32(sum1);

    // ---- pass 3: probabilities x V.  The A operand of the next 32-key step
    // is computed between the MMA groups of the current one.
    int oacc[16][4];
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) oacc[nt][0] = oacc[nt][1] = oacc[nt][2] = oacc[nt][3] = 0;
    auto pass3 = [&](auto f24_tag, uint32_t fa, uint32_t fb) -> bool {
        constexpr bool F24 = decltype(f24_tag)::value;
        const int nsteps = 2 * nchunks;
        uint32_t af[4];
        const int kvalid_last = len - (nchunks - 1) * NK;   // valid keys of the last chunk
        {
            const uint4 sv = sc_ld128<GS>(scores, lane * 16);
            uint32_t pw[4] = {prob_word<F24>(sv.x, lut_g, mx4h, fa, fb),
                              prob_word<F24>(sv.y, lut_g, mx4h, fa, fb),
                              prob_word<F24>(sv.z, lut_g, mx4h, fa, fb),
                              prob_word<F24>(sv.w, lut_g, mx4h, fa, fb)};
            if (nchunks == 1 && kvalid_last < NK) {
#pragma unroll
                for (int q = 0; q < 4; ++q) pw[q] &= key_mask(0, q, t4, kvalid_last);
            }
            prob_operand(pw, af);
        }
        for (int c = 0; c < nchunks; ++c) {
            const int u = u0 + nchunks + c;
            if (!warp_wait(R.ready(u), Ring::parity(u), prm.timeout_cycles)) {
                if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
                return false;
            }
            const uint32_t vtile = R.stage(u);
#pragma unroll
            for (int ks = 0; ks < 2; ++ks) {
                const int nxt = min(2 * c + ks + 1, nsteps - 1);
                const uint4 svn = sc_ld128<GS>(
                    scores, (nxt >> 1) * CHUNK_SCORE_BYTES + (nxt & 1) * 512 + lane * 16);
                const uint32_t wn[4] = {svn.x, svn.y, svn.z, svn.w};
                uint32_t pw[4];
#pragma unroll
                for (int grp = 0; grp < 4; ++grp) {
                    uint32_t b[2][4];
#pragma unroll
                    for (int i = 0; i < 2; ++i)   // d chunk 2 grp + i: n-tiles 4 grp + 2 i, + 1
                        vfrag(vtile, ks, 2 * grp + i, lane, b[i][0], b[i][1], b[i][2], b[i][3]);
#pragma unroll
                    for (int i = 0; i < 2; ++i) {
                        mma_u8s8(oacc[4 * grp + 2 * i], af, b[i][0], b[i][1]);
                        mma_u8s8(oacc[4 * grp + 2 * i + 1], af, b[i][2], b[i][3]);
                    }
                    pw[grp] = prob_word<F24>(wn[grp], lut_g, mx4h, fa, fb);
                }
                if ((nxt >> 1) == nchunks - 1 && kvalid_last < NK) {
                    const int kbase = (nxt & 1) * 32;
#pragma unroll
                    for (int q = 0; q < 4; ++q) pw[q] &= key_mask(kbase, q, t4, kvalid_last);
                }
                prob_operand(pw, af);
            }
            release_stage(R.empty(u), lane);
        }
        return true;
    };
    const bool ok3 = prm.f24 ? pass3(BoolTag<true>(), f0 << 8, f1 << 8)
                             : pass3(BoolTag<false>(), f0, f1);
    if (!ok3) return false;

    // ---- output requantisation (Eq. 7): per d chunk c and row, four bytes
    // d = 16c + 4t .. 16c + 4t + 3 (n-tiles 2c, 2c + 1, columns 2t, 2t + 1).
    // The d chunks go in the order their last MMAs were issued, so the
    // first ones are requantised while the pipe finishes the others.
    const long long m_o = prm.m_o;
    const long long half_o = 1ll << (prm.sh_o - 1);
#pragma unroll
    for (int c = 0; c < 8; ++c) {
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
            const int row = wrow0 + g + 8 * rr;
            uint32_t w = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const long long x = m_o * oacc[2 * c + (e & 1)][2 * rr + (e >> 1)] + half_o;
                const int o = row < len ? clamp127(x >> prm.sh_o) : 0;
                w |= (static_cast<uint32_t>(o) & 0xffu) << (8 * e);
            }
            if (row < T)
                *reinterpret_cast<uint32_t *>(prm.out + out_offset(prm, it.b, it.h, row) + 4 * t4 +
                                              16 * c) = w;
        }
    }
    return true;
}

// -------------------------------------------------------- consumer: half tile --
// One 32-row half of a tile: the two warps of a 16-row strip take the key
// halves [0, 32) and [32, 64) of every chunk and combine row maxima,
// exponential sums and attn.V partial sums through their exchange areas
// behind the strip pair's barrier (four phases per half: maxima, sums,
// partials, and the partner done reading before the areas are reused).
template <bool GS>
__device__ __forceinline__ bool consume_half(const FusedParams &prm, const Item &it, int u0,
                                             const Ring &R, uint32_t remap,
                                             const ScoreBuf &scores, uint32_t lut, uint32_t pair,
                                             int warp, int lane) {
    const int len = it.len, nchunks = it.nchunks;
    const int g = lane >> 2, t4 = lane & 3;
    const int strip = 2 * it.part + (warp >> 1);
    const int wrow0 = it.i0 + strip * 16;
    const long long m_c = prm.m_c, m_p = prm.m_p;
    const long long half_s = 1ll << (prm.sh_s - 1);
    const int s_s = prm.sh_s - 31;
    const int band_row0 = 48 - 16 * strip;
    int mx0 = -128, mx1 = -128;
    const int hk = warp & 1;                   // key half of every chunk
    const int nt0 = 4 * hk;
    const uint32_t xown = remap;
    const uint32_t xpart = hk ? remap - REMAP_BYTES : remap + REMAP_BYTES;   // warp ^ 1
    const uint32_t lut_g = lut + 4 * (g & (LUT_COPIES - 1));
    uint32_t qa[4][4];
    load_q(R.qtile(), strip, lane, qa);

    // pass 1: scores of this warp's key half of every chunk
    for (int c = 0; c < nchunks; ++c) {
        const int u = u0 + c;
        if (!warp_wait(R.ready(u), Ring::parity(u), prm.timeout_cycles)) {
            if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
            return false;
        }
        int hb[6][4], hc[4][4];
        half_chunk_mma(hb, hc, qa, R.stage(u) + K_TILE_BYTES + band_row0 * 128,
                       R.stage(u) + PV_OFF + band_row0 * 4, R.stage(u), R.stage(u) + KU_OFF, nt0,
                       lane);
        release_stage(R.empty(u), lane);
        __syncwarp();   // the remap reads of the previous chunk are done
#pragma unroll
        for (int i = 0; i < 6; ++i) {
            sts64(remap + (g * REMAP_STRIDE + (nt0 + i) * 8 + 2 * t4) * 4, hb[i][0], hb[i][1]);
            sts64(remap + ((g + 8) * REMAP_STRIDE + (nt0 + i) * 8 + 2 * t4) * 4, hb[i][2],
                  hb[i][3]);
        }
        __syncwarp();
        const int kvalid = len - c * NK;
        uint32_t pk[4];
        if (kvalid < NK) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                pk[i] = score_tile<true>(hc[i], nt0 + i, remap, lane, m_c, m_p, half_s, s_s,
                                         kvalid, mx0, mx1);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                pk[i] = score_tile<false>(hc[i], nt0 + i, remap, lane, m_c, m_p, half_s, s_s,
                                          kvalid, mx0, mx1);
        }
        sc_st128<GS>(scores, c * CHUNK_SCORE_BYTES + hk * 512 + lane * 16, pk[0], pk[1], pk[2],
                     pk[3]);
    }
    release_stage(R.qempty(), lane);   // done with the Q tile
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    __syncwarp();   // the remap reads of the last chunk are done
    sts64(xown + XMAX_OFF + lane * 8, mx0, mx1);
    __syncwarp();
    if (lane == 0) mbar_arrive(pair);
    if (!warp_wait(pair, 0, prm.timeout_cycles)) {
        if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
        return false;
    }
    {
        const int2 pm = lds64(xpart + XMAX_OFF + lane * 8);
        mx0 = max(mx0, pm.x);
        mx1 = max(mx1, pm.y);
    }

    // pass 2: exponential sums of the key half, then of the whole row
    const uint32_t mx4h = max4h(mx0, mx1);
    unsigned long long sum0 = 0, sum1 = 0;
    for (int c = 0; c < nchunks; ++c) {
        const int kvalid = len - c * NK;
        const uint4 sv = sc_ld128<GS>(scores, c * CHUNK_SCORE_BYTES + hk * 512 + lane * 16);
        if (kvalid < NK)
            exp_sums<true>(sv, lut_g, mx4h, t4, 32 * hk, kvalid, sum0, sum1);
        else
            exp_sums<false>(sv, lut_g, mx4h, t4, 32 * hk, kvalid, sum0, sum1);
    }
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 1);
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 2);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 1);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 2);
    sts64(xown + XSUM_OFF + lane * 16, static_cast<int>(sum0), static_cast<int>(sum0 >> 32));
    sts64(xown + XSUM_OFF + lane * 16 + 8, static_cast<int>(sum1), static_cast<int>(sum1 >> 32));
    __syncwarp();
    if (lane == 0) mbar_arrive(pair);
    if (!warp_wait(pair, 1, prm.timeout_cycles)) {
        if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
        return false;
    }
    {
        const int2 a = lds64(xpart + XSUM_OFF + lane * 16);
        const int2 bq = lds64(xpart + XSUM_OFF + lane * 16 + 8);
        sum0 += (static_cast<unsigned long long>(static_cast<uint32_t>(a.y)) << 32) |
                static_cast<uint32_t>(a.x);
        sum1 += (static_cast<unsigned long long>(static_cast<uint32_t>(bq.y)) << 32) |
                static_cast<uint32_t>(bq.x);
    }
    const uint32_t f0 = div_2pow32(sum0);
    const uint32_t f1 = div_2pow32(sum1);

    // pass 3: probabilities of the key half x V (k step hk of every chunk)
    int oacc[16][4];
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) oacc[nt][0] = oacc[nt][1] = oacc[nt][2] = oacc[nt][3] = 0;
    const int kvalid_last = len - (nchunks - 1) * NK;
    for (int c = 0; c < nchunks; ++c) {
        const uint4 sv = sc_ld128<GS>(scores, c * CHUNK_SCORE_BYTES + hk * 512 + lane * 16);
        uint32_t pw[4] = {prob_word<false>(sv.x, lut_g, mx4h, f0, f1),
                          prob_word<false>(sv.y, lut_g, mx4h, f0, f1),
                          prob_word<false>(sv.z, lut_g, mx4h, f0, f1),
                          prob_word<false>(sv.w, lut_g, mx4h, f0, f1)};
        if (c == nchunks - 1 && kvalid_last < NK) {
#pragma unroll
            for (int q = 0; q < 4; ++q) pw[q] &= key_mask(32 * hk, q, t4, kvalid_last);
        }
        uint32_t af[4];
        prob_operand(pw, af);
        const int u = u0 + nchunks + c;
        if (!warp_wait(R.ready(u), Ring::parity(u), prm.timeout_cycles)) {
            if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
            return false;
        }
        const uint32_t vtile = R.stage(u);
#pragma unroll
        for (int grp = 0; grp < 4; ++grp) {
            uint32_t bv[2][4];
#pragma unroll
            for (int i = 0; i < 2; ++i)
                vfrag(vtile, hk, 2 * grp + i, lane, bv[i][0], bv[i][1], bv[i][2], bv[i][3]);
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                mma_u8s8(oacc[4 * grp + 2 * i], af, bv[i][0], bv[i][1]);
                mma_u8s8(oacc[4 * grp + 2 * i + 1], af, bv[i][2], bv[i][3]);
            }
        }
        release_stage(R.empty(u), lane);
    }

    // the partner finishes the other half of the output columns
    if (hk == 0) send_partial<0>(oacc, xown + XO_OFF, lane);
    else send_partial<1>(oacc, xown + XO_OFF, lane);
    __syncwarp();
    if (lane == 0) mbar_arrive(pair);
    if (!warp_wait(pair, 0, prm.timeout_cycles)) {
        if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
        return false;
    }
    const long long m_o = prm.m_o;
    const long long half_o = 1ll << (prm.sh_o - 1);
    if (hk == 0)
        finish_half<0>(oacc, xpart + XO_OFF, lane, wrow0, len, prm, it.b, it.h, m_o, half_o);
    else
        finish_half<1>(oacc, xpart + XO_OFF, lane, wrow0, len, prm, it.b, it.h, m_o, half_o);
    // both warps are done reading the partner's area before either reuses its own
    __syncwarp();
    if (lane == 0) mbar_arrive(pair);
    if (!warp_wait(pair, 1, prm.timeout_cycles)) {
        if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
        return false;
    }
    return true;
}

// ------------------------------------------------------ consumer: quarter tile --
// Band n-tiles nt0 .. nt0 + 3 and content n-tiles nt0, nt0 + 1 of one
// 16-key slice of a chunk (nt0 = 2 w): the band columns of keys 16 w ..
// 16 w + 15 of 16 rows are 16 w .. 16 w + 30.
__device__ __forceinline__ void quarter_chunk_mma(int (&bacc)[4][4], int (&cacc)[2][4],
                                                  const uint32_t (&qa)[4][4], uint32_t ptile,
                                                  uint32_t pv, uint32_t ktile, uint32_t ku,
                                                  int nt0, int lane) {
    const int t4 = lane & 3;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int2 v = lds64(pv + ((nt0 + i) * 8 + 2 * t4) * 4);
        bacc[i][0] = v.x;
        bacc[i][1] = v.y;
        bacc[i][2] = v.x;
        bacc[i][3] = v.y;
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        const int2 v = lds64(ku + ((nt0 + i) * 8 + 2 * t4) * 4);
        cacc[i][0] = v.x;
        cacc[i][1] = v.y;
        cacc[i][2] = v.x;
        cacc[i][3] = v.y;
    }
    const int lm_row = lane & 7, lm_mat = lane >> 3;
#pragma unroll
    for (int kh = 0; kh < 2; ++kh) {
        uint32_t b[4][4], kb[2][4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
            ldsm_x4(ptile + swz((nt0 + i) * 8 + lm_row, kh * 4 + lm_mat), b[i][0], b[i][1],
                    b[i][2], b[i][3]);
#pragma unroll
        for (int i = 0; i < 2; ++i)
            ldsm_x4(ktile + swz((nt0 + i) * 8 + lm_row, kh * 4 + lm_mat), kb[i][0], kb[i][1],
                    kb[i][2], kb[i][3]);
#pragma unroll
        for (int i = 0; i < 4; ++i) mma_s8s8(bacc[i], qa[2 * kh], b[i][0], b[i][1]);
#pragma unroll
        for (int i = 0; i < 2; ++i) mma_s8s8(cacc[i], qa[2 * kh], kb[i][0], kb[i][1]);
#pragma unroll
        for (int i = 0; i < 4; ++i) mma_s8s8(bacc[i], qa[2 * kh + 1], b[i][2], b[i][3]);
#pragma unroll
        for (int i = 0; i < 2; ++i) mma_s8s8(cacc[i], qa[2 * kh + 1], kb[i][2], kb[i][3]);
    }
}

// One 16-row quarter (strip `part`) of a tile, for the tail of the work:
// the four warps share the strip, warp w taking the keys [16 w, 16 w + 16)
// of every chunk, and its attn.V product on those keys as m16n8k16 MMAs
// (k order 2t, 2t + 1, 8 + 2t, 9 + 2t on both operands, as in the 32-key
// steps).  Row maxima, exponential sums and the attn.V partial sums (warp w
// finishes d = 32 w .. 32 w + 31) are combined through the warps' exchange
// areas behind the quad barrier, eight phases per quarter.
template <bool GS>
__device__ __forceinline__ bool consume_quarter(const FusedParams &prm, const Item &it, int u0,
                                                const Ring &R, uint32_t remap, uint32_t remap0,
                                                const ScoreBuf &scores, uint32_t lut, uint32_t quad,
                                                int warp, int lane) {
    const int len = it.len, nchunks = it.nchunks;
    const int g = lane >> 2, t4 = lane & 3;
    const int strip = it.part;
    const int wrow0 = it.i0 + strip * 16;
    const long long m_c = prm.m_c, m_p = prm.m_p;
    const long long half_s = 1ll << (prm.sh_s - 1);
    const int s_s = prm.sh_s - 31;
    const int band_row0 = 48 - 16 * strip;
    const int nt0 = 2 * warp;                  // this warp's key slice: n-tiles nt0, nt0 + 1
    int mx0 = -128, mx1 = -128;
    const uint32_t lut_g = lut + 4 * (g & (LUT_COPIES - 1));
    int qph = 0;   // phases of the quad barrier used in this quarter
    auto quad_sync = [&]() -> bool {
        __syncwarp();
        if (lane == 0) mbar_arrive(quad);
        const bool ok = warp_wait(quad, static_cast<uint32_t>(qph) & 1u, prm.timeout_cycles);
        ++qph;
        if (!ok && lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
        return ok;
    };
    uint32_t qa[4][4];
    load_q(R.qtile(), strip, lane, qa);

    // pass 1: scores of this warp's key slice of every chunk
    for (int c = 0; c < nchunks; ++c) {
        const int u = u0 + c;
        if (!warp_wait(R.ready(u), Ring::parity(u), prm.timeout_cycles)) {
            if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
            return false;
        }
        int qb[4][4], qc[2][4];
        quarter_chunk_mma(qb, qc, qa, R.stage(u) + K_TILE_BYTES + band_row0 * 128,
                          R.stage(u) + PV_OFF + band_row0 * 4, R.stage(u), R.stage(u) + KU_OFF, nt0,
                          lane);
        release_stage(R.empty(u), lane);
        __syncwarp();   // the remap reads of the previous chunk are done
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            sts64(remap + (g * REMAP_STRIDE + i * 8 + 2 * t4) * 4, qb[i][0], qb[i][1]);
            sts64(remap + ((g + 8) * REMAP_STRIDE + i * 8 + 2 * t4) * 4, qb[i][2], qb[i][3]);
        }
        __syncwarp();
        // band columns stored from the slice's first one: key jj of the slice
        // and row rho take the band value at jj - rho + 15, as in a chunk
        const int kvalid = len - c * NK - 16 * warp;   // valid keys of the slice
        uint32_t pk[2];
        if (kvalid < 16) {
#pragma unroll
            for (int i = 0; i < 2; ++i)
                pk[i] = score_tile<true>(qc[i], i, remap, lane, m_c, m_p, half_s, s_s, kvalid,
                                         mx0, mx1);
        } else {
#pragma unroll
            for (int i = 0; i < 2; ++i)
                pk[i] = score_tile<false>(qc[i], i, remap, lane, m_c, m_p, half_s, s_s, kvalid,
                                          mx0, mx1);
        }
        sc_st64<GS>(scores, c * CHUNK_SCORE_BYTES + lane * 8, static_cast<int>(pk[0]),
              static_cast<int>(pk[1]));
    }
    release_stage(R.qempty(), lane);   // done with the Q tile
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    __syncwarp();   // the remap reads of the last chunk are done
    sts64(remap + XMAX_OFF + lane * 8, mx0, mx1);
    if (!quad_sync()) return false;
#pragma unroll
    for (int w = 0; w < NCWARPS; ++w) {
        const int2 pm = lds64(remap0 + w * REMAP_BYTES + XMAX_OFF + lane * 8);
        mx0 = max(mx0, pm.x);
        mx1 = max(mx1, pm.y);
    }
    const uint32_t mx4h = max4h(mx0, mx1);

    // pass 2: exponential sums of the slice, then of the whole row
    unsigned long long sum0 = 0, sum1 = 0;
    for (int c = 0; c < nchunks; ++c) {
        const int kvalid = len - c * NK - 16 * warp;
        const int2 wv = sc_ld64<GS>(scores, c * CHUNK_SCORE_BYTES + lane * 8);
        const uint32_t w2[2] = {static_cast<uint32_t>(wv.x), static_cast<uint32_t>(wv.y)};
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const uint32_t d4 = exp_index4(w2[q], mx4h);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                uint32_t ev = lds32(lut_at(lut_g, d4, e));
                if (q * 8 + 2 * t4 + (e & 1) >= kvalid) ev = 0u;
                if (e < 2) sum0 += ev;
                else sum1 += ev;
            }
        }
    }
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 1);
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 2);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 1);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 2);
    sts64(remap + XSUM_OFF + lane * 16, static_cast<int>(sum0), static_cast<int>(sum0 >> 32));
    sts64(remap + XSUM_OFF + lane * 16 + 8, static_cast<int>(sum1), static_cast<int>(sum1 >> 32));
    if (!quad_sync()) return false;
    sum0 = 0;
    sum1 = 0;
#pragma unroll
    for (int w = 0; w < NCWARPS; ++w) {
        const int2 a = lds64(remap0 + w * REMAP_BYTES + XSUM_OFF + lane * 16);
        const int2 bq = lds64(remap0 + w * REMAP_BYTES + XSUM_OFF + lane * 16 + 8);
        sum0 += (static_cast<unsigned long long>(static_cast<uint32_t>(a.y)) << 32) |
                static_cast<uint32_t>(a.x);
        sum1 += (static_cast<unsigned long long>(static_cast<uint32_t>(bq.y)) << 32) |
                static_cast<uint32_t>(bq.x);
    }
    const uint32_t f0 = div_2pow32(sum0);
    const uint32_t f1 = div_2pow32(sum1);

    // pass 3: probabilities of the slice x V (m16n8k16, k = the slice's keys)
    int oacc[16][4];
#pragma unroll
    for (int nt = 0; nt < 16; ++nt) oacc[nt][0] = oacc[nt][1] = oacc[nt][2] = oacc[nt][3] = 0;
    const int vkey = 16 * warp + 8 * ((lane >> 3) & 1) + (lane & 7);
    for (int c = 0; c < nchunks; ++c) {
        const int kvalid = len - c * NK - 16 * warp;
        const int2 wv = sc_ld64<GS>(scores, c * CHUNK_SCORE_BYTES + lane * 8);
        uint32_t pw0 = prob_word<false>(static_cast<uint32_t>(wv.x), lut_g, mx4h, f0, f1);
        uint32_t pw1 = prob_word<false>(static_cast<uint32_t>(wv.y), lut_g, mx4h, f0, f1);
        if (kvalid < 16) {
            pw0 &= key_mask(0, 0, t4, kvalid);
            pw1 &= key_mask(0, 1, t4, kvalid);
        }
        // A: row g, then g + 8, keys 2t, 2t + 1, 8 + 2t, 9 + 2t of the slice
        const uint32_t a0 = __byte_perm(pw0, pw1, 0x5410);
        const uint32_t a1 = __byte_perm(pw0, pw1, 0x7632);
        const int u = u0 + nchunks + c;
        if (!warp_wait(R.ready(u), Ring::parity(u), prm.timeout_cycles)) {
            if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_READY);
            return false;
        }
        const uint32_t vtile = R.stage(u);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            // d chunks 2j, 2j + 1: the slice's keys 0-7 and 8-15 of each
            uint32_t r0, r1, r2, r3;
            ldsm_x4_trans(vtile + swz(vkey, 2 * j + (lane >> 4)), r0, r1, r2, r3);
            mma_u8s8_k16(oacc[4 * j], a0, a1, __byte_perm(r0, r1, 0x6420));
            mma_u8s8_k16(oacc[4 * j + 1], a0, a1, __byte_perm(r0, r1, 0x7531));
            mma_u8s8_k16(oacc[4 * j + 2], a0, a1, __byte_perm(r2, r3, 0x6420));
            mma_u8s8_k16(oacc[4 * j + 3], a0, a1, __byte_perm(r2, r3, 0x7531));
        }
        release_stage(R.empty(u), lane);
    }

    // the partial sums: in round r each warp sends the n-tiles of warp
    // (w + r) mod 4 and adds those warp (w - r) mod 4 sent it
    const uint32_t xo = remap + XO_OFF;
#pragma unroll 1
    for (int r = 1; r < NCWARPS; ++r) {
        const int dst = (warp + r) & (NCWARPS - 1);
        const int src = (warp - r) & (NCWARPS - 1);
#pragma unroll
        for (int w = 0; w < NCWARPS; ++w)
            if (w == dst) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        sts32(xo + ((i * 4 + e) * 32 + lane) * 4, static_cast<uint32_t>(oacc[4 * w + i][e]));
            }
        if (!quad_sync()) return false;
        const uint32_t xs = remap0 + src * REMAP_BYTES + XO_OFF;
#pragma unroll
        for (int w = 0; w < NCWARPS; ++w)
            if (w == warp) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        oacc[4 * w + i][e] += static_cast<int>(lds32(xs + ((i * 4 + e) * 32 + lane) * 4));
            }
        if (!quad_sync()) return false;
    }

    // Eq. 7 and the stores of d chunks 2w, 2w + 1 (n-tiles 4w .. 4w + 3)
    const long long m_o = prm.m_o;
    const long long half_o = 1ll << (prm.sh_o - 1);
    const int T = prm.T;
#pragma unroll
    for (int cc = 0; cc < 8; ++cc) {
        if ((cc >> 1) != warp) continue;
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
            const int row = wrow0 + g + 8 * rr;
            if (row >= T) continue;
            uint32_t w = 0;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const long long x = m_o * oacc[2 * cc + (e & 1)][2 * rr + (e >> 1)] + half_o;
                const int o = row < len ? clamp127(x >> prm.sh_o) : 0;
                w |= (static_cast<uint32_t>(o) & 0xffu) << (8 * e);
            }
            *reinterpret_cast<uint32_t *>(prm.out + out_offset(prm, it.b, it.h, row) + 4 * t4 +
                                          16 * cc) = w;
        }
    }
    return true;
}

// ------------------------------------------------------------ fused kernel --
// Persistent: one CTA per resident slot.  The copy warp claims the items in
// order from a counter in the workspace, so the last items (the halves of
// the tail) go to the CTAs that finish first; it writes the zeros of
// padding items itself and publishes each live item to the other warps
// through a shared-memory slot.  The stage ring runs on across items, so
// the copies and bias vectors of the next item's first chunks overlap the
// end of the current one.

// Zero output rows of a padding item (every row is at or beyond its length).
__device__ __forceinline__ void zero_rows(const FusedParams &p, const Item &it, int lane) {
    const int nrows = MROWS >> it.plog2;
    const int r0 = it.part < 0 ? it.i0 : it.i0 + nrows * it.part;
    const int rows = (p.T - r0) < nrows ? (p.T - r0) : nrows;
    for (int c = lane; c < rows * (DH / 16); c += 32)
        *reinterpret_cast<int4 *>(p.out + out_offset(p, it.b, it.h, r0 + (c >> 3)) + 16 * (c & 7)) =
            make_int4(0, 0, 0, 0);
}

template <bool GS>
__global__ void __launch_bounds__(NTHREADS, 2)
    relpos_mhsa_fused_kernel(const __grid_constant__ CUtensorMap tm_q,
                             const __grid_constant__ CUtensorMap tm_k,
                             const __grid_constant__ CUtensorMap tm_v,
                             const __grid_constant__ CUtensorMap tm_p, const FusedParams prm) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const SmemLayout L = smem_layout(prm.nchunk_max, GS);
    const int T = prm.T;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    const uint32_t lut = smem_u32(smem + L.lut);
    Ring R;
    R.stage_base = smem_u32(smem + L.stages);
    R.bar_base = smem_u32(smem + L.bars);
    const uint32_t never_bar = R.bar_base + 8u * (3 * NSTAGE);   // test hook only
    auto pair_bar = [&](int strip2) { return R.bar_base + 8u * (3 * NSTAGE + 1 + strip2); };

    // Copy of ring use `pos` of item `it` (pos < nchunks: K chunk and the
    // P band of the tile's rows; else V chunk pos - nchunks) into stage s.
    auto issue = [&](const Item &it, int pos, int u) {
        const uint32_t dst = R.stage(u);
        const uint32_t full = R.full(u);
        if (pos < it.nchunks) {
            const int j0 = pos * NK;
            mbar_expect_tx(full, K_TILE_BYTES + P_TILE_BYTES);
            tma_load_3d(dst, &tm_k, 0, j0, it.bh, full);
            tma_load_3d(dst + K_TILE_BYTES, &tm_p, 0, j0 - it.i0 - (MROWS - 1) + T - 1, it.h, full);
        } else {
            const int j0 = (pos - it.nchunks) * NK;
            mbar_expect_tx(full, K_TILE_BYTES);
            tma_load_3d(dst, &tm_v, 0, j0, it.bh, full);
        }
    };

    // Copy warp: the item being issued, its next ring use, and the item
    // claims.  claim() takes items from the counter until a live one (the
    // padding ones get their zeros here); false once the work is gone.
    Item iss{};
    int iss_pos = 0, issued = 0;
    int kq = 0;   // live items published (slots written, Q tiles sent)
    auto claim = [&](uint32_t &item) -> bool {
        for (;;) {
            uint32_t x = 0;
            if (lane == 0) x = atomicAdd(prm.sched, 1u);
            item = __shfl_sync(0xffffffffu, x, 0);
            if (item >= prm.nitems) return false;
            iss = decode_item(prm, item);
            if (!iss.pad) return true;
            zero_rows(prm, iss, lane);
        }
    };
    // Publishes the claimed item as live item kq: its slot, then its Q tile
    // (the arrive on qfull releases the slot write).
    auto publish = [&](uint32_t item) {
        if (lane == 0) {
            sts32(R.slot(kq), item);
            mbar_expect_tx(R.qfull(), Q_TILE_BYTES);
            tma_load_3d(R.qtile(), &tm_q, 0, iss.i0, iss.bh, R.qfull());
        }
        ++kq;
        iss_pos = 0;
    };
    // No more work: the slot of live item kq says so, and the barriers the
    // consumers (qfull) and the bias warp (full of ring use u) wait on next
    // complete without a copy.  The counters are reset by the last CTA.
    auto finish = [&](int u) {
        if (lane == 0) {
            sts32(R.slot(kq), NO_ITEM);
            mbar_arrive(R.qfull());
            mbar_arrive(R.full(u));
        }
    };
    auto done_claiming = [&]() {
        if (lane == 0 && atomicAdd(prm.sched + 16, 1u) == gridDim.x - 1) {
            atomicExch(prm.sched, 0u);
            atomicExch(prm.sched + 16, 0u);
        }
    };

    // A launch that follows this one on its stream may start now: its CTAs
    // take the SM slots this grid frees at its end and wait (below) for its
    // completion before they touch global memory.
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    // The copy warp initialises the barriers, waits for the grid before it
    // on the stream (its outputs and the reset work counters visible),
    // claims its first item and sends its first two uses off at once; the
    // exponential table is built meanwhile.
    bool live0 = false;
    if (warp == NCWARPS) {
        if (lane == 0) {
            for (int s = 0; s < NSTAGE; ++s) {
                mbar_init(R.full(s), 1);
                mbar_init(R.ready(s), 1);
                mbar_init(R.empty(s), NCWARPS);
            }
            mbar_init(never_bar, 1);
            mbar_init(pair_bar(0), 2);
            mbar_init(pair_bar(1), 2);
            mbar_init(R.qfull(), 1);
            mbar_init(R.qempty(), NCWARPS);
            mbar_init(R.quad(), NCWARPS);
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        }
        __syncwarp();
        asm volatile("griddepcontrol.wait;" ::: "memory");
        uint32_t item = 0;
        live0 = claim(item);
        if (live0) {
            publish(item);
            for (int u = 0; u < NSTAGE; ++u) {   // an item has at least two uses
                if (lane == 0) issue(iss, iss_pos, u);
                ++iss_pos;
                ++issued;
            }
        } else {
            finish(0);
            done_claiming();
        }
    }
    for (int d = threadIdx.x; d < LUT_ENTRIES; d += NTHREADS) {
        const uint32_t e = iexp_neg(d, prm.q_ln2, prm.q_b, prm.q_c, prm.ln2_magic);
#pragma unroll
        for (int c = 0; c < LUT_COPIES; ++c) sts32(lut + (d * LUT_COPIES + c) * 4, e);
    }
    asm volatile("griddepcontrol.wait;" ::: "memory");
    __syncthreads();

    // ------------------------------------------------------------ producers
    if (warp == NCWARPS) {
        // copy warp: refills the stage of use u with use u + 2 once every
        // consumer warp has released u
        if (!live0) return;
        int landed = 0;
        bool ok = true;
        for (int u = 0;; ++u) {
            if (!warp_wait(R.empty(u), Ring::parity(u), prm.timeout_cycles)) {
                if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_EMPTY);
                ok = false;
                break;
            }
            landed = u + 1;   // released by the consumers, so it had landed
            if (iss_pos == 2 * iss.nchunks) {
                // the next use starts a new item, whose Q tile replaces the
                // previous one once every consumer warp is done with that
                if (!warp_wait(R.qempty(), static_cast<uint32_t>(kq - 1) & 1u, prm.timeout_cycles)) {
                    if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_EMPTY);
                    ok = false;
                    break;
                }
                uint32_t item = 0;
                if (!claim(item)) {
                    finish(u + 2);
                    break;
                }
                publish(item);
            }
            if (lane == 0) issue(iss, iss_pos, u + 2);
            ++iss_pos;
            issued = u + 3;
        }
        done_claiming();
        if (!ok) {
            // Let the copies already issued land before the CTA exits
            // (bounded by a fixed budget independent of the caller's).
            for (int u = landed; u < issued; ++u)
                mbar_wait(R.full(u), Ring::parity(u), DRAIN_CYCLES);
            mbar_wait(R.qfull(), static_cast<uint32_t>(kq - 1) & 1u, DRAIN_CYCLES);
        }
        return;
    }
    if (warp == NCWARPS + 1) {
        // bias warp: K u and P v of every staged score-pass chunk, off the
        // consumers' path (a chunk lands one use ahead of its consumers).
        // Every use is acknowledged on `ready` (an attn.V use with no work),
        // so that each barrier's phases follow the ring uses.
        uint32_t uw[32], vw[32];
        int cur_h = -1;
        int u = 0;
        for (int kb = 0;; ++kb) {
            if (!warp_wait(R.full(u), Ring::parity(u), prm.timeout_cycles)) {
                if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_FULL);
                return;
            }
            const uint32_t item = lds32(R.slot(kb));
            if (item == NO_ITEM) return;
            const Item it = decode_item(prm, item);
            if (it.h != cur_h) {
                cur_h = it.h;
                const uint4 *u4 = reinterpret_cast<const uint4 *>(prm.u + static_cast<size_t>(cur_h) * DH);
                const uint4 *v4 = reinterpret_cast<const uint4 *>(prm.vb + static_cast<size_t>(cur_h) * DH);
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    const uint4 a = __ldg(u4 + c), bq = __ldg(v4 + c);
                    uw[4 * c] = a.x; uw[4 * c + 1] = a.y; uw[4 * c + 2] = a.z; uw[4 * c + 3] = a.w;
                    vw[4 * c] = bq.x; vw[4 * c + 1] = bq.y; vw[4 * c + 2] = bq.z; vw[4 * c + 3] = bq.w;
                }
            }
            for (int pos = 0; pos < 2 * it.nchunks; ++pos, ++u) {
                if (pos > 0 && !warp_wait(R.full(u), Ring::parity(u), prm.timeout_cycles)) {
                    if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_FULL);
                    return;
                }
                if (pos < it.nchunks)
                    prep_bias(R.stage(u), R.stage(u) + K_TILE_BYTES, R.stage(u) + KU_OFF,
                              R.stage(u) + PV_OFF, uw, vw, lane);
                release_stage(R.ready(u), lane);
            }
        }
    }

    // ------------------------------------------------------------ consumers
    const uint32_t remap = smem_u32(smem + L.remap) + warp * REMAP_BYTES;
    ScoreBuf scores;
    scores.s = smem_u32(smem + L.scores) + warp * (prm.nchunk_max * CHUNK_SCORE_BYTES);
    scores.g = GS ? prm.gscores + (static_cast<size_t>(blockIdx.x) * NCWARPS + warp) *
                                      static_cast<size_t>(prm.nchunk_max) * CHUNK_SCORE_BYTES
                  : nullptr;
    if (prm.stall_injection && !warp_wait(never_bar, 0, prm.timeout_cycles)) {
        if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_INJECTED);
        return;
    }
    int u0 = 0;
    for (int k = 0;; ++k) {
        if (!warp_wait(R.qfull(), static_cast<uint32_t>(k) & 1u, prm.timeout_cycles)) {
            if (lane == 0) atomicOr(prm.err, ERR_TIMEOUT_FULL);
            return;
        }
        const uint32_t item = lds32(R.slot(k));
        if (item == NO_ITEM) return;
        const Item it = decode_item(prm, item);
        const bool ok =
            it.nparts == 1   ? consume_whole<GS>(prm, it, u0, R, remap, scores, lut, warp, lane)
            : it.nparts == 2 ? consume_half<GS>(prm, it, u0, R, remap, scores, lut, pair_bar(warp >> 1),
                                            warp, lane)
                             : consume_quarter<GS>(prm, it, u0, R, remap, smem_u32(smem + L.remap),
                                               scores, lut, R.quad(), warp, lane);
        if (!ok) return;
        u0 += 2 * it.nchunks;
    }
}

}  // namespace ipk
