// Device code of the integer linear layer (I-Parakeet, Sec. 2.2, Eqs. 6-7)
// for sm_103a: Y = requant(X W^T + bias) with one dyadic multiplier per
// output channel.  Integer arithmetic only: no floating-point type and no
// division by a run-time value.
//
// Persistent kernel: one CTA per SM takes the 128 x 128 tiles of Y (128
// frames x 128 output channels) round-robin.  With a row-major X the frames
// of all utterances form one axis of B T rows; with a head-split X a tile
// stays inside one utterance.  A producer warp streams K in stages of 128
// bytes: the 128 x 128 int8 tiles of X and W land through TMA with the
// 128-byte swizzle in a ring of four stages that runs on across tiles, so
// the next tile's first stages load during the current tile's epilogue.
// The integer MMA pipe and the dp4a pipe of an SM sub-partition work at the
// same time, so a tile's channels are split between them: eight MMA warps
// (2 along the frames x 4 along the channels, 64 x 16 each) take channels
// 0-63 with the integer warp MMA (mma.sync m16n8k32 s8 x s8 -> s32, from
// ldmatrix; sm_103a has no integer tcgen05 kind), and eight dp4a warps
// (16 frames each) take channels 64-127 with dp4a on the same stages.  The
// epilogue adds the int32 bias, multiplies by m[n] in int64, shifts right by
// 31 + s[n] with rounding, clamps to [-127, 127] (and, in the feed-forward
// variant, applies the minimax integer Swish); the MMA warps write their
// 64 x 16 bytes through shared memory as 16-byte row segments, the dp4a
// warps their 8-byte row segments directly, either row-major [B][T][N] or
// head-split [G][B][N/G/128][T][128].
#pragma once

#include <cuda.h>
#include <stdint.h>

#include "ip_ptx.cuh"

namespace ipl {

using namespace ipk;

constexpr int BM = 128;                 // frames per CTA
constexpr int BN = 128;                 // output channels per CTA
constexpr int BK = 128;                 // K bytes per stage
constexpr int NCW = 8;                  // MMA warps: 2 (frames) x 4 (channels)
constexpr int NDW_LOG2 = 3;
constexpr int NDW = 1 << NDW_LOG2;      // dp4a warps, along the frames (two per SM sub-partition)
constexpr int DW_ROWS = BM >> NDW_LOG2; // frames of one dp4a warp
constexpr int RI = DW_ROWS >> 2;        // frames of one dp4a lane (four row groups of lanes)
constexpr int MMA_COLS = 64;            // channels 0 .. 63 of a tile on the MMA pipe, the rest on dp4a
constexpr int DW_UNROLL = 2;     // k chunks of a stage unrolled in the dp4a loop
constexpr int THREADS = (NCW + NDW + 1) * 32;
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * BK;
constexpr int B_BYTES = BN * BK;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int OUT_ROW = 48;             // staged output row of an MMA warp: 16 bytes, stride 48 (3 x 16: rows spread over the bank groups)
constexpr int OUT_WARP_BYTES = 64 * OUT_ROW;
constexpr int SMEM_OUT = STAGES * STAGE_BYTES;
constexpr int SMEM_BARS = SMEM_OUT + NCW * OUT_WARP_BYTES;
constexpr int SMEM_LUT = SMEM_BARS + 8 * (2 * STAGES);     // Swish of every int8 z
constexpr int SMEM_BYTES = SMEM_LUT + 256;
constexpr int SMEM_LAUNCH = SMEM_BYTES + 1024;   // + alignment of the dynamic base

constexpr int LAYOUT_ROWS = 0;
constexpr int LAYOUT_HEADS = 1;
constexpr int ERR_PARAM = 16;           // a multiplier, shift or bias out of its domain

static_assert(STAGE_BYTES % 1024 == 0, "128-byte swizzle needs 1024-byte aligned tiles");
static_assert((STAGES & (STAGES - 1)) == 0, "stage index by mask");

struct LinearParams {
    const int32_t *bias;      // [N] or nullptr
    const int32_t *m;         // [N]
    const int32_t *s;         // [N]
    int8_t *y;
    int B, T, K, N;
    int ntn;                  // N / 128 channel tiles
    int tpu;                  // frame tiles per utterance (head-split X)
    unsigned ntiles;          // all tiles
    unsigned long long magic_ntn, magic_T, magic_tpu;   // exact division constants
    int heads_per_group;      // N / G / 128 (head-split output)
    int y_layout;
    int x_layout;
    int *err;
    long long timeout_cycles;
    // minimax Swish of the requantised output (Eqs. 12-13), SWISH kernels only
    int sw_qc, sw_qone, sw_m, sw_e;
    // residual addition of the output to res (Eqs. 1-4), RES kernels only
    const int8_t *res;        // [B][T][N], row-major like the output
    int res_mx, res_my, res_s;
};

struct Tile {
    int nt;        // channel tile
    int b, t0;     // utterance and frame of the first row
    int m0;        // flat row of the first row (b T + t0)
};

__device__ __forceinline__ Tile tile_of(unsigned idx, const LinearParams &p) {
    Tile L;
    const unsigned mt = udiv_magic(idx, p.magic_ntn);
    L.nt = static_cast<int>(idx - mt * static_cast<unsigned>(p.ntn));
    if (p.x_layout == LAYOUT_ROWS) {
        L.m0 = static_cast<int>(mt) * BM;
        L.b = static_cast<int>(udiv_magic(static_cast<unsigned>(L.m0), p.magic_T));
        L.t0 = L.m0 - L.b * p.T;
    } else {
        L.b = static_cast<int>(udiv_magic(mt, p.magic_tpu));
        L.t0 = (static_cast<int>(mt) - L.b * p.tpu) * BM;
        L.m0 = L.b * p.T + L.t0;
    }
    return L;
}

// Integer Swish of one int8 value z on the grid S_z (Eqs. 12-13): the
// clipped parabola L = q_one - (min(|z|, q_c) - q_c)^2 is |tanh(z S_z / 2)|
// on the grid S_t, t = q_one + sgn(z) L is 1 + tanh, and z t is requantised
// onto the output grid.  |z t| < 2^31 since t <= 2 q_one < 2^24.
__device__ __forceinline__ int swish_i8(int z, const LinearParams &p) {
    const int a = z < 0 ? -z : z;
    const int dc = (a < p.sw_qc ? a : p.sw_qc) - p.sw_qc;
    const int L = p.sw_qone - dc * dc;
    const int t = z > 0 ? p.sw_qone + L : (z < 0 ? p.sw_qone - L : p.sw_qone);
    const long long v = static_cast<long long>(p.sw_m) * (z * t) + (1ll << (p.sw_e - 1));
    return clamp127(v >> p.sw_e);
}

// Gated linear unit of Eq. 5 on two requantised int8 values: a sigma(b)
// with sigma(b) = (1 + tanh(b/2)) / 2 and the minimax tanh on b's grid;
// |a t| < 2^31 (t <= 2 q_one < 2^24).
__device__ __forceinline__ int glu_i8(int a, int b, const LinearParams &p) {
    const int mag = b < 0 ? -b : b;
    const int dc = (mag < p.sw_qc ? mag : p.sw_qc) - p.sw_qc;
    const int L = p.sw_qone - dc * dc;
    const int t = b > 0 ? p.sw_qone + L : (b < 0 ? p.sw_qone - L : p.sw_qone);
    const long long v = static_cast<long long>(p.sw_m) * (a * t) + (1ll << (p.sw_e - 1));
    return clamp127(v >> p.sw_e);
}

constexpr int EPI_PLAIN = 0;   // requantised int8
constexpr int EPI_SWISH = 1;   // + minimax Swish
constexpr int EPI_GLU = 2;     // interleaved pairs (a_c, b_c) -> a_c sigma(b_c)
constexpr int EPI_RES = 3;     // requantised int8, then the residual addition to res

// Offset in Y of tile row r (0 .. BM - 1) at tile column col, or -1 past the
// last frame.  Row-major Y [B][T][N] (or [B][T][N / 2] for the gated unit,
// with `width` its row length) or head-split Y [G][B][N / G / 128][T][128];
// hh, grp: the tile's head within its group and the group.
__device__ __forceinline__ long long y_offset(const LinearParams &p, const Tile &L, int r, int col,
                                              int width, int hh, int grp) {
    int b = L.b, t = L.t0 + r;
    if (p.x_layout == LAYOUT_ROWS) {
        if (L.m0 + r >= p.B * p.T) return -1;
        if (p.y_layout == LAYOUT_ROWS)
            return static_cast<long long>(L.m0 + r) * width + col;
        while (t >= p.T) {   // rows of a flat tile may run into later utterances
            t -= p.T;
            ++b;
        }
    } else if (t >= p.T) {
        return -1;
    }
    if (p.y_layout == LAYOUT_ROWS) return (static_cast<long long>(b) * p.T + t) * width + col;
    return (((static_cast<long long>(grp) * p.B + b) * p.heads_per_group + hh) * p.T + t) * 128 + col;
}

// Per-channel constants of Eq. 7 for channel n, clipped into their domain
// (bad is set when one was out of it).
__device__ __forceinline__ void channel_consts(const LinearParams &p, int n, int &cb, int &cm,
                                               int &ce, bool &bad) {
    int bi = p.bias != nullptr ? __ldg(p.bias + n) : 0;
    int mi = __ldg(p.m + n);
    int si = __ldg(p.s + n);
    if (mi < 0 || si < 0 || si > 31 || bi >= (1 << 30) || bi <= -(1 << 30)) {
        bad = true;
        mi = mi < 0 ? 0 : mi;
        si = si < 0 ? 0 : (si > 31 ? 31 : si);
        bi = 0;
    }
    cb = bi;
    cm = mi;
    ce = 31 + si;
}

// Eq. 7 for one accumulator: clamp(round(m (acc + bias) / 2^(31 + s))).
__device__ __forceinline__ int requant(int acc, int cb, int cm, int ce) {
    const long long v = static_cast<long long>(cm) * (acc + cb) + (1ll << (ce - 1));
    return clamp127(v >> ce);
}

template <int EPI>
__global__ void __launch_bounds__(THREADS, 1)
    linear_i8_kernel(const __grid_constant__ CUtensorMap tm_x,
                     const __grid_constant__ CUtensorMap tm_w, const LinearParams prm) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int kt = prm.K / BK;     // BK is a power of two: a shift

    const uint32_t base = smem_u32(smem);
    const uint32_t bars = base + SMEM_BARS;
    auto full_bar = [&](int s) { return bars + 8u * s; };
    auto empty_bar = [&](int s) { return bars + 8u * (STAGES + s); };
    auto stage = [&](int s) { return base + s * STAGE_BYTES; };

    const uint32_t lut = base + SMEM_LUT;
    const uint8_t *swish_lut = smem + SMEM_LUT;
    pdl_launch_dependents();
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), NCW + NDW);
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (EPI == EPI_SWISH && threadIdx.x < 256) {
        // the Swish of every int8 input, entry at the byte value of z
        const int z = static_cast<int>(static_cast<int8_t>(static_cast<uint8_t>(threadIdx.x)));
        const uint32_t y = static_cast<uint32_t>(swish_i8(z, prm)) & 0xffu;
        asm volatile("st.shared.u8 [%0], %1;" ::"r"(lut + threadIdx.x), "r"(y) : "memory");
    }
    pdl_wait();   // the grid before this one on the stream: complete, memory visible
    __syncthreads();

    // ---------------------------------------------------------- producer
    // Use u of the ring: stage u & 3, phase (u / 4) & 1.
    if (warp == NCW + NDW) {
        unsigned u = 0, landed_from = 0;
        bool ok = true;
        for (unsigned idx = blockIdx.x; idx < prm.ntiles && ok; idx += gridDim.x) {
            const Tile L = tile_of(idx, prm);
            for (int it = 0; it < kt; ++it, ++u) {
                const int s = static_cast<int>(u & (STAGES - 1));
                if (u >= STAGES &&
                    !warp_wait(empty_bar(s), ((u / STAGES) - 1) & 1, prm.timeout_cycles)) {
                    if (lane == 0) atomicOr(prm.err, 2);
                    ok = false;
                    break;
                }
                if (lane == 0) {
                    mbar_expect_tx(full_bar(s), STAGE_BYTES);
                    if (prm.x_layout == LAYOUT_ROWS)
                        tma_load_2d(stage(s), &tm_x, it * BK, L.m0, full_bar(s));
                    else
                        tma_load_4d(stage(s), &tm_x, 0, L.t0, it, L.b, full_bar(s));
                    tma_load_2d(stage(s) + A_BYTES, &tm_w, it * BK, L.nt * BN, full_bar(s));
                }
            }
        }
        if (!ok) {
            // let the copies in flight land before the CTA exits
            landed_from = u > STAGES ? u - STAGES : 0;
            for (unsigned v = landed_from; v < u; ++v)
                mbar_wait(full_bar(static_cast<int>(v & (STAGES - 1))), (v / STAGES) & 1,
                          2000000000ll);
        }
        return;
    }

    const int frames = prm.B * prm.T;

    // ---------------------------------------------------------- dp4a warps
    // Channels MMA_COLS .. BN - 1 of every tile, rows DW_ROWS dw .. DW_ROWS dw
    // + DW_ROWS - 1: lane (rg, cg) = (lane / 8, lane % 8) accumulates rows
    // DW_ROWS dw + RI rg + i (i < RI) and channels MMA_COLS + 8 cg + j (j < 8)
    // with dp4a on the same stages the MMA warps read.  Each lane walks the
    // eight 16-byte k chunks of a stage starting at chunk cg: the four lanes
    // of a channel group then read the same W chunk (one broadcast) and the
    // eight groups' chunks fall on the eight bank groups of the swizzled
    // rows, while the X loads of a row group cover every bank group too.
    if (warp >= NCW) {
        const int dw = warp - NCW;
        const int rg = lane >> 3, cg = lane & 7;
        const int r0 = DW_ROWS * dw + RI * rg;
        const int r7 = r0 & 7;          // 0 or 4: r7 + i = r7 | i for i < RI
        const int c0 = MMA_COLS + 8 * cg;
        unsigned u = 0;
        for (unsigned idx = blockIdx.x; idx < prm.ntiles; idx += gridDim.x) {
            const Tile L = tile_of(idx, prm);
            const int n0 = L.nt * BN;
            int acc[RI][8];
#pragma unroll
            for (int i = 0; i < RI; ++i)
#pragma unroll
                for (int j = 0; j < 8; ++j) acc[i][j] = 0;
            for (int it = 0; it < kt; ++it, ++u) {
                const int s = static_cast<int>(u & (STAGES - 1));
                if (!warp_wait(full_bar(s), (u / STAGES) & 1, prm.timeout_cycles)) {
                    if (lane == 0) atomicOr(prm.err, 1);
                    return;
                }
                const uint32_t abase = stage(s) + r0 * 128;
                const uint32_t bbase = stage(s) + A_BYTES + c0 * 128;
#pragma unroll (DW_UNROLL)
                for (int c = 0; c < 8; ++c) {
                    const int kc = (c + cg) & 7;
                    uint4 a[RI];
#pragma unroll
                    for (int i = 0; i < RI; ++i)
                        a[i] = lds128(abase + i * 128 + ((kc ^ (r7 | i)) << 4));
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint4 b = lds128(bbase + j * 128 + ((kc ^ j) << 4));
#pragma unroll
                        for (int i = 0; i < RI; ++i) {
                            acc[i][j] = __dp4a(static_cast<int>(a[i].x), static_cast<int>(b.x), acc[i][j]);
                            acc[i][j] = __dp4a(static_cast<int>(a[i].y), static_cast<int>(b.y), acc[i][j]);
                            acc[i][j] = __dp4a(static_cast<int>(a[i].z), static_cast<int>(b.z), acc[i][j]);
                            acc[i][j] = __dp4a(static_cast<int>(a[i].w), static_cast<int>(b.w), acc[i][j]);
                        }
                    }
                }
                release_stage(empty_bar(s), lane);
            }

            // epilogue: eight channels per lane, one 8-byte (4-byte gated)
            // segment per row, straight to global memory
            int cb[8], cm[8], ce[8];
            bool bad = false;
#pragma unroll
            for (int j = 0; j < 8; ++j) channel_consts(prm, n0 + c0 + j, cb[j], cm[j], ce[j], bad);
            if (bad) atomicOr(prm.err, ERR_PARAM);
            int hh = L.nt, grp = 0;
            if (prm.y_layout == LAYOUT_HEADS)
                while (hh >= prm.heads_per_group) {   // at most G - 1 steps
                    hh -= prm.heads_per_group;
                    ++grp;
                }
#pragma unroll
            for (int i = 0; i < RI; ++i) {
                if (EPI == EPI_GLU) {
                    uint32_t w = 0;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const int za = requant(acc[i][2 * q], cb[2 * q], cm[2 * q], ce[2 * q]);
                        const int zb = requant(acc[i][2 * q + 1], cb[2 * q + 1], cm[2 * q + 1],
                                               ce[2 * q + 1]);
                        w |= (static_cast<uint32_t>(glu_i8(za, zb, prm)) & 0xffu) << (8 * q);
                    }
                    const long long off = y_offset(prm, L, r0 + i, (n0 + c0) >> 1, prm.N >> 1, hh, grp);
                    if (off >= 0) *reinterpret_cast<uint32_t *>(prm.y + off) = w;
                } else {
                    uint32_t w[2] = {0u, 0u};
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        uint32_t o = static_cast<uint32_t>(requant(acc[i][j], cb[j], cm[j], ce[j])) & 0xffu;
                        if (EPI == EPI_SWISH) o = swish_lut[o];
                        w[j >> 2] |= o << (8 * (j & 3));
                    }
                    const int col = prm.y_layout == LAYOUT_ROWS ? n0 + c0 : c0;
                    const long long off = y_offset(prm, L, r0 + i, col, prm.N, hh, grp);
                    if (off >= 0) {
                        if (EPI == EPI_RES) {
                            const uint2 xr = *reinterpret_cast<const uint2 *>(prm.res + off);
                            w[0] = residual4(xr.x, w[0], prm.res_mx, prm.res_my, prm.res_s);
                            w[1] = residual4(xr.y, w[1], prm.res_mx, prm.res_my, prm.res_s);
                        }
                        *reinterpret_cast<uint2 *>(prm.y + off) = make_uint2(w[0], w[1]);
                    }
                }
            }
        }
        return;
    }

    // ---------------------------------------------------------- MMA warps
    // Channels 0 .. MMA_COLS - 1: warp (wm, wn) takes rows 64 wm .. 64 wm +
    // 63 and channels 16 wn .. 16 wn + 15 (two n8 tiles).
    const int wm = warp & 1;
    const int wn = warp >> 1;
    const int g = lane >> 2, t4 = lane & 3;
    const int lm_row = lane & 7, lm_mat = lane >> 3;
    const uint32_t ob = base + SMEM_OUT + warp * OUT_WARP_BYTES;

    unsigned u = 0;
    for (unsigned idx = blockIdx.x; idx < prm.ntiles; idx += gridDim.x) {
        const Tile L = tile_of(idx, prm);
        const int n0 = L.nt * BN;

        int acc[4][2][4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 2; ++j)
                acc[i][j][0] = acc[i][j][1] = acc[i][j][2] = acc[i][j][3] = 0;

        for (int it = 0; it < kt; ++it, ++u) {
            const int s = static_cast<int>(u & (STAGES - 1));
            if (!warp_wait(full_bar(s), (u / STAGES) & 1, prm.timeout_cycles)) {
                if (lane == 0) atomicOr(prm.err, 1);
                return;
            }
            const uint32_t at = stage(s) + (64 * wm) * 128;
            const uint32_t bt = stage(s) + A_BYTES + (16 * wn) * 128;
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
                uint32_t af[4][4], bf[2][2];
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    ldsm_x4(at + swz(16 * i + (lm_mat & 1) * 8 + lm_row, 2 * ks + (lm_mat >> 1)),
                            af[i][0], af[i][1], af[i][2], af[i][3]);
                ldsm_x4(bt + swz((lm_mat >> 1) * 8 + lm_row, 2 * ks + (lm_mat & 1)), bf[0][0],
                        bf[0][1], bf[1][0], bf[1][1]);
#pragma unroll
                for (int i = 0; i < 4; ++i)
#pragma unroll
                    for (int j = 0; j < 2; ++j) mma_s8s8(acc[i][j], af[i], bf[j][0], bf[j][1]);
            }
            release_stage(empty_bar(s), lane);
        }

        // ------------------------------------------------------ epilogue
        // per-channel constants of this thread's four channels (Eq. 7),
        // loaded after the main loop so that they hold no registers during it
        int cb[4], cm[4], ce[4];
        bool bad = false;
#pragma unroll
        for (int j = 0; j < 2; ++j)
#pragma unroll
            for (int q = 0; q < 2; ++q)
                channel_consts(prm, n0 + 16 * wn + 8 * j + 2 * t4 + q, cb[2 * j + q], cm[2 * j + q],
                               ce[2 * j + q], bad);
        if (bad) atomicOr(prm.err, ERR_PARAM);

        if (EPI == EPI_GLU) {
            // pairs (a_c, b_c) in columns (2t, 2t + 1) of each n8 tile: output
            // channel 4j + t of this warp's 8 (row of 8 bytes)
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 2; ++j)
#pragma unroll
                    for (int rr = 0; rr < 2; ++rr) {
                        const int za = requant(acc[i][j][2 * rr], cb[2 * j], cm[2 * j], ce[2 * j]);
                        const int zb = requant(acc[i][j][2 * rr + 1], cb[2 * j + 1], cm[2 * j + 1],
                                               ce[2 * j + 1]);
                        const uint32_t o = static_cast<uint32_t>(glu_i8(za, zb, prm)) & 0xffu;
                        const int r = 16 * i + g + 8 * rr;
                        asm volatile("st.shared.u8 [%0], %1;" ::"r"(ob + r * OUT_ROW + 4 * j + t4),
                                     "r"(o)
                                     : "memory");
                    }
            __syncwarp();
            // 64 rows x 8 bytes: lane -> rows lane, lane + 32
#pragma unroll
            for (int it = 0; it < 2; ++it) {
                const int r = 32 * it + lane;
                const int2 v2 = lds64(ob + r * OUT_ROW);
                const uint2 v = make_uint2(static_cast<uint32_t>(v2.x), static_cast<uint32_t>(v2.y));
                if (L.m0 + 64 * wm + r < frames) {
                    const size_t off = static_cast<size_t>(L.m0 + 64 * wm + r) * (prm.N >> 1) +
                                       (n0 >> 1) + 8 * wn;
                    *reinterpret_cast<uint2 *>(prm.y + off) = v;
                }
            }
            __syncwarp();
            continue;
        }

#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
            for (int j = 0; j < 2; ++j)
#pragma unroll
                for (int rr = 0; rr < 2; ++rr) {
                    uint32_t two = 0;
#pragma unroll
                    for (int q = 0; q < 2; ++q) {
                        const int c = 2 * j + q;
                        uint32_t o = static_cast<uint32_t>(requant(acc[i][j][2 * rr + q], cb[c], cm[c],
                                                                   ce[c])) & 0xffu;
                        if (EPI == EPI_SWISH) o = swish_lut[o];
                        two |= o << (8 * q);
                    }
                    const int r = 16 * i + g + 8 * rr;
                    asm volatile("st.shared.u16 [%0], %1;" ::"r"(ob + r * OUT_ROW + 8 * j + 2 * t4),
                                 "h"(static_cast<unsigned short>(two))
                                 : "memory");
                }
        __syncwarp();

        int hh = L.nt, grp = 0;
        if (prm.y_layout == LAYOUT_HEADS)
            while (hh >= prm.heads_per_group) {   // at most G - 1 steps
                hh -= prm.heads_per_group;
                ++grp;
            }
        // 64 rows x 16 bytes: lane -> rows lane, lane + 32
#pragma unroll
        for (int it = 0; it < 2; ++it) {
            const int r = 32 * it + lane;
            uint4 v = lds128(ob + r * OUT_ROW);
            const int col = prm.y_layout == LAYOUT_ROWS ? n0 + 16 * wn : 16 * wn;
            const long long off = y_offset(prm, L, 64 * wm + r, col, prm.N, hh, grp);
            if (off >= 0) {
                if (EPI == EPI_RES) {
                    const uint4 xr = *reinterpret_cast<const uint4 *>(prm.res + off);
                    v = make_uint4(residual4(xr.x, v.x, prm.res_mx, prm.res_my, prm.res_s),
                                   residual4(xr.y, v.y, prm.res_mx, prm.res_my, prm.res_s),
                                   residual4(xr.z, v.z, prm.res_mx, prm.res_my, prm.res_s),
                                   residual4(xr.w, v.w, prm.res_mx, prm.res_my, prm.res_s));
                }
                *reinterpret_cast<uint4 *>(prm.y + off) = v;
            }
        }
        __syncwarp();
    }
}

}  // namespace ipl
