// Device code of the remaining integer parts of the I-Parakeet Conformer
// block for sm_103a (Sec. 2.1 Eqs. 1-5, Sec. 2.2, Sec. 3.2, Sec. 3.3):
// residual additions, and the ConvBlock's depthwise convolution with folded
// BatchNorm onto the INT16 grid followed by the minimax Swish.  Integer
// arithmetic only: no floating-point type, no division by a run-time value.
#pragma once

#include <stdint.h>

#include "ip_ptx.cuh"

namespace ipb {

using namespace ipk;

constexpr int RES_THREADS = 256;
constexpr int DW_THREADS = 256;      // one thread per channel of a 256-channel block
constexpr int DW_FRAMES = 32;        // frames per CTA
constexpr int DW_KMAX = 15;          // largest (odd) kernel
constexpr int ERR_PARAM = 16;

struct ResidualParams {
    const int8_t *x, *y;
    int8_t *z;
    long long n;
    int m_x, m_y, s;
};


__global__ void __launch_bounds__(RES_THREADS) residual_i8_kernel(const ResidualParams p) {
    pdl_launch_dependents();
    pdl_wait();   // the grid before this one on the stream: complete, memory visible
    const long long nv = p.n >> 4;   // 16-byte vectors
    const long long stride = static_cast<long long>(gridDim.x) * RES_THREADS;
    for (long long i = static_cast<long long>(blockIdx.x) * RES_THREADS + threadIdx.x; i < nv;
         i += stride) {
        const uint4 a = __ldcs(reinterpret_cast<const uint4 *>(p.x) + i);
        const uint4 b = __ldcs(reinterpret_cast<const uint4 *>(p.y) + i);
        __stcs(reinterpret_cast<uint4 *>(p.z) + i,
               make_uint4(residual4(a.x, b.x, p.m_x, p.m_y, p.s), residual4(a.y, b.y, p.m_x, p.m_y, p.s),
                          residual4(a.z, b.z, p.m_x, p.m_y, p.s), residual4(a.w, b.w, p.m_x, p.m_y, p.s)));
    }
    // the tail of n (fewer than 16 bytes)
    const long long tail = nv << 4;
    const long long k = tail + static_cast<long long>(blockIdx.x) * RES_THREADS + threadIdx.x;
    if (k < p.n && k < tail + 16)
        p.z[k] = static_cast<int8_t>(residual_one(p.x[k], p.y[k], p.m_x, p.m_y, p.s));
}

struct DwParams {
    const int8_t *x;          // [B][T][C]
    const int8_t *w;          // [C][K]
    const int32_t *bias;      // [C]
    const int32_t *m, *s;     // [C], onto the INT16 grid
    int8_t *y;                // [B][T][C]
    int B, T, C, K;
    int sw_qc, sw_m, sw_s;    // Swish of the INT16 value onto int8
    long long sw_qone;
    int *err;
    // four-channels-per-thread kernel: CTA (j, cb) takes channel block cb
    // and the frames [j per, (j + 1) per) of the B T frames in (b, t) order
    uint32_t frames_per_cta;
    unsigned long long t_magic;   // udiv_magic constant of T
};

// Swish of one INT16 value z (Eqs. 12-13 on the grid of z): t = q_one +
// sgn(z) (q_one - D^2) < 2^32, P = z t with |P| < 2^47, and round(m P /
// 2^(31+s)) with m P up to 78 bits, exactly: P = P_hi 2^31 + P_lo with
// 0 <= P_lo < 2^31, so floor((m P + 2^(30+s)) / 2^(31+s)) =
// floor((m P_hi + floor((m P_lo + 2^(30+s)) / 2^31)) / 2^s).
__device__ __forceinline__ int swish16(int z, const DwParams &p) {
    const long long a = z < 0 ? -z : z;
    const long long dc = (a < p.sw_qc ? a : p.sw_qc) - p.sw_qc;
    const long long L = p.sw_qone - dc * dc;
    const long long t = z > 0 ? p.sw_qone + L : (z < 0 ? p.sw_qone - L : p.sw_qone);
    const long long P = static_cast<long long>(z) * t;
    const long long phi = P >> 31;                       // floor(P / 2^31)
    const long long plo = P & 0x7fffffffll;
    const long long m = p.sw_m;
    const long long q1 = m * phi + ((m * plo + (1ll << (30 + p.sw_s))) >> 31);
    const long long r = q1 >> p.sw_s;
    return r > 127 ? 127 : (r < -127 ? -127 : static_cast<int>(r));
}

// Depthwise convolution over time (zero padding at both ends of each
// utterance), per-channel requantisation onto INT16 (folded BatchNorm), and
// the Swish onto int8.  Thread: one channel; CTA: 256 channels x DW_FRAMES
// frames of one utterance, a sliding window of the K input frames in
// registers (K, odd, a compile-time constant: no unused taps).
template <int K>
__global__ void __launch_bounds__(DW_THREADS) dwconv_swish_kernel(const DwParams p) {
    pdl_launch_dependents();
    pdl_wait();   // the grid before this one on the stream: complete, memory visible
    const int c = blockIdx.x * DW_THREADS + threadIdx.x;
    const int t0 = blockIdx.y * DW_FRAMES;
    const int b = blockIdx.z;
    if (c >= p.C) return;
    constexpr int half = K >> 1;
    int w[K];
#pragma unroll
    for (int k = 0; k < K; ++k) w[k] = p.w[static_cast<size_t>(c) * K + k];
    int bias = p.bias[c], mm = p.m[c], ss = p.s[c];
    if (mm < 0 || ss < 0 || ss > 31 || bias >= (1 << 30) || bias <= -(1 << 30)) {
        atomicOr(p.err, ERR_PARAM);
        mm = mm < 0 ? 0 : mm;
        ss = ss < 0 ? 0 : (ss > 31 ? 31 : ss);
        bias = 0;
    }
    const int8_t *xb = p.x + static_cast<size_t>(b) * p.T * p.C + c;
    int8_t *yb = p.y + static_cast<size_t>(b) * p.T * p.C + c;
    // window[k] holds x[t + k - half] for the current output frame t
    int win[K];
#pragma unroll
    for (int k = 0; k < K; ++k) {
        const int tt = t0 + k - half;
        win[k] = (tt >= 0 && tt < p.T) ? xb[static_cast<size_t>(tt) * p.C] : 0;
    }
    const int tend = t0 + DW_FRAMES < p.T ? t0 + DW_FRAMES : p.T;
    for (int t = t0; t < tend; ++t) {
        int acc = bias;
#pragma unroll
        for (int k = 0; k < K; ++k) acc += w[k] * win[k];   // |acc| < 2^30 + 2^18
        // onto INT16: round(m acc / 2^(31+s)); |m acc| < 2^62 + 2^50
        const long long v = static_cast<long long>(mm) * acc + (1ll << (30 + ss));
        const long long h = v >> (31 + ss);
        const int z16 = static_cast<int>(h > 32767 ? 32767 : (h < -32767 ? -32767 : h));
        yb[static_cast<size_t>(t) * p.C] = static_cast<int8_t>(swish16(z16, p));
        // slide the window by one frame
#pragma unroll
        for (int k = 0; k < K - 1; ++k) win[k] = win[k + 1];
        const int tn = t + 1 + (K - 1) - half;   // frame entering at slot K - 1
        win[K - 1] = (tn < p.T) ? xb[static_cast<size_t>(tn) * p.C] : 0;
    }
}

// ---- four channels per thread ----------------------------------------------
// The same computation for C a multiple of 4 (and 4-byte aligned x, y, w):
// a thread takes the four channels of one 32-bit word of a frame.  Four
// frame words are byte-transposed into four channel words (four
// consecutive frames of one channel each), so that one dp4a covers four
// taps: output frame t of channel c is the sum over q of dp4a(the four
// frames t - K/2 + 4q .. + 3, taps 4q .. 4q + 3), the frame words taken at
// any byte offset by a funnel shift of two neighbouring channel words.  The
// two roundings are done in sign and magnitude with 32 x 32 -> 64-bit
// products: for n = [v < 0], A = |v| and h = 2^(e-1),
//   floor((m v + h) / 2^e) = (1 - 2n) floor((m A + h - n) / 2^e),
// because floor((h - X) / 2h) = -floor((X + h - 1) / 2h).
constexpr int DW4_THREADS = 64;      // 256 channels per CTA
constexpr int DW4_BLOCKS = 2;        // blocks of four output frames per step

struct Swish16K {
    uint32_t q_c, two_qone, m;
    int s;
    unsigned long long h;            // 2^(30+s)
};

// Eq. 7 onto the INT16 grid, then the Swish of that INT16 value onto int8
// (Eqs. 12-13), for one channel: acc the convolution sum with bias, m and s
// the channel's multiplier and shift, h = 2^(30+s).  The INT16 value is z =
// (1 - 2n) a with a = min(floor((m |acc| + h - n) / 2^(31+s)), 32767); its
// Swish product z t is (1 - 2n) U with U = a t' < 2^47, t' = 2 q_one - D^2
// for z > 0 and D^2 for z < 0 (D = q_c - min(a, q_c)); m_sw U (up to 78 bits)
// is split at bit 31, U = u_hi 2^31 + u_lo.  Returns the int8 in the low byte.
__device__ __forceinline__ uint32_t dw_out(int acc, uint32_t m, int s, unsigned long long h,
                                           const Swish16K &sw) {
    const uint32_t n = acc < 0 ? 1u : 0u;
    const uint32_t A = acc < 0 ? 0u - static_cast<uint32_t>(acc) : static_cast<uint32_t>(acc);
    const unsigned long long w = static_cast<unsigned long long>(m) * A + (h - n);   // < 2^63
    const uint32_t R = __funnelshift_r(static_cast<uint32_t>(w), static_cast<uint32_t>(w >> 32), 31) >> s;
    const uint32_t a = min(R, 32767u);
    const uint32_t dc = sw.q_c - min(a, sw.q_c);
    const uint32_t d2 = dc * dc;                          // <= q_c^2 <= q_one < 2^31
    const uint32_t tt = n ? d2 : sw.two_qone - d2;
    const unsigned long long U = static_cast<unsigned long long>(a) * tt;
    const uint32_t ulo = static_cast<uint32_t>(U) & 0x7fffffffu;
    const uint32_t uhi = __funnelshift_r(static_cast<uint32_t>(U), static_cast<uint32_t>(U >> 32), 31);
    const unsigned long long w2 = static_cast<unsigned long long>(sw.m) * ulo + (sw.h - n);
    const uint32_t f = __funnelshift_r(static_cast<uint32_t>(w2), static_cast<uint32_t>(w2 >> 32), 31);
    const unsigned long long X = static_cast<unsigned long long>(sw.m) * uhi + f;   // < 2^48
    const uint32_t xlo = __funnelshift_r(static_cast<uint32_t>(X), static_cast<uint32_t>(X >> 32), sw.s);
    const uint32_t xhi = static_cast<uint32_t>(X >> 32) >> sw.s;
    const uint32_t r = xhi != 0u ? 127u : min(xlo, 127u);
    return n ? 0u - r : r;
}

// Byte transpose of a 4x4 block: y_c = [x0.b_c, x1.b_c, x2.b_c, x3.b_c].
__device__ __forceinline__ void dw_transpose4(uint32_t x0, uint32_t x1, uint32_t x2, uint32_t x3,
                                              uint32_t (&y)[4]) {
    const uint32_t t0 = __byte_perm(x0, x1, 0x5140);   // x0.b0 x1.b0 x0.b1 x1.b1
    const uint32_t t1 = __byte_perm(x0, x1, 0x7362);   // x0.b2 x1.b2 x0.b3 x1.b3
    const uint32_t t2 = __byte_perm(x2, x3, 0x5140);
    const uint32_t t3 = __byte_perm(x2, x3, 0x7362);
    y[0] = __byte_perm(t0, t2, 0x5410);
    y[1] = __byte_perm(t0, t2, 0x7632);
    y[2] = __byte_perm(t1, t3, 0x5410);
    y[3] = __byte_perm(t1, t3, 0x7632);
}

// Output frames [ts, te) of one utterance for the thread's four channels.
// Frames are taken in blocks of four from p0 = ts - K/2 (frames outside
// [0, T) read as zero): block u holds frames p0 + 4u .. p0 + 4u + 3, as one
// channel word per channel.  Output frame ts + 4v + i reads the stream at
// offsets 4v + i .. 4v + i + K - 1, i.e. the words of blocks v .. v + Q
// shifted by i bytes.  A step makes DW4_BLOCKS blocks of four outputs; the
// frame words of the next step's new blocks are loaded before this step's
// arithmetic, so their latency hides behind it.
template <int K>
__device__ __forceinline__ void dw4_segment(const DwParams &p, const uint32_t *xb, uint32_t *yb,
                                            int cw, int ts, int te, const uint32_t (&wq)[4][(K + 3) / 4],
                                            const uint32_t (&mq)[4], const int (&sq)[4],
                                            const int (&bq)[4], const unsigned long long (&hq)[4],
                                            const Swish16K &sw) {
    constexpr int Q = (K + 3) / 4;    // weight words (taps in fours)
    constexpr int NB = DW4_BLOCKS;
    constexpr int NA = Q + NB;        // blocks a step reads
    const int T = p.T;
    const int p0 = ts - (K >> 1);
    auto load_block = [&](int u, uint32_t (&xw)[4]) {
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int tt = p0 + 4 * u + r;
            xw[r] = (tt >= 0 && tt < T) ? __ldg(xb + static_cast<size_t>(tt) * cw) : 0u;
        }
    };
    uint32_t A[NA][4];   // A[u][j]: channel j of block NB v + u for step v
    uint32_t nx[NB][4];  // frame words of the next step's new blocks
#pragma unroll
    for (int u = 0; u < Q; ++u) {
        load_block(u, nx[0]);
        dw_transpose4(nx[0][0], nx[0][1], nx[0][2], nx[0][3], A[u]);
    }
#pragma unroll
    for (int b = 0; b < NB; ++b) load_block(Q + b, nx[b]);
    const int nsteps = (te - ts + 4 * NB - 1) / (4 * NB);
#pragma unroll 1
    for (int v = 0; v < nsteps; ++v) {
#pragma unroll
        for (int b = 0; b < NB; ++b) dw_transpose4(nx[b][0], nx[b][1], nx[b][2], nx[b][3], A[Q + b]);
        if (v + 1 < nsteps) {
#pragma unroll
            for (int b = 0; b < NB; ++b) load_block(NB * (v + 1) + Q + b, nx[b]);
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            uint32_t o[4][4];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    int acc = bq[j];
#pragma unroll
                    for (int q = 0; q < Q; ++q) {
                        const uint32_t win =
                            i == 0 ? A[b + q][j] : __funnelshift_r(A[b + q][j], A[b + q + 1][j], 8 * i);
                        acc = __dp4a(static_cast<int>(win), static_cast<int>(wq[j][q]), acc);
                    }
                    o[i][j] = dw_out(acc, mq[j], sq[j], hq[j], sw);
                }
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int t = ts + 4 * (NB * v + b) + i;
                if (t < te)
                    yb[static_cast<size_t>(t) * cw] = __byte_perm(
                        __byte_perm(o[i][0], o[i][1], 0x0040), __byte_perm(o[i][2], o[i][3], 0x0040), 0x5410);
            }
        }
#pragma unroll
        for (int u = 0; u < Q; ++u)
#pragma unroll
            for (int j = 0; j < 4; ++j) A[u][j] = A[u + NB][j];
    }
}

// Thread: channels 4 c4 .. 4 c4 + 3 of channel block blockIdx.y (256
// channels); CTA: a contiguous run of frames_per_cta of the B T frames,
// split at utterance boundaries (the zero padding of each utterance).  The
// grid holds one CTA per resident slot, so there is no partial second wave.
template <int K>
__global__ void __launch_bounds__(DW4_THREADS) dwconv_swish_x4_kernel(const DwParams p) {
    pdl_launch_dependents();
    pdl_wait();   // the grid before this one on the stream: complete, memory visible
    constexpr int Q = (K + 3) / 4;
    const int cw = p.C >> 2;                               // words per frame
    const int c4 = blockIdx.y * DW4_THREADS + threadIdx.x;
    if (c4 >= cw) return;
    // weights: wq[j][q] = taps 4q .. 4q + 3 of channel 4 c4 + j (zero past
    // K), from the 4 K consecutive bytes of the four channels in w
    uint32_t wq[4][Q];
    {
        const uint32_t *wp = reinterpret_cast<const uint32_t *>(p.w) + static_cast<size_t>(c4) * K;
        uint32_t raw[K];
#pragma unroll
        for (int i = 0; i < K; ++i) raw[i] = __ldg(wp + i);
#pragma unroll
        for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int q = 0; q < Q; ++q) {
                uint32_t v = 0;
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    const int k = 4 * q + r;
                    if (k < K) {
                        const int i = j * K + k;   // byte i of the four channels' taps
                        v |= ((raw[i >> 2] >> (8 * (i & 3))) & 0xffu) << (8 * r);
                    }
                }
                wq[j][q] = v;
            }
    }
    uint32_t mq[4];
    int sq[4], bq[4];
    unsigned long long hq[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int c = 4 * c4 + j;
        int bias = p.bias[c], mm = p.m[c], ss = p.s[c];
        if (mm < 0 || ss < 0 || ss > 31 || bias >= (1 << 30) || bias <= -(1 << 30)) {
            atomicOr(p.err, ERR_PARAM);
            mm = mm < 0 ? 0 : mm;
            ss = ss < 0 ? 0 : (ss > 31 ? 31 : ss);
            bias = 0;
        }
        mq[j] = static_cast<uint32_t>(mm);
        sq[j] = ss;
        bq[j] = bias;
        hq[j] = 1ull << (30 + ss);
    }
    Swish16K sw;
    sw.q_c = static_cast<uint32_t>(p.sw_qc);
    sw.two_qone = static_cast<uint32_t>(2 * p.sw_qone);
    sw.m = static_cast<uint32_t>(p.sw_m);
    sw.s = p.sw_s;
    sw.h = 1ull << (30 + p.sw_s);
    const uint32_t nframes = static_cast<uint32_t>(p.B) * static_cast<uint32_t>(p.T);   // < 2^31
    uint32_t f = blockIdx.x * p.frames_per_cta;
    const uint32_t fend = min(nframes, f + p.frames_per_cta);
    while (f < fend) {
        const uint32_t b = udiv_magic(f, p.t_magic);
        const int ts = static_cast<int>(f - b * static_cast<uint32_t>(p.T));
        const int te = min(p.T, ts + static_cast<int>(fend - f));
        const size_t base = static_cast<size_t>(b) * p.T * cw + c4;
        dw4_segment<K>(p, reinterpret_cast<const uint32_t *>(p.x) + base,
                       reinterpret_cast<uint32_t *>(p.y) + base, cw, ts, te, wq, mq, sq, bq, hq, sw);
        f += static_cast<uint32_t>(te - ts);
    }
}

}  // namespace ipb
