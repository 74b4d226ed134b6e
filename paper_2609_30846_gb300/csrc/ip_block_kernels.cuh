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

}  // namespace ipb
