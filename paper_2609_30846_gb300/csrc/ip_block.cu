// Host side of the remaining Conformer-block parts of the C ABI
// (include/ip_mhsa.h): residual additions, the depthwise convolution with
// folded BatchNorm and Swish, and their offline constants.  Device code:
// ip_block_kernels.cuh.
#include "ip_mhsa.h"
#include "ip_block_kernels.cuh"
#include "ip_host_util.h"

#include <cuda_runtime.h>

#include <cmath>
#include <mutex>

namespace {

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

std::mutex g_mu;
int g_sms[64] = {0};

int sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_sms[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
        g_sms[dev] = n;
    }
    return g_sms[dev];
}

// Resident CTAs of dwconv_swish_x4_kernel<K> on the current device (SMs x
// CTAs per SM), looked up once per device and K.
int g_dw4_slots[64][ipb::DW_KMAX + 1] = {{0}};

template <int K>
cudaError_t launch_dw4(ipb::DwParams p, cudaStream_t st) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    int slots = 0;
    {
        std::lock_guard<std::mutex> lock(g_mu);
        slots = g_dw4_slots[dev][K];
    }
    if (slots == 0) {
        int per_sm = 0;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ipb::dwconv_swish_x4_kernel<K>,
                                                          ipb::DW4_THREADS, 0);
        if (e != cudaSuccess) return e;
        slots = (per_sm > 0 ? per_sm : 1) * sm_count();
        if (slots <= 0) return cudaErrorInvalidValue;
        std::lock_guard<std::mutex> lock(g_mu);
        g_dw4_slots[dev][K] = slots;
    }
    // channel blocks of 256 channels; the frames of each split evenly over
    // the slots left for it
    const int ncb = (p.C / 4 + ipb::DW4_THREADS - 1) / ipb::DW4_THREADS;
    const long long frames = static_cast<long long>(p.B) * p.T;
    long long per_block = slots / ncb > 0 ? slots / ncb : 1;
    // a multiple of the frames of one step, so that only utterance ends
    // leave a partly used step
    constexpr int step = 4 * ipb::DW4_BLOCKS;
    const long long per = ((frames + per_block - 1) / per_block + step - 1) / step * step;
    per_block = (frames + per - 1) / per;
    p.frames_per_cta = static_cast<uint32_t>(per);
    p.t_magic = iph::div_magic(static_cast<unsigned long long>(p.T));
    return iph::launch_pdl(ipb::dwconv_swish_x4_kernel<K>,
                           dim3(static_cast<unsigned>(per_block), static_cast<unsigned>(ncb)),
                           dim3(ipb::DW4_THREADS), 0, st, p);
}

int check_swish16(const ip_swish16_params *p) {
    if (p->q_c < 1 || p->q_c >= (1 << 16) || p->q_one < 1 || p->q_one >= (1ll << 31) ||
        p->q_one < static_cast<long long>(p->q_c) * p->q_c || p->m < 0 || p->s < 0 || p->s > 31)
        return IP_ERR_PARAM;
    return IP_OK;
}

}  // namespace

extern "C" {

int ip_residual_i8(const int8_t *x, const int8_t *y, long long n, int32_t m_x, int32_t m_y,
                   int32_t s, int8_t *z, ip_stream_t stream) {
    if (n < 0) return IP_ERR_SHAPE;
    if (m_x < 0 || m_y < 0 || s < 0 || s > 31) return IP_ERR_PARAM;
    if (n == 0) return IP_OK;
    if (!x || !y || !z) return IP_ERR_NULL;
    if (!aligned(x, 16) || !aligned(y, 16) || !aligned(z, 16)) return IP_ERR_ALIGN;
    const int nsm = sm_count();
    if (nsm <= 0) return IP_ERR_CUDA;
    ipb::ResidualParams p;
    p.x = x;
    p.y = y;
    p.z = z;
    p.n = n;
    p.m_x = m_x;
    p.m_y = m_y;
    p.s = s;
    const long long vec = (n >> 4) + 1;
    long long blocks = (vec + ipb::RES_THREADS - 1) / ipb::RES_THREADS;
    const long long cap = static_cast<long long>(nsm) * 8;
    blocks = blocks < cap ? blocks : cap;
    if (iph::launch_pdl(ipb::residual_i8_kernel, dim3(static_cast<unsigned>(blocks)),
                        dim3(ipb::RES_THREADS), 0, reinterpret_cast<cudaStream_t>(stream), p) !=
        cudaSuccess)
        return IP_ERR_CUDA;
    return cudaGetLastError() == cudaSuccess ? IP_OK : IP_ERR_CUDA;
}

int ip_dwconv_swish_i8(const int8_t *x, int B, int T, int C, const int8_t *w, int K,
                       const int32_t *bias, const int32_t *m, const int32_t *s,
                       const ip_swish16_params *sw, int8_t *y, void *workspace,
                       size_t workspace_bytes, ip_stream_t stream) {
    if (B < 0 || B > IP_MAX_B || T < 1 || C < 1 || K < 1 || K % 2 == 0 || K > ipb::DW_KMAX)
        return IP_ERR_SHAPE;
    if ((T + ipb::DW_FRAMES - 1) / ipb::DW_FRAMES > 65535) return IP_ERR_SHAPE;
    if (!sw) return IP_ERR_NULL;
    int rc = check_swish16(sw);
    if (rc != IP_OK) return rc;
    if (B == 0) return IP_OK;
    if (!x || !w || !bias || !m || !s || !y || !workspace) return IP_ERR_NULL;
    if (!aligned(bias, 4) || !aligned(m, 4) || !aligned(s, 4) || !aligned(workspace, 256))
        return IP_ERR_ALIGN;
    if (workspace_bytes < 256) return IP_ERR_WORKSPACE;
    ipb::DwParams p;
    p.x = x;
    p.w = w;
    p.bias = bias;
    p.m = m;
    p.s = s;
    p.y = y;
    p.B = B;
    p.T = T;
    p.C = C;
    p.K = K;
    p.sw_qc = sw->q_c;
    p.sw_qone = sw->q_one;
    p.sw_m = sw->m;
    p.sw_s = sw->s;
    p.err = static_cast<int *>(workspace);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t lrc;
    if (C % 4 == 0 && aligned(x, 4) && aligned(y, 4) && aligned(w, 4) &&
        static_cast<long long>(B) * T < (1ll << 31)) {
        // four channels per thread, one CTA per resident slot
        switch (K) {   // odd, 1 .. DW_KMAX (checked above)
            case 1: lrc = launch_dw4<1>(p, st); break;
            case 3: lrc = launch_dw4<3>(p, st); break;
            case 5: lrc = launch_dw4<5>(p, st); break;
            case 7: lrc = launch_dw4<7>(p, st); break;
            case 9: lrc = launch_dw4<9>(p, st); break;
            case 11: lrc = launch_dw4<11>(p, st); break;
            case 13: lrc = launch_dw4<13>(p, st); break;
            default: lrc = launch_dw4<15>(p, st); break;
        }
        if (lrc != cudaSuccess) return IP_ERR_CUDA;
        return cudaGetLastError() == cudaSuccess ? IP_OK : IP_ERR_CUDA;
    }
    const dim3 grid((C + ipb::DW_THREADS - 1) / ipb::DW_THREADS,
                    (T + ipb::DW_FRAMES - 1) / ipb::DW_FRAMES, B);
    switch (K) {   // odd, 1 .. DW_KMAX (checked above)
        case 1: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<1>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
        case 3: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<3>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
        case 5: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<5>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
        case 7: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<7>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
        case 9: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<9>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
        case 11: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<11>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
        case 13: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<13>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
        default: lrc = iph::launch_pdl(ipb::dwconv_swish_kernel<15>, grid, dim3(ipb::DW_THREADS), 0, st, p); break;
    }
    if (lrc != cudaSuccess) return IP_ERR_CUDA;
    return cudaGetLastError() == cudaSuccess ? IP_OK : IP_ERR_CUDA;
}

int ip_residual_params(double S_x, double S_y, double S_z, double alpha, int32_t *m_x,
                       int32_t *m_y, int32_t *s) {
    if (!m_x || !m_y || !s) return IP_ERR_NULL;
    if (!(S_x > 0.0) || !(S_y > 0.0) || !(S_z > 0.0) || !(alpha > 0.0)) return IP_ERR_PARAM;
    return ip_dyadic_pair(S_x / S_z, alpha * S_y / S_z, m_x, m_y, s);
}

int ip_glu_params(double S_a, double S_b, double S_y, ip_swish_params *out) {
    if (!out) return IP_ERR_NULL;
    if (!(S_a > 0.0) || !(S_b > 0.0) || !(S_y > 0.0) || !std::isfinite(S_a) ||
        !std::isfinite(S_b) || !std::isfinite(S_y))
        return IP_ERR_PARAM;
    const double s_t = -IP_SWISH_A * (S_b / 2.0) * (S_b / 2.0);
    const double qc = std::floor(2.0 * IP_SWISH_C / S_b + 0.5);
    const double qone = std::floor(1.0 / s_t + 0.5);
    if (qc < 1.0 || qc >= 32768.0 || qone < 1.0 || qone >= 8388608.0 || qone < qc * qc)
        return IP_ERR_PARAM;
    ip_swish_params p;
    p.q_c = static_cast<int32_t>(qc);
    p.q_one = static_cast<int32_t>(qone);
    const int rc = ip_dyadic_multiplier(S_a * s_t / (2.0 * S_y), &p.m, &p.s);
    if (rc != IP_OK) return rc;
    *out = p;
    return IP_OK;
}

int ip_swish16_params_from_scales(double S_z, double S_y, ip_swish16_params *out) {
    if (!out) return IP_ERR_NULL;
    if (!(S_z > 0.0) || !(S_y > 0.0) || !std::isfinite(S_z) || !std::isfinite(S_y))
        return IP_ERR_PARAM;
    const double s_t = -IP_SWISH_A * (S_z / 2.0) * (S_z / 2.0);
    const double qc = std::floor(2.0 * IP_SWISH_C / S_z + 0.5);
    const double qone = std::floor(1.0 / s_t + 0.5);
    if (qc < 1.0 || qc >= 65536.0 || qone < 1.0 || qone >= 2147483648.0 || qone < qc * qc)
        return IP_ERR_PARAM;
    ip_swish16_params p;
    p.q_c = static_cast<int32_t>(qc);
    p.q_one = static_cast<long long>(qone);
    const int rc = ip_dyadic_multiplier(S_z * s_t / (2.0 * S_y), &p.m, &p.s);
    if (rc != IP_OK) return rc;
    *out = p;
    return IP_OK;
}

}  // extern "C"
