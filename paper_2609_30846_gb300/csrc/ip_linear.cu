// Host side of the integer linear layer of the C ABI (include/ip_mhsa.h):
// argument validation, TMA tensor maps and the launch.  Device code:
// ip_linear_kernels.cuh.
#include "ip_mhsa.h"
#include "ip_linear_kernels.cuh"
#include "ip_host_util.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <mutex>

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// int8 tensor map of `rank` dimensions (innermost first; byte strides of
// dimensions 1..rank-1) with a box of 128 x 128 (x 1 ...), 128-byte swizzle;
// elements outside the tensor read as zero.
bool make_map(CUtensorMap *m, const void *base, int rank, const cuuint64_t *dims,
              const cuuint64_t *strides) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint32_t box[4] = {128, 128, 1, 1};
    const cuuint32_t estride[4] = {1, 1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, rank, const_cast<void *>(base), dims, strides,
              box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

std::mutex g_mu;
int g_smem_set[64] = {0};
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

int ensure_smem() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IP_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    if (g_smem_set[dev]) return IP_OK;
    if (cudaFuncSetAttribute(ipl::linear_i8_kernel<ipl::EPI_PLAIN>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             ipl::SMEM_LAUNCH) != cudaSuccess ||
        cudaFuncSetAttribute(ipl::linear_i8_kernel<ipl::EPI_SWISH>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             ipl::SMEM_LAUNCH) != cudaSuccess ||
        cudaFuncSetAttribute(ipl::linear_i8_kernel<ipl::EPI_GLU>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             ipl::SMEM_LAUNCH) != cudaSuccess ||
        cudaFuncSetAttribute(ipl::linear_i8_kernel<ipl::EPI_RES>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             ipl::SMEM_LAUNCH) != cudaSuccess)
        return IP_ERR_CUDA;
    g_smem_set[dev] = 1;
    return IP_OK;
}

int check_swish(const ip_swish_params *p) {
    if (p->q_c < 1 || p->q_c >= (1 << 15) || p->q_one < 1 || p->q_one >= (1 << 23) ||
        static_cast<long long>(p->q_one) < static_cast<long long>(p->q_c) * p->q_c ||
        p->m < 0 || p->s < 0 || p->s > 31)
        return IP_ERR_PARAM;
    return IP_OK;
}

// Residual operand of the RES epilogue: the tensor added and its constants.
struct ResidualArg {
    const int8_t *x;
    int32_t m_x, m_y, s;
};

int linear_launch(const int8_t *x, int x_layout, const int8_t *w, const int32_t *bias,
                  const int32_t *m, const int32_t *s, const ip_swish_params *sw, int epi, int B,
                  int T, int K, int N, int G, int8_t *y, int y_layout, void *workspace,
                  size_t workspace_bytes, ip_stream_t stream, const ResidualArg *res = nullptr) {
    if ((x_layout != IP_LAYOUT_ROWS && x_layout != IP_LAYOUT_HEADS) ||
        (y_layout != IP_LAYOUT_ROWS && y_layout != IP_LAYOUT_HEADS))
        return IP_ERR_PARAM;
    if (B < 0 || B > IP_MAX_B || T < 1 || G < 1) return IP_ERR_SHAPE;
    if (static_cast<long long>(B) * T > IP_LINEAR_MAX_FRAMES) return IP_ERR_SHAPE;
    if (K < 128 || K > IP_LINEAR_MAX_K || K % 128 != 0) return IP_ERR_SHAPE;
    if (N < 128 || N > IP_LINEAR_MAX_N || N % 128 != 0) return IP_ERR_SHAPE;
    if (y_layout == IP_LAYOUT_HEADS && N % (128 * G) != 0) return IP_ERR_SHAPE;
    if (y_layout == IP_LAYOUT_ROWS && G != 1) return IP_ERR_SHAPE;
    if (B == 0) return IP_OK;
    if (!x || !w || !m || !s || !y || !workspace) return IP_ERR_NULL;
    if (!aligned(x, 16) || !aligned(w, 16) || !aligned(y, 16) || !aligned(m, 4) ||
        !aligned(s, 4) || (bias && !aligned(bias, 4)) || !aligned(workspace, 256))
        return IP_ERR_ALIGN;
    if (workspace_bytes < 256) return IP_ERR_WORKSPACE;

    CUtensorMap tm_x, tm_w;
    const cuuint64_t kk = static_cast<cuuint64_t>(K), tt = static_cast<cuuint64_t>(T);
    bool okm;
    if (x_layout == IP_LAYOUT_ROWS) {
        // all frames of all utterances as one axis of B T rows
        const cuuint64_t dims[2] = {kk, tt * static_cast<cuuint64_t>(B)};
        const cuuint64_t strides[1] = {kk};
        okm = make_map(&tm_x, x, 2, dims, strides);
    } else {
        const cuuint64_t dims[4] = {128, tt, kk / 128, static_cast<cuuint64_t>(B)};
        const cuuint64_t strides[3] = {128, tt * 128, tt * kk};
        okm = make_map(&tm_x, x, 4, dims, strides);
    }
    const cuuint64_t wdims[2] = {kk, static_cast<cuuint64_t>(N)};
    const cuuint64_t wstrides[1] = {kk};
    if (!okm || !make_map(&tm_w, w, 2, wdims, wstrides)) return IP_ERR_CUDA;
    int rc = ensure_smem();
    if (rc != IP_OK) return rc;

    ipl::LinearParams prm;
    prm.bias = bias;
    prm.m = m;
    prm.s = s;
    prm.y = y;
    prm.B = B;
    prm.T = T;
    prm.K = K;
    prm.N = N;
    prm.heads_per_group = N / G / 128;
    prm.y_layout = y_layout;
    prm.x_layout = x_layout;
    prm.err = static_cast<int *>(workspace);
    prm.timeout_cycles = 4000000000ll;
    prm.ntn = N / ipl::BN;
    prm.tpu = (T + ipl::BM - 1) / ipl::BM;
    const long long frame_tiles = x_layout == IP_LAYOUT_ROWS
                                      ? (static_cast<long long>(B) * T + ipl::BM - 1) / ipl::BM
                                      : static_cast<long long>(B) * prm.tpu;
    prm.ntiles = static_cast<unsigned>(frame_tiles * prm.ntn);
    prm.magic_ntn = iph::div_magic(prm.ntn);
    prm.magic_T = iph::div_magic(T);
    prm.magic_tpu = iph::div_magic(prm.tpu);
    prm.sw_qc = sw ? sw->q_c : 0;
    prm.sw_qone = sw ? sw->q_one : 0;
    prm.sw_m = sw ? sw->m : 0;
    prm.sw_e = sw ? 31 + sw->s : 0;
    prm.res = res ? res->x : nullptr;
    prm.res_mx = res ? res->m_x : 0;
    prm.res_my = res ? res->m_y : 0;
    prm.res_s = res ? res->s : 0;
    const int nsm = sm_count();
    if (nsm <= 0) return IP_ERR_CUDA;
    const unsigned grid = prm.ntiles < static_cast<unsigned>(nsm) ? prm.ntiles
                                                                  : static_cast<unsigned>(nsm);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t lrc;
    if (epi == ipl::EPI_SWISH)
        lrc = iph::launch_pdl(ipl::linear_i8_kernel<ipl::EPI_SWISH>, dim3(grid), dim3(ipl::THREADS),
                              ipl::SMEM_LAUNCH, st, tm_x, tm_w, prm);
    else if (epi == ipl::EPI_GLU)
        lrc = iph::launch_pdl(ipl::linear_i8_kernel<ipl::EPI_GLU>, dim3(grid), dim3(ipl::THREADS),
                              ipl::SMEM_LAUNCH, st, tm_x, tm_w, prm);
    else if (epi == ipl::EPI_RES)
        lrc = iph::launch_pdl(ipl::linear_i8_kernel<ipl::EPI_RES>, dim3(grid), dim3(ipl::THREADS),
                              ipl::SMEM_LAUNCH, st, tm_x, tm_w, prm);
    else
        lrc = iph::launch_pdl(ipl::linear_i8_kernel<ipl::EPI_PLAIN>, dim3(grid), dim3(ipl::THREADS),
                              ipl::SMEM_LAUNCH, st, tm_x, tm_w, prm);
    if (lrc != cudaSuccess || cudaGetLastError() != cudaSuccess) return IP_ERR_CUDA;
    return IP_OK;
}

}  // namespace

extern "C" {

int ip_linear_i8(const int8_t *x, int x_layout, const int8_t *w, const int32_t *bias,
                 const int32_t *m, const int32_t *s, int B, int T, int K, int N, int G,
                 int8_t *y, int y_layout, void *workspace, size_t workspace_bytes,
                 ip_stream_t stream) {
    return linear_launch(x, x_layout, w, bias, m, s, nullptr, ipl::EPI_PLAIN, B, T, K, N, G, y,
                         y_layout, workspace, workspace_bytes, stream);
}

int ip_linear_swish_i8(const int8_t *x, const int8_t *w, const int32_t *bias, const int32_t *m,
                       const int32_t *s, const ip_swish_params *sw, int B, int T, int K, int N,
                       int8_t *y, void *workspace, size_t workspace_bytes, ip_stream_t stream) {
    if (!sw) return IP_ERR_NULL;
    const int rc = check_swish(sw);
    if (rc != IP_OK) return rc;
    return linear_launch(x, IP_LAYOUT_ROWS, w, bias, m, s, sw, ipl::EPI_SWISH, B, T, K, N, 1, y,
                         IP_LAYOUT_ROWS, workspace, workspace_bytes, stream);
}

int ip_linear_glu_i8(const int8_t *x, const int8_t *w, const int32_t *bias, const int32_t *m,
                     const int32_t *s, const ip_swish_params *glu, int B, int T, int K, int N,
                     int8_t *y, void *workspace, size_t workspace_bytes, ip_stream_t stream) {
    if (!glu) return IP_ERR_NULL;
    const int rc = check_swish(glu);
    if (rc != IP_OK) return rc;
    return linear_launch(x, IP_LAYOUT_ROWS, w, bias, m, s, glu, ipl::EPI_GLU, B, T, K, N, 1, y,
                         IP_LAYOUT_ROWS, workspace, workspace_bytes, stream);
}

int ip_linear_residual_i8(const int8_t *x, const int8_t *w, const int32_t *bias,
                          const int32_t *m, const int32_t *s, const int8_t *res, int32_t m_x,
                          int32_t m_y, int32_t s_r, int B, int T, int K, int N, int8_t *y,
                          void *workspace, size_t workspace_bytes, ip_stream_t stream) {
    if (m_x < 0 || m_y < 0 || s_r < 0 || s_r > 31) return IP_ERR_PARAM;
    if (B > 0 && !res) return IP_ERR_NULL;
    if (res && !aligned(res, 16)) return IP_ERR_ALIGN;
    if (res && y && res != y && B > 0 && T > 0 && N > 0) {
        // in place (res == y) is fine: every element is read by the thread
        // that then writes it; a partial overlap would race across CTAs
        const uintptr_t a = reinterpret_cast<uintptr_t>(res), b = reinterpret_cast<uintptr_t>(y);
        const uintptr_t n = static_cast<uintptr_t>(B) * static_cast<uintptr_t>(T) *
                            static_cast<uintptr_t>(N);
        if (a < b + n && b < a + n) return IP_ERR_PARAM;
    }
    const ResidualArg ra{res, m_x, m_y, s_r};
    return linear_launch(x, IP_LAYOUT_ROWS, w, bias, m, s, nullptr, ipl::EPI_RES, B, T, K, N, 1, y,
                         IP_LAYOUT_ROWS, workspace, workspace_bytes, stream, &ra);
}

int ip_linear_constants(double S_x, const double *S_w, const double *S_y, int N, int32_t *m,
                        int32_t *s) {
    if (!S_w || !S_y || !m || !s) return IP_ERR_NULL;
    if (N < 1 || !(S_x > 0.0) || !std::isfinite(S_x)) return IP_ERR_PARAM;
    for (int n = 0; n < N; ++n)   // every channel valid before any output is written
        if (!(S_w[n] > 0.0) || !std::isfinite(S_w[n]) || !(S_y[n] > 0.0) || !std::isfinite(S_y[n]))
            return IP_ERR_PARAM;
    for (int n = 0; n < N; ++n) {
        int32_t mm = 0, ss = 0;
        if (ip_dyadic_multiplier(S_x * S_w[n] / S_y[n], &mm, &ss) != IP_OK) return IP_ERR_PARAM;
    }
    for (int n = 0; n < N; ++n)
        ip_dyadic_multiplier(S_x * S_w[n] / S_y[n], &m[n], &s[n]);
    return IP_OK;
}

int ip_swish_params_from_scales(double S_z, double S_y, ip_swish_params *out) {
    if (!out) return IP_ERR_NULL;
    if (!(S_z > 0.0) || !(S_y > 0.0) || !std::isfinite(S_z) || !std::isfinite(S_y))
        return IP_ERR_PARAM;
    const double a = IP_SWISH_A, c = IP_SWISH_C;
    const double s_t = -a * (S_z / 2.0) * (S_z / 2.0);
    const double qc = std::floor(2.0 * c / S_z + 0.5);
    const double qone = std::floor(1.0 / s_t + 0.5);
    if (qc < 1.0 || qc >= 32768.0 || qone < 1.0 || qone >= 8388608.0) return IP_ERR_PARAM;
    ip_swish_params p;
    p.q_c = static_cast<int32_t>(qc);
    p.q_one = static_cast<int32_t>(qone);
    const int rc = ip_dyadic_multiplier(S_z * s_t / (2.0 * S_y), &p.m, &p.s);
    if (rc != IP_OK) return rc;
    if (check_swish(&p) != IP_OK) return IP_ERR_PARAM;
    *out = p;
    return IP_OK;
}

}  // extern "C"
