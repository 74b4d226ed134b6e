// Host side of the integer LayerNorm of the C ABI (include/ip_mhsa.h):
// argument validation, the launch, and the offline per-channel constants.
// Device code: ip_norm_kernels.cuh.
#include "ip_mhsa.h"
#include "ip_norm_kernels.cuh"
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

// CTAs of the C-segment kernel on the whole GPU: one per SM, so that its
// eight warps take two or more batches each and load the next batch's rows
// while they normalise the current one (cached; 0 if one does not fit).
template <int C>
long long resident(int nsm) {
    static int per_sm[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::lock_guard<std::mutex> lock(g_mu);
    if (per_sm[dev] == 0) {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, ipn::layernorm_i8_kernel<C>,
                                                          ipn::THREADS, C * 8192) != cudaSuccess ||
            n < 1)
            return 0;
        per_sm[dev] = 1;
    }
    return static_cast<long long>(per_sm[dev]) * nsm;
}

template <int C>
int launch(const ipn::NormParams &prm, int nsm, cudaStream_t st) {
    // every resident CTA gets batches (dealt warp-major), up to one per CTA
    const long long batches = (prm.rows + ipn::NB - 1) / ipn::NB;
    const long long cap = resident<C>(nsm);
    if (cap <= 0) return IP_ERR_CUDA;
    const unsigned grid = static_cast<unsigned>(batches < cap ? batches : cap);
    if (iph::launch_pdl(ipn::layernorm_i8_kernel<C>, dim3(grid), dim3(ipn::THREADS), C * 8192, st,
                        prm) != cudaSuccess)
        return IP_ERR_CUDA;
    return cudaGetLastError() == cudaSuccess ? IP_OK : IP_ERR_CUDA;
}

}  // namespace

extern "C" {

int ip_layernorm_i8(const int8_t *x, long long rows, int d, long long eps_c, const int32_t *M,
                    const long long *B, const int32_t *E, int8_t *y, void *workspace,
                    size_t workspace_bytes, ip_stream_t stream) {
    if (rows < 0 || rows > IP_NORM_MAX_ROWS) return IP_ERR_SHAPE;
    if (d != 512 && d != 1024 && d != 1536 && d != 2048) return IP_ERR_UNSUPPORTED;
    if (eps_c < 0 || eps_c > (1ll << 40)) return IP_ERR_PARAM;
    if (rows == 0) return IP_OK;
    if (!x || !M || !B || !E || !y || !workspace) return IP_ERR_NULL;
    if (!aligned(x, 16) || !aligned(y, 16) || !aligned(M, 4) || !aligned(E, 4) ||
        !aligned(B, 8) || !aligned(workspace, 256))
        return IP_ERR_ALIGN;
    if (workspace_bytes < 256) return IP_ERR_WORKSPACE;
    const int nsm = sm_count();
    if (nsm <= 0) return IP_ERR_CUDA;
    ipn::NormParams prm;
    prm.x = x;
    prm.y = y;
    prm.rows = rows;
    prm.eps_c = eps_c;
    prm.M = M;
    prm.B = B;
    prm.E = E;
    prm.err = static_cast<int *>(workspace);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    switch (d / 512) {
        case 1: return launch<1>(prm, nsm, st);
        case 2: return launch<2>(prm, nsm, st);
        case 3: return launch<3>(prm, nsm, st);
        default: return launch<4>(prm, nsm, st);
    }
}

int ip_layernorm_constants(double S_x, const double *gamma, const double *beta, int d,
                           double S_y, double eps, long long *eps_c, int32_t *M, long long *B,
                           int32_t *E) {
    if (!gamma || !beta || !eps_c || !M || !B || !E) return IP_ERR_NULL;
    if (d < 1 || !(S_x > 0.0) || !(S_y > 0.0) || !(eps >= 0.0) || !std::isfinite(S_x) ||
        !std::isfinite(S_y) || !std::isfinite(eps))
        return IP_ERR_PARAM;
    for (int i = 0; i < d; ++i) {
        const double g = gamma[i];
        if (!std::isfinite(g) || !std::isfinite(beta[i])) return IP_ERR_PARAM;
        int32_t m = 0, s = 0;
        if (g != 0.0) {
            const int rc = ip_dyadic_multiplier(std::fabs(g) * std::ldexp(1.0, -15) / S_y, &m, &s);
            if (rc != IP_OK) return rc;
        }
        M[i] = g > 0.0 ? m : -m;
        E[i] = 31 + s;
        const double b = std::floor(beta[i] / S_y * std::ldexp(1.0, E[i]) + 0.5);
        if (!(std::fabs(b) < std::ldexp(1.0, 60))) return IP_ERR_PARAM;
        B[i] = static_cast<long long>(b);
    }
    const double ec = std::floor(eps * static_cast<double>(d) * d / (S_x * S_x) + 0.5);
    if (!(ec <= std::ldexp(1.0, 40))) return IP_ERR_PARAM;
    *eps_c = static_cast<long long>(ec);
    return IP_OK;
}

}  // extern "C"
