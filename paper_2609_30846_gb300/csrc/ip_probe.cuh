// Throughput probe of the integer warp MMA on this GPU: the measured INT8
// peak that the roofline of the attention kernel is reported against
// (sm_103a offers no integer tcgen05 MMA kind).  Each warp keeps eight
// independent m16n8k32 s8 x s8 -> s32 accumulators busy for `iters` rounds.
#pragma once

#include <stdint.h>

namespace ipk {

constexpr int PROBE_THREADS = 256;
constexpr int PROBE_CHAINS = 8;

__global__ void __launch_bounds__(PROBE_THREADS) int8_mma_probe_kernel(int *sink, uint32_t seed,
                                                                       int iters) {
    const uint32_t a0 = seed ^ threadIdx.x, a1 = seed * 3u + threadIdx.x, a2 = seed + 7u,
                   a3 = seed ^ 0x5a5a5a5au, b0 = seed * 5u, b1 = seed ^ 0x01020304u;
    int d[PROBE_CHAINS][4];
#pragma unroll
    for (int c = 0; c < PROBE_CHAINS; ++c) d[c][0] = d[c][1] = d[c][2] = d[c][3] = 0;
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int c = 0; c < PROBE_CHAINS; ++c)
            asm volatile(
                "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7},"
                " {%8,%9}, {%0,%1,%2,%3};"
                : "+r"(d[c][0]), "+r"(d[c][1]), "+r"(d[c][2]), "+r"(d[c][3])
                : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
    int s = 0;
#pragma unroll
    for (int c = 0; c < PROBE_CHAINS; ++c) s += d[c][0] + d[c][1] + d[c][2] + d[c][3];
    sink[blockIdx.x * PROBE_THREADS + threadIdx.x] = s;
}

// Probe of the two integer pipes at once: in each block the first
// `mma_warps` warps run four m16n8k32 MMA chains for `iters` rounds, the
// others eight dp4a chains for 4 x `iters` rounds of four (about the same
// time per warp), so that the launch time shows whether the tensor pipe and
// the dp4a pipe work concurrently.
constexpr int MIX_MMA_CHAINS = 4;
constexpr int MIX_DP4A_CHAINS = 8;

__global__ void __launch_bounds__(PROBE_THREADS) int8_mix_probe_kernel(int *sink, uint32_t seed,
                                                                      int iters, int mma_warps) {
    const int warp = threadIdx.x >> 5;
    int s = 0;
    if (warp < mma_warps) {
        const uint32_t a0 = seed ^ threadIdx.x, a1 = seed * 3u + threadIdx.x, a2 = seed + 7u,
                       a3 = seed ^ 0x5a5a5a5au, b0 = seed * 5u, b1 = seed ^ 0x01020304u;
        int d[MIX_MMA_CHAINS][4];
#pragma unroll
        for (int c = 0; c < MIX_MMA_CHAINS; ++c) d[c][0] = d[c][1] = d[c][2] = d[c][3] = 0;
        for (int it = 0; it < iters; ++it) {
#pragma unroll
            for (int c = 0; c < MIX_MMA_CHAINS; ++c)
                asm volatile(
                    "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7},"
                    " {%8,%9}, {%0,%1,%2,%3};"
                    : "+r"(d[c][0]), "+r"(d[c][1]), "+r"(d[c][2]), "+r"(d[c][3])
                    : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
        }
#pragma unroll
        for (int c = 0; c < MIX_MMA_CHAINS; ++c) s += d[c][0] + d[c][1] + d[c][2] + d[c][3];
    } else {
        const uint32_t y = seed * 7u + threadIdx.x;
        uint32_t x[MIX_DP4A_CHAINS];
        int acc[MIX_DP4A_CHAINS];
#pragma unroll
        for (int c = 0; c < MIX_DP4A_CHAINS; ++c) {
            x[c] = seed + c * 0x01010101u + threadIdx.x;
            acc[c] = c;
        }
        for (int it = 0; it < 4 * iters; ++it) {
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int c = 0; c < MIX_DP4A_CHAINS; ++c)
                    asm volatile("dp4a.s32.s32 %0, %1, %2, %0;" : "+r"(acc[c]) : "r"(x[c]), "r"(y));
        }
#pragma unroll
        for (int c = 0; c < MIX_DP4A_CHAINS; ++c) s += acc[c];
    }
    sink[blockIdx.x * PROBE_THREADS + threadIdx.x] = s;
}

}  // namespace ipk
