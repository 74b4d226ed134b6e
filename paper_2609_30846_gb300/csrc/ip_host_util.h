// Host-side constants of the device helpers (compiled into the host code of
// the library only).
#pragma once

#include <cuda_runtime.h>

namespace iph {

// Launches `kernel` with programmatic dependent launch allowed: it may be
// scheduled while the kernel before it on `stream` finishes (every kernel of
// this library waits for that grid before its first global access).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

// The constant of udiv_magic (device side) for d: floor(2^64 / d) + 1, or 0
// for d = 1, so that floor(n / d) = the high word of n times it.
inline unsigned long long div_magic(unsigned long long d) {
    if (d <= 1) return 0;
    const unsigned __int128 one = static_cast<unsigned __int128>(1) << 64;
    return static_cast<unsigned long long>(one / d) + 1;
}

}  // namespace iph
