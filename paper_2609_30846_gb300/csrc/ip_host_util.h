// Host-side constants of the device helpers (compiled into the host code of
// the library only).
#pragma once

namespace iph {

// The constant of udiv_magic (device side) for d: floor(2^64 / d) + 1, or 0
// for d = 1, so that floor(n / d) = the high word of n times it.
inline unsigned long long div_magic(unsigned long long d) {
    if (d <= 1) return 0;
    const unsigned __int128 one = static_cast<unsigned __int128>(1) << 64;
    return static_cast<unsigned long long>(one / d) + 1;
}

}  // namespace iph
