// Device primitives shared by the kernels of this library (sm_103a):
// shared-memory addressing and accesses, mbarriers with bounded waits, TMA
// tile loads, ldmatrix and the integer warp MMA.  Integer arithmetic only.
#pragma once

#include <cuda.h>
#include <stdint.h>

namespace ipk {

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Hands a shared-memory stage that this warp has read with generic loads
// (ldmatrix, ld.shared) back to the warp that refills it by TMA: the proxy
// fence orders those reads before the async-proxy writes of the refill
// (without it a refill could land before a read was performed), then lane 0
// arrives on `bar`.
__device__ __forceinline__ void release_stage(uint32_t bar, int lane) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    __syncwarp();
    if (lane == 0) mbar_arrive(bar);
}

// Waits for the phase of `parity` to complete; gives up after `limit` clock
// cycles and returns false.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, long long limit) {
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity)) {
        if (clock64() - t0 > limit) return false;
    }
    return true;
}

// Warp-wide wait: every lane polls, then the warp agrees on the outcome, so
// that a timeout takes all lanes down the same path.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, long long limit) {
    const bool ok = mbar_wait(bar, parity, limit);
    return __all_sync(0xffffffffu, ok) != 0;
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, int c0, int c1,
                                            int c2, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int c0, int c1,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, int c0, int c1,
                                            int c2, int c3, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}

// floor(n / d) for 0 <= n < 2^32 and 1 <= d < 2^32 without a division
// instruction: M = floor(2^64 / d) + 1 (computed once on the host; M = 0
// stands for d = 1).  With e = M - 2^64/d in (0, 1], n M / 2^64 lies in
// [n/d, n/d + n/2^64), and n/2^64 < 1/d <= 1 - frac(n/d) when frac(n/d) > 0
// (n d < 2^64), so the floor is floor(n / d).
__device__ __forceinline__ uint32_t udiv_magic(uint32_t n, unsigned long long magic) {
    return magic == 0 ? n : static_cast<uint32_t>(__umul64hi(static_cast<unsigned long long>(n), magic));
}

// Barrier `id` (1..15) over the first `count` threads of the CTA.
__device__ __forceinline__ void named_sync(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

// Four 8x8 matrices of 16-bit elements, transposed: thread l receives, of
// matrix i, the elements (2 (l & 3), l >> 2) and (2 (l & 3) + 1, l >> 2).
__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t &r0, uint32_t &r1,
                                              uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(addr));
    return v;
}

__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}

__device__ __forceinline__ int2 lds64(uint32_t addr) {
    int2 v;
    asm volatile("ld.shared.v2.s32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr));
    return v;
}

__device__ __forceinline__ void sts32(uint32_t addr, uint32_t v) {
    asm volatile("st.shared.u32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}

__device__ __forceinline__ void sts64(uint32_t addr, int x, int y) {
    asm volatile("st.shared.v2.s32 [%0], {%1,%2};" ::"r"(addr), "r"(x), "r"(y) : "memory");
}

__device__ __forceinline__ void sts128(uint32_t addr, uint32_t x, uint32_t y, uint32_t z,
                                       uint32_t w) {
    asm volatile("st.shared.v4.u32 [%0], {%1,%2,%3,%4};" ::"r"(addr), "r"(x), "r"(y), "r"(z),
                 "r"(w)
                 : "memory");
}

// Global memory cached in L2 only (.cg): the long-sequence score slices,
// written and read back by the same thread.
__device__ __forceinline__ void stg128_cg(void *addr, uint32_t x, uint32_t y, uint32_t z,
                                          uint32_t w) {
    asm volatile("st.global.cg.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(addr), "r"(x), "r"(y), "r"(z),
                 "r"(w)
                 : "memory");
}

__device__ __forceinline__ uint4 ldg128_cg(const void *addr) {
    uint4 v;
    asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(addr)
                 : "memory");
    return v;
}

__device__ __forceinline__ void stg64_cg(void *addr, int x, int y) {
    asm volatile("st.global.cg.v2.s32 [%0], {%1,%2};" ::"l"(addr), "r"(x), "r"(y) : "memory");
}

__device__ __forceinline__ int2 ldg64_cg(const void *addr) {
    int2 v;
    asm volatile("ld.global.cg.v2.s32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(addr) : "memory");
    return v;
}

// D += A B with A 16x32 s8 (row), B 32x8 s8 (col), D 16x8 s32.
__device__ __forceinline__ void mma_s8s8(int (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm("mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7},"
        " {%8,%9}, {%0,%1,%2,%3};"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// D += A B with A 16x32 u8 (row), B 32x8 s8 (col), D 16x8 s32.
__device__ __forceinline__ void mma_u8s8(int (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm("mma.sync.aligned.m16n8k32.row.col.s32.u8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7},"
        " {%8,%9}, {%0,%1,%2,%3};"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// D += A B with A 16x16 u8 (row), B 16x8 s8 (col), D 16x8 s32.
__device__ __forceinline__ void mma_u8s8_k16(int (&d)[4], uint32_t a0, uint32_t a1, uint32_t b0) {
    asm("mma.sync.aligned.m16n8k16.row.col.s32.u8.s8.s32 {%0,%1,%2,%3}, {%4,%5}, {%6},"
        " {%0,%1,%2,%3};"
        : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
        : "r"(a0), "r"(a1), "r"(b0));
}

// Programmatic dependent launch: let the next launch on the stream be
// scheduled now (its CTAs take the SM slots this grid frees), and wait for
// the grid before this one on the stream to complete, with its memory
// visible, before the first global access.
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Offset of the 16-byte chunk `chunk` of row `row` in a tile written by TMA
// with the 128-byte swizzle (rows of 128 bytes, 1024-byte aligned).
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
    return static_cast<uint32_t>(row * 128 + (((chunk ^ row) & 7) << 4));
}

__device__ __forceinline__ int clamp127(long long x) {
    return x > 127 ? 127 : (x < -127 ? -127 : static_cast<int>(x));
}

// Residual addition of Eqs. 1-4 for one element: round((m_x x + m_y y) /
// 2^(31+s)) clamped to [-127, 127]; |m_x x + m_y y| < 2^39, so the quotient
// by 2^31 is a 32-bit value (funnel shift), then a shift by s.
__device__ __forceinline__ int residual_one(int x, int y, int m_x, int m_y, int s) {
    const long long v = static_cast<long long>(m_x) * x + static_cast<long long>(m_y) * y +
                        (1ll << (30 + s));
    const int h = static_cast<int>(__funnelshift_r(static_cast<uint32_t>(v),
                                                   static_cast<uint32_t>(v >> 32), 31));
    return clamp127(h >> s);
}

// Residual addition of four packed int8 pairs (byte e of x with byte e of y).
__device__ __forceinline__ uint32_t residual4(uint32_t x, uint32_t y, int m_x, int m_y, int s) {
    uint32_t w = 0;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const int xa = static_cast<int>(static_cast<int8_t>((x >> (8 * e)) & 0xffu));
        const int yb = static_cast<int>(static_cast<int8_t>((y >> (8 * e)) & 0xffu));
        w |= (static_cast<uint32_t>(residual_one(xa, yb, m_x, m_y, s)) & 0xffu) << (8 * e);
    }
    return w;
}

// (c << 16) | (sat8(a) << 8) | sat8(b): two int32 values saturated to
// [-128, 127] and packed below the low half of c (cvt.pack.sat).
__device__ __forceinline__ uint32_t pack_sat2(int a, int b, uint32_t c) {
    uint32_t w;
    asm("cvt.pack.sat.s8.s32.b32 %0, %1, %2, %3;" : "=r"(w) : "r"(a), "r"(b), "r"(c));
    return w;
}

// Bytes [y0, y1, y2, y3] of four int32 values, each saturated to [-128, 127].
__device__ __forceinline__ uint32_t pack_sat4(int y0, int y1, int y2, int y3) {
    return pack_sat2(y1, y0, pack_sat2(y3, y2, 0u));
}

// Sign-extended byte e (0..3) of w: one prmt, byte e in the low byte and
// its sign bit replicated in the three above (selector bit 3).
__device__ __forceinline__ int sbyte(uint32_t w, int e) {
    const uint32_t s = 0x8u | static_cast<uint32_t>(e);
    const uint32_t sel = (s << 12) | (s << 8) | (s << 4) | static_cast<uint32_t>(e);
    uint32_t r;
    asm("prmt.b32 %0, %1, 0, %2;" : "=r"(r) : "r"(w), "r"(sel));
    return static_cast<int>(r);
}

}  // namespace ipk
