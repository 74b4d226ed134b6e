// Host side of the C ABI declared in include/ip_mhsa.h: argument
// validation, tensor-map encoding for the TMA loads, workspace layout and
// kernel launches.  The device code lives in ip_mhsa_kernels.cuh.
#include "ip_mhsa.h"
#include "ip_mhsa_kernels.cuh"
#include "ip_probe.cuh"
#include "ip_host_util.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <math.h>
#include <mutex>
#include <string.h>

namespace {

constexpr size_t WS_HEADER = 256;          // error word and padding
constexpr long long DEFAULT_TIMEOUT = 4000000000ll;   // ~2 s at 2 GHz
long long g_timeout_cycles = DEFAULT_TIMEOUT;
int g_stall_injection = 0;
int g_split_mode = -1;   // -1 planned, 0 never, 1 / 2: every tile in halves / quarters (test hook)
int g_wide_sums = 0;     // 1: general softmax arithmetic always (test hook)
// the default workspace registered by ip_set_workspace
std::mutex g_ws_mu;
void *g_ws_ptr = nullptr;
size_t g_ws_bytes = 0;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// The workspace holds the device error word of the calls that use it (byte
// 0) and the attention kernel's item counters (bytes 64 and 128), which the
// last CTA of every launch returns to zero.
size_t ws_bytes() { return WS_HEADER; }

int check_shape(int B, int H, int T, int dh) {
    if (dh != IP_DH) return IP_ERR_UNSUPPORTED;
    if (B < 0 || H < 0 || T < 1 || T > IP_MAX_T) return IP_ERR_SHAPE;
    if (B > IP_MAX_B || H > IP_MAX_H) return IP_ERR_SHAPE;   // grid y, z limits
    return IP_OK;
}

int check_softmax(const ip_isoftmax_params *sm) {
    if (sm->q_ln2 < 1 || sm->q_b < 0 || sm->q_c < 0) return IP_ERR_PARAM;
    const long long t0 = sm->q_b, t1 = static_cast<long long>(sm->q_b) - sm->q_ln2 + 1;
    const long long l0 = t0 * t0 + sm->q_c, l1 = t1 * t1 + sm->q_c;
    if (l0 < 2 || l0 >= (1ll << 31) || l1 >= (1ll << 31)) return IP_ERR_PARAM;
    return IP_OK;
}

// cuTensorMapEncodeTiled through the runtime's driver entry point.
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

// 3-D int8 map [d2][d1][128] with a box of 128 x rows x 1 and the 128-byte
// swizzle; rows outside [0, d1) read as zero.
bool make_map(CUtensorMap *m, const void *base, unsigned long long d1, unsigned long long d2,
              unsigned rows) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[3] = {static_cast<cuuint64_t>(IP_DH), d1, d2};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(IP_DH), d1 * IP_DH};
    const cuuint32_t box[3] = {static_cast<cuuint32_t>(IP_DH), rows, 1};
    const cuuint32_t estride[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 3, const_cast<void *>(base), dims, strides, box,
              estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Encoded maps of recent calls, keyed by base pointer and shape (a map
// depends on nothing else), so that calls on the same buffers skip the
// encoding; a small table with round-robin replacement.
struct MapEntry {
    const void *base;
    unsigned long long d1, d2;
    unsigned rows;
    bool used;
    CUtensorMap map;
};
constexpr int MAP_CACHE = 32;
std::mutex g_map_mu;
MapEntry g_maps[MAP_CACHE];
int g_map_next = 0;

bool cached_map(CUtensorMap *m, const void *base, unsigned long long d1, unsigned long long d2,
                unsigned rows) {
    std::lock_guard<std::mutex> lock(g_map_mu);
    for (const MapEntry &e : g_maps)
        if (e.used && e.base == base && e.d1 == d1 && e.d2 == d2 && e.rows == rows) {
            *m = e.map;
            return true;
        }
    if (!make_map(m, base, d1, d2, rows)) return false;
    MapEntry &e = g_maps[g_map_next];
    g_map_next = (g_map_next + 1) % MAP_CACHE;
    e.base = base;
    e.d1 = d1;
    e.d2 = d2;
    e.rows = rows;
    e.used = true;
    e.map = *m;
    return true;
}

// The fused kernel in its two forms: int8 scores kept in shared memory, or
// (gs, long sequences) in the caller's workspace.
using FusedKernel = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap,
                             const CUtensorMap, const ipk::FusedParams);
FusedKernel fused_kernel(bool gs) {
    return gs ? ipk::relpos_mhsa_fused_kernel<true> : ipk::relpos_mhsa_fused_kernel<false>;
}

std::mutex g_attr_mu;
int g_attr_smem[2][64] = {{0}};

int ensure_smem(bool gs, int bytes) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IP_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_attr_mu);
    if (g_attr_smem[gs][dev] >= bytes) return IP_OK;
    if (cudaFuncSetAttribute(fused_kernel(gs), cudaFuncAttributeMaxDynamicSharedMemorySize,
                             bytes) != cudaSuccess)
        return IP_ERR_CUDA;
    g_attr_smem[gs][dev] = bytes;
    return IP_OK;
}

// CTAs of the fused kernel resident on the whole GPU at once (its SMs x the
// CTAs an SM holds at this shared-memory size), cached for the last query
// of each form.
std::mutex g_occ_mu;
int g_occ_dev[2] = {-1, -1}, g_occ_smem[2] = {-1, -1}, g_occ_slots[2] = {0, 0};

int resident_ctas(bool gs, int smem) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    std::lock_guard<std::mutex> lock(g_occ_mu);
    if (dev == g_occ_dev[gs] && smem == g_occ_smem[gs]) return g_occ_slots[gs];
    int nsm = 0, per_sm = 0;
    if (ensure_smem(gs, smem) != IP_OK ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fused_kernel(gs), ipk::NTHREADS,
                                                      smem) != cudaSuccess)
        return 0;
    g_occ_dev[gs] = dev;
    g_occ_smem[gs] = smem;
    g_occ_slots[gs] = nsm * per_sm;
    return g_occ_slots[gs];
}

// Sequences longer than this keep their scores in the workspace when it
// has room: the shared-memory slices of T <= 384 (6 chunks) let two CTAs
// share an SM, longer ones only one.
constexpr int GS_MIN_T = 6 * ipk::NK + 1;

int fused_smem(int T, bool gs) {
    return ipk::smem_layout((T + ipk::NK - 1) / ipk::NK, gs).total + 1024;
}

// Bytes of the workspace's score region for T (0 when the scores stay in
// shared memory or the device cannot be queried): one slice of nchunk KB
// per consumer warp of every resident CTA.
size_t gs_scores_bytes(int T) {
    if (T < GS_MIN_T) return 0;
    const int slots = resident_ctas(true, fused_smem(T, true));
    if (slots < 1) return 0;
    return static_cast<size_t>(slots) * ipk::NCWARPS *
           static_cast<size_t>((T + ipk::NK - 1) / ipk::NK) * ipk::CHUNK_SCORE_BYTES;
}

// Work items of the persistent kernel.  The N whole tiles run on G resident
// CTAs in rounds; when the last round is at most a quarter full (r = N mod G
// tiles, 4 r <= G) its r tiles become 4 r quarters of 16 rows, when at most
// half full (2 r <= G) 2 r halves of 32 rows, whose warps split the keys of
// every chunk, so that the last round takes a fraction of a tile's time.
struct ItemPlan {
    uint32_t nwhole = 0, nitems = 0, grid = 0;
    int split_log2 = 1;
};

ItemPlan plan_items(long long N, int slots) {
    ItemPlan ip;
    long long nwhole = N, nitems = N;
    if (g_split_mode == 1 || g_split_mode == 2) {
        ip.split_log2 = g_split_mode;
        nwhole = 0;
        nitems = N << g_split_mode;
    } else if (g_split_mode < 0 && slots > 0) {
        const long long r = N % slots;
        if (r > 0 && 4 * r <= slots) {
            ip.split_log2 = 2;
            nwhole = N - r;
            nitems = N + 3 * r;
        } else if (r > 0 && 2 * r <= slots) {
            nwhole = N - r;
            nitems = N + r;
        }
    }
    ip.nwhole = static_cast<uint32_t>(nwhole);
    ip.nitems = static_cast<uint32_t>(nitems);
    ip.grid = static_cast<uint32_t>(nitems < slots ? nitems : slots);
    return ip;
}

}  // namespace

extern "C" {

size_t ip_relpos_mhsa_workspace_bytes(int B, int H, int T, int dh) {
    if (check_shape(B, H, T, dh) != IP_OK) return 0;
    return ws_bytes() + gs_scores_bytes(T);
}

int ip_relpos_mhsa_i8(const int8_t *q, const int8_t *k, const int8_t *v, const int8_t *p,
                      const int8_t *u, const int8_t *v_bias, const int32_t *multipliers,
                      const int32_t *shifts, const ip_isoftmax_params *sm,
                      const int32_t *lengths, int B, int H, int T, int dh, int8_t *out,
                      void *workspace, size_t workspace_bytes, ip_stream_t stream) {
    return ip_relpos_mhsa_i8_ex(q, k, v, p, u, v_bias, multipliers, shifts, sm, lengths, B, H, T,
                                dh, out, IP_LAYOUT_HEADS, workspace, workspace_bytes, stream);
}

int ip_relpos_mhsa_i8_ex(const int8_t *q, const int8_t *k, const int8_t *v, const int8_t *p,
                         const int8_t *u, const int8_t *v_bias, const int32_t *multipliers,
                         const int32_t *shifts, const ip_isoftmax_params *sm,
                         const int32_t *lengths, int B, int H, int T, int dh, int8_t *out,
                         int out_layout, void *workspace, size_t workspace_bytes,
                         ip_stream_t stream) {
    if (out_layout != IP_LAYOUT_ROWS && out_layout != IP_LAYOUT_HEADS) return IP_ERR_PARAM;
    int rc = check_shape(B, H, T, dh);
    if (rc != IP_OK) return rc;
    if (B == 0 || H == 0) return IP_OK;   // empty problem: nothing to read or write
    if (workspace == nullptr) {
        std::lock_guard<std::mutex> lock(g_ws_mu);
        workspace = g_ws_ptr;
        workspace_bytes = g_ws_bytes;
    }
    if (!q || !k || !v || !p || !u || !v_bias || !multipliers || !shifts || !sm || !out ||
        !workspace)
        return IP_ERR_NULL;
    for (const void *ptr : {static_cast<const void *>(q), static_cast<const void *>(k),
                            static_cast<const void *>(v), static_cast<const void *>(p),
                            static_cast<const void *>(u), static_cast<const void *>(v_bias),
                            static_cast<const void *>(out)})
        if (!aligned(ptr, 16)) return IP_ERR_ALIGN;
    if (!aligned(workspace, 256)) return IP_ERR_ALIGN;
    if (lengths && !aligned(lengths, 4)) return IP_ERR_ALIGN;
    for (int c = 0; c < 3; ++c)
        if (multipliers[c] < 0) return IP_ERR_PARAM;
    for (int c = 0; c < 2; ++c)
        if (shifts[c] < 0 || shifts[c] > 31) return IP_ERR_PARAM;
    rc = check_softmax(sm);
    if (rc != IP_OK) return rc;
    if (workspace_bytes < ws_bytes()) return IP_ERR_WORKSPACE;

    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    int *err = static_cast<int *>(workspace);

    CUtensorMap tm_q, tm_k, tm_v, tm_p;
    const unsigned long long bh = static_cast<unsigned long long>(B) * H;
    if (!cached_map(&tm_q, q, T, bh, ipk::MROWS) || !cached_map(&tm_k, k, T, bh, ipk::NK) ||
        !cached_map(&tm_v, v, T, bh, ipk::NK) || !cached_map(&tm_p, p, 2ull * T - 1, H, ipk::BAND_ROWS))
        return IP_ERR_CUDA;

    const int ntiles = (T + ipk::MROWS - 1) / ipk::MROWS;
    const long long N = static_cast<long long>(B) * H * ntiles;   // whole tiles
    if (N >= IP_MAX_TILES) return IP_ERR_SHAPE;   // item indices stay below 2^31
    const int nchunk_max = (T + ipk::NK - 1) / ipk::NK;
    // long sequences: scores in the workspace when it holds their region
    const size_t gsb = gs_scores_bytes(T);
    const bool gs = gsb > 0 && workspace_bytes >= ws_bytes() + gsb;
    const int smem = fused_smem(T, gs);
    rc = ensure_smem(gs, smem);
    if (rc != IP_OK) return rc;

    ipk::FusedParams prm;
    prm.u = u;
    prm.vb = v_bias;
    prm.out = out;
    prm.lengths = lengths;
    prm.err = err;
    prm.sched = reinterpret_cast<unsigned int *>(static_cast<char *>(workspace) + 64);
    prm.B = B;
    prm.H = H;
    prm.T = T;
    prm.nchunk_max = nchunk_max;
    prm.m_c = multipliers[0];
    prm.m_p = multipliers[1];
    prm.m_o = multipliers[2];
    prm.sh_s = 31 + shifts[0];
    prm.sh_o = 31 + shifts[1];
    prm.q_ln2 = sm->q_ln2;
    prm.q_b = sm->q_b;
    prm.q_c = sm->q_c;
    prm.ln2_magic = iph::div_magic(static_cast<unsigned long long>(sm->q_ln2));
    // exp(0) = q_b^2 + q_c bounds every table entry; a thread adds 16 of
    // them per row and chunk
    const unsigned long long e0 =
        static_cast<unsigned long long>(sm->q_b) * sm->q_b + static_cast<unsigned long long>(sm->q_c);
    prm.sum32 =
        !g_wide_sums && e0 * 16ull * static_cast<unsigned long long>(nchunk_max) < (1ull << 32) ? 1 : 0;
    // a row's sum includes exp(0) (its maximum's own term)
    prm.f24 = !g_wide_sums && e0 > 256ull ? 1 : 0;
    prm.timeout_cycles = g_timeout_cycles;
    prm.stall_injection = g_stall_injection;
    const int slots = resident_ctas(gs, smem);
    if (slots < 1) return IP_ERR_CUDA;
    const ItemPlan ip = plan_items(N, slots);
    prm.ntiles = ntiles;
    prm.tiles_magic = iph::div_magic(static_cast<unsigned long long>(ntiles));
    prm.heads_magic = iph::div_magic(static_cast<unsigned long long>(H));
    prm.nwhole = ip.nwhole;
    prm.split_log2 = ip.split_log2;
    prm.nitems = ip.nitems;
    prm.out_rows = out_layout == IP_LAYOUT_ROWS ? 1 : 0;
    prm.gscores = gs ? static_cast<uint8_t *>(workspace) + ws_bytes() : nullptr;
    // Programmatic dependent launch: this grid may be scheduled while the
    // kernel before it on the stream finishes (the kernel waits for that
    // grid before its first global access, so the order of the two is kept).
    if (iph::launch_pdl(fused_kernel(gs), dim3(ip.grid), dim3(ipk::NTHREADS),
                        static_cast<size_t>(smem), st, tm_q, tm_k, tm_v, tm_p, prm) != cudaSuccess)
        return IP_ERR_CUDA;
    if (cudaGetLastError() != cudaSuccess) return IP_ERR_CUDA;
    return IP_OK;
}

int ip_set_workspace(void *ptr, size_t bytes) {
    if (ptr != nullptr) {
        if (!aligned(ptr, 256)) return IP_ERR_ALIGN;
        if (bytes < ws_bytes()) return IP_ERR_WORKSPACE;
    }
    std::lock_guard<std::mutex> lock(g_ws_mu);
    g_ws_ptr = ptr;
    g_ws_bytes = ptr != nullptr ? bytes : 0;
    return IP_OK;
}

int ip_relpos_mhsa_status(const void *workspace, ip_stream_t stream) {
    if (workspace == nullptr) {
        std::lock_guard<std::mutex> lock(g_ws_mu);
        workspace = g_ws_ptr;
    }
    if (!workspace) return IP_ERR_NULL;
    int word = 0;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(&word, workspace, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess)
        return IP_ERR_CUDA;
    if (cudaMemsetAsync(const_cast<void *>(workspace), 0, ws_bytes(), st) != cudaSuccess)
        return IP_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return IP_ERR_CUDA;
    if (word & 15) return IP_ERR_TIMEOUT;   // a bounded barrier wait ran out
    return word == 0 ? IP_OK : IP_ERR_PARAM;   // a device-side constant out of its domain
}

size_t ip_relpos_mhsa_host_arena_bytes(int B, int H, int T, int dh) {
    if (check_shape(B, H, T, dh) != IP_OK) return 0;
    const size_t act = align_up(static_cast<size_t>(B) * H * T * dh, 256);
    const size_t pb = align_up(static_cast<size_t>(H) * (2ull * T - 1) * dh, 256);
    const size_t bias = align_up(static_cast<size_t>(H) * dh, 256);
    const size_t lens = align_up(4ull * (B > 0 ? B : 1), 256);
    return 4 * act + pb + 2 * bias + lens + ws_bytes() + gs_scores_bytes(T);
}

namespace {

// Arena of the host-buffer entry points: inputs, output, lengths and the
// status word, each 256-byte aligned, in this order.
struct HostArena {
    int8_t *q, *k, *v, *out, *p, *u, *vb;
    int32_t *len;
    void *ws;
};

HostArena host_arena(void *arena, int B, int H, int T, int dh) {
    const size_t nact = static_cast<size_t>(B) * H * T * dh;
    const size_t np = static_cast<size_t>(H) * (2ull * T - 1) * dh;
    const size_t nb = static_cast<size_t>(H) * dh;
    uint8_t *a = static_cast<uint8_t *>(arena);
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t *r = a + off;
        off += align_up(bytes, 256);
        return r;
    };
    HostArena h;
    h.q = reinterpret_cast<int8_t *>(take(nact));
    h.k = reinterpret_cast<int8_t *>(take(nact));
    h.v = reinterpret_cast<int8_t *>(take(nact));
    h.out = reinterpret_cast<int8_t *>(take(nact));
    h.p = reinterpret_cast<int8_t *>(take(np));
    h.u = reinterpret_cast<int8_t *>(take(nb));
    h.vb = reinterpret_cast<int8_t *>(take(nb));
    h.len = reinterpret_cast<int32_t *>(take(4ull * (B > 0 ? B : 1)));
    h.ws = take(ws_bytes() + gs_scores_bytes(T));
    return h;
}

// Enqueues zeroing of the status word, the uploads, the kernel and the
// download on `stream`; nothing waits.
int host_enqueue(const int8_t *q, const int8_t *k, const int8_t *v, const int8_t *p,
                 const int8_t *u, const int8_t *v_bias, const int32_t *multipliers,
                 const int32_t *shifts, const ip_isoftmax_params *sm, const int32_t *lengths,
                 int B, int H, int T, int dh, int8_t *out, void *arena, size_t arena_bytes,
                 ip_stream_t stream, HostArena *where) {
    int rc = check_shape(B, H, T, dh);
    if (rc != IP_OK) return rc;
    if (B == 0 || H == 0) return IP_OK;
    if (!q || !k || !v || !p || !u || !v_bias || !out || !arena) return IP_ERR_NULL;
    if (!aligned(arena, 256)) return IP_ERR_ALIGN;
    if (arena_bytes < ip_relpos_mhsa_host_arena_bytes(B, H, T, dh)) return IP_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t nact = static_cast<size_t>(B) * H * T * dh;
    const size_t np = static_cast<size_t>(H) * (2ull * T - 1) * dh;
    const size_t nb = static_cast<size_t>(H) * dh;
    const HostArena h = host_arena(arena, B, H, T, dh);
    *where = h;
    if (cudaMemsetAsync(h.ws, 0, ws_bytes(), st) != cudaSuccess) return IP_ERR_CUDA;
    struct Copy {
        void *dst;
        const void *src;
        size_t n;
    } copies[] = {{h.q, q, nact}, {h.k, k, nact}, {h.v, v, nact}, {h.p, p, np},
                  {h.u, u, nb},   {h.vb, v_bias, nb}, {h.len, lengths, lengths ? 4ull * B : 0}};
    for (const Copy &c : copies)
        if (c.n && cudaMemcpyAsync(c.dst, c.src, c.n, cudaMemcpyHostToDevice, st) != cudaSuccess)
            return IP_ERR_CUDA;
    rc = ip_relpos_mhsa_i8(h.q, h.k, h.v, h.p, h.u, h.vb, multipliers, shifts, sm,
                           lengths ? h.len : nullptr, B, H, T, dh, h.out, h.ws,
                           ws_bytes() + gs_scores_bytes(T),
                           stream);
    if (rc != IP_OK) return rc;
    if (nact && cudaMemcpyAsync(out, h.out, nact, cudaMemcpyDeviceToHost, st) != cudaSuccess)
        return IP_ERR_CUDA;
    return IP_OK;
}

}  // namespace

int ip_relpos_mhsa_i8_host(const int8_t *q, const int8_t *k, const int8_t *v, const int8_t *p,
                           const int8_t *u, const int8_t *v_bias, const int32_t *multipliers,
                           const int32_t *shifts, const ip_isoftmax_params *sm,
                           const int32_t *lengths, int B, int H, int T, int dh, int8_t *out,
                           void *arena, size_t arena_bytes, ip_stream_t stream) {
    HostArena h;
    const int rc = host_enqueue(q, k, v, p, u, v_bias, multipliers, shifts, sm, lengths, B, H, T,
                                dh, out, arena, arena_bytes, stream, &h);
    if (rc != IP_OK || B == 0 || H == 0) return rc;
    return ip_relpos_mhsa_status(h.ws, stream);
}

int ip_relpos_mhsa_i8_host_async(const int8_t *q, const int8_t *k, const int8_t *v,
                                 const int8_t *p, const int8_t *u, const int8_t *v_bias,
                                 const int32_t *multipliers, const int32_t *shifts,
                                 const ip_isoftmax_params *sm, const int32_t *lengths, int B,
                                 int H, int T, int dh, int8_t *out, void *arena,
                                 size_t arena_bytes, ip_stream_t stream) {
    HostArena h;
    return host_enqueue(q, k, v, p, u, v_bias, multipliers, shifts, sm, lengths, B, H, T, dh,
                        out, arena, arena_bytes, stream, &h);
}

int ip_relpos_mhsa_host_status(const void *arena, int B, int H, int T, int dh,
                               ip_stream_t stream) {
    if (!arena) return IP_ERR_NULL;
    const int rc = check_shape(B, H, T, dh);
    if (rc != IP_OK) return rc;
    return ip_relpos_mhsa_status(host_arena(const_cast<void *>(arena), B, H, T, dh).ws, stream);
}

const char *ip_strerror(int code) {
    switch (code) {
    case IP_OK: return "ok";
    case IP_ERR_NULL: return "a required pointer is NULL";
    case IP_ERR_SHAPE: return "shape out of range (B, H >= 0; 1 <= T <= IP_MAX_T)";
    case IP_ERR_ALIGN: return "pointer misaligned (16 bytes; workspace and arena 256)";
    case IP_ERR_UNSUPPORTED: return "unsupported head width (dh must be 128)";
    case IP_ERR_CUDA: return "CUDA runtime call failed";
    case IP_ERR_TIMEOUT: return "kernel barrier wait timed out";
    case IP_ERR_PARAM: return "multiplier, shift or softmax constant out of its domain";
    case IP_ERR_WORKSPACE: return "workspace or arena too small";
    default: return "unknown error code";
    }
}

// Offline constants: float64 on the host, once per layer.
// ---- entry point without allocation --------------------------------------
// File-scope device scratch of ip_relpos_mhsa_i8_noalloc: the status word
// that ip_relpos_mhsa_i8 otherwise keeps in the caller's workspace.  Every
// GPU that loads the library holds it until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_scratch[IP_NOALLOC_SCRATCH_BYTES];

static std::mutex g_noalloc_mu;
static void *g_noalloc_addr[64] = {nullptr};

// Device address of g_noalloc_scratch on the current device, looked up
// once per device (with that device current) and cached.
static int noalloc_scratch(void **addr) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IP_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (g_noalloc_addr[dev] == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr)
            return IP_ERR_CUDA;
        g_noalloc_addr[dev] = p;
    }
    *addr = g_noalloc_addr[dev];
    return IP_OK;
}

int ip_relpos_mhsa_i8_noalloc(const int8_t *q, const int8_t *k, const int8_t *v, const int8_t *p,
                              const int8_t *u, const int8_t *v_bias, const int32_t *multipliers,
                              const int32_t *shifts, const ip_isoftmax_params *sm,
                              const int32_t *lengths, int B, int H, int T, int dh, int8_t *out,
                              ip_stream_t stream) {
    int rc = check_shape(B, H, T, dh);
    if (rc != IP_OK) return rc;
    if (B == 0 || H == 0) return IP_OK;
    const size_t need = ws_bytes();
    if (need > IP_NOALLOC_SCRATCH_BYTES) return IP_ERR_WORKSPACE;
    void *scratch = nullptr;
    rc = noalloc_scratch(&scratch);
    if (rc != IP_OK) return rc;
    // The status word is shared by every call and keeps the last call's
    // value: clear it in stream order before this call's kernel.
    if (cudaMemsetAsync(scratch, 0, need, reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess)
        return IP_ERR_CUDA;
    return ip_relpos_mhsa_i8(q, k, v, p, u, v_bias, multipliers, shifts, sm, lengths, B, H, T, dh,
                             out, scratch, IP_NOALLOC_SCRATCH_BYTES, stream);
}

int ip_relpos_mhsa_noalloc_status(ip_stream_t stream) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return IP_ERR_CUDA;
    {
        std::lock_guard<std::mutex> lock(g_noalloc_mu);
        if (g_noalloc_addr[dev] == nullptr) return IP_OK;   // no call on this device yet
    }
    void *scratch = nullptr;
    const int rc = noalloc_scratch(&scratch);
    if (rc != IP_OK) return rc;
    return ip_relpos_mhsa_status(scratch, stream);
}

int ip_dyadic_multiplier(double ratio, int32_t *m, int32_t *s) {
    if (!m || !s) return IP_ERR_NULL;
    if (!(ratio > 0.0) || !isfinite(ratio)) return IP_ERR_PARAM;
    int e = 0;
    const double frac = frexp(ratio, &e);   // ratio = frac 2^e, frac in [0.5, 1)
    int sh = -e;
    if (sh > 31) {
        const double mm = floor(ratio * ldexp(1.0, 62) + 0.5);
        *m = static_cast<int32_t>(mm);
        *s = 31;
        return IP_OK;
    }
    if (sh < 0) return IP_ERR_PARAM;
    double mm = floor(frac * ldexp(1.0, 31) + 0.5);
    if (mm >= ldexp(1.0, 31)) {
        mm = ldexp(1.0, 30);
        sh -= 1;
        if (sh < 0) return IP_ERR_PARAM;
    }
    *m = static_cast<int32_t>(mm);
    *s = sh;
    return IP_OK;
}

int ip_dyadic_pair(double r_c, double r_p, int32_t *m_c, int32_t *m_p, int32_t *s) {
    if (!m_c || !m_p || !s) return IP_ERR_NULL;
    if (!(r_c > 0.0) || !(r_p > 0.0) || !isfinite(r_c) || !isfinite(r_p)) return IP_ERR_PARAM;
    int32_t mbig = 0, sh = 0;
    const int rc = ip_dyadic_multiplier(r_c > r_p ? r_c : r_p, &mbig, &sh);
    if (rc != IP_OK) return rc;
    const double scale = ldexp(1.0, 31 + sh);
    const double mc = floor(r_c * scale + 0.5), mp = floor(r_p * scale + 0.5);
    if (mc >= ldexp(1.0, 31) || mp >= ldexp(1.0, 31)) return IP_ERR_PARAM;
    *m_c = static_cast<int32_t>(mc);
    *m_p = static_cast<int32_t>(mp);
    *s = sh;
    return IP_OK;
}

int ip_isoftmax_params_from_scale(double S_s, ip_isoftmax_params *out) {
    if (!out) return IP_ERR_NULL;
    if (!(S_s > 0.0) || !isfinite(S_s)) return IP_ERR_PARAM;
    const double ln2 = 0.6931471805599453;
    const double qln2 = floor(ln2 / S_s), qb = floor(1.353 / S_s),
                 qc = floor(0.344 / (0.3585 * (S_s * S_s)));
    if (qln2 > 2147483647.0 || qb > 2147483647.0 || qc > 2147483647.0) return IP_ERR_PARAM;
    out->q_ln2 = static_cast<int32_t>(qln2);
    out->q_b = static_cast<int32_t>(qb);
    out->q_c = static_cast<int32_t>(qc);
    return IP_OK;
}

int ip_relpos_layer_constants(double S_Q, double S_K, double S_P, double S_V, double S_s,
                              double S_O, int dh, int32_t *multipliers, int32_t *shifts,
                              ip_isoftmax_params *softmax) {
    if (!multipliers || !shifts || !softmax) return IP_ERR_NULL;
    const double sc[6] = {S_Q, S_K, S_P, S_V, S_s, S_O};
    for (double x : sc)
        if (!(x > 0.0) || !isfinite(x)) return IP_ERR_PARAM;
    if (dh < 1) return IP_ERR_PARAM;
    const double root = sqrt(static_cast<double>(dh));
    const double r_c = S_Q * S_K / (S_s * root);   // Eq. 11, content branch
    const double r_p = S_Q * S_P / (S_s * root);   // Eq. 11, position branch
    const double r_o = S_V / (S_O * 256.0);        // Eq. 7, probabilities on 2^-8
    int32_t m_c = 0, m_p = 0, s_s = 0, m_o = 0, s_o = 0;
    ip_isoftmax_params sm{};
    int rc = ip_dyadic_pair(r_c, r_p, &m_c, &m_p, &s_s);
    if (rc == IP_OK) rc = ip_dyadic_multiplier(r_o, &m_o, &s_o);
    if (rc == IP_OK) rc = ip_isoftmax_params_from_scale(S_s, &sm);
    if (rc != IP_OK) return rc;
    multipliers[0] = m_c;
    multipliers[1] = m_p;
    multipliers[2] = m_o;
    shifts[0] = s_s;
    shifts[1] = s_o;
    *softmax = sm;
    return IP_OK;
}

long long ip_probe_int8_mma(int blocks, int iters, int *sink, ip_stream_t stream) {
    if (blocks < 1 || iters < 1 || !sink) return -1;
    ipk::int8_mma_probe_kernel<<<blocks, ipk::PROBE_THREADS, 0,
                                 reinterpret_cast<cudaStream_t>(stream)>>>(sink, 0x9e3779b9u,
                                                                            iters);
    if (cudaGetLastError() != cudaSuccess) return -1;
    return static_cast<long long>(blocks) * (ipk::PROBE_THREADS / 32) * iters * ipk::PROBE_CHAINS *
           (16ll * 8 * 32 * 2);
}

long long ip_probe_int8_mix(int blocks, int iters, int mma_warps, int *sink, ip_stream_t stream) {
    if (blocks < 1 || iters < 1 || mma_warps < 0 || mma_warps > ipk::PROBE_THREADS / 32 || !sink)
        return -1;
    ipk::int8_mix_probe_kernel<<<blocks, ipk::PROBE_THREADS, 0,
                                 reinterpret_cast<cudaStream_t>(stream)>>>(sink, 0x9e3779b9u, iters,
                                                                           mma_warps);
    if (cudaGetLastError() != cudaSuccess) return -1;
    const long long mma = static_cast<long long>(mma_warps) * iters * ipk::MIX_MMA_CHAINS *
                          (16ll * 8 * 32 * 2);
    const long long dp4a = static_cast<long long>(ipk::PROBE_THREADS / 32 - mma_warps) * 4 * iters *
                           4 * ipk::MIX_DP4A_CHAINS * (32ll * 4 * 2);
    return static_cast<long long>(blocks) * (mma + dp4a);
}

int ip_debug_set_timeout_cycles(long long cycles) {
    g_timeout_cycles = cycles >= 0 ? cycles : DEFAULT_TIMEOUT;
    return IP_OK;
}

int ip_debug_set_split_mode(int mode) {
    g_split_mode = mode < 0 ? -1 : (mode > 2 ? 2 : mode);
    return IP_OK;
}

int ip_debug_set_wide_sums(int on) {
    g_wide_sums = on ? 1 : 0;
    return IP_OK;
}

int ip_debug_set_stall_injection(int on) {
    g_stall_injection = on ? 1 : 0;
    return IP_OK;
}

}  // extern "C"
