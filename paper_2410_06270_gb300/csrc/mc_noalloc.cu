// mc_noalloc.cu -- mc_moe_forward_static: the layer forward of mc_moe_forward
// on the mma.sync expert path, with its scratch in a fixed device array that
// belongs to this library instead of a caller-provided workspace.
//
// For callers that must not allocate device memory once they are running: a
// serving loop that freezes its memory plan at start-up, a plug-in whose device
// memory belongs to a host framework, a plain C caller with no device allocator
// of its own.  Nothing here allocates: the scratch is a file-scope __device__
// array (one instance per device), and its address is taken once per device
// with cudaGetSymbolAddress.
#include <math.h>
#include <string.h>

#include <mutex>

#include "mc_host.h"
#include "mc_kernels.h"

namespace mc {

constexpr size_t kStaticScratchBytes = (size_t)16 << 20;  // 16 MiB
static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
static std::mutex g_static_mu;
static void *g_static_ptr[kMaxDevices];

// Device address of this device's scratch.  The first call on a device (with
// that device current) takes it with cudaGetSymbolAddress; later calls reuse it.
static int static_scratch(void **out)
{
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(err));
    if (dev < 0 || dev >= kMaxDevices) return set_error(MC_ERR_UNSUPPORTED, "device ordinal %d >= %d", dev, kMaxDevices);
    std::lock_guard<std::mutex> lock(g_static_mu);
    if (!g_static_ptr[dev]) {
        void *p = nullptr;
        err = cudaGetSymbolAddress(&p, g_static_scratch);
        if (err != cudaSuccess)
            return set_error(MC_ERR_CUDA, "cudaGetSymbolAddress(scratch): %s", cudaGetErrorString(err));
        g_static_ptr[dev] = p;
    }
    *out = g_static_ptr[dev];
    return MC_OK;
}

// The scratch of the mma.sync path, carved like mc_moe_forward's workspace
// minus the buffers only the tensor-core path uses.
struct StaticWs {
    int32_t *status, *idx, *offsets, *perm, *inv, *nchunks, *counters;
    float *w, *opart;
    uint8_t *pruned, *xvec, *hvec;
    ChunkInfo *chunks;
    int max_chunks, KS;
    size_t total;
};

// KS: column splits of the W2 pass (the fp32 partial outputs hold KS copies).
static StaticWs carve_static(const mc_shape *s, int T, int KS, uint8_t *base)
{
    StaticWs w;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t *r = base ? base + off : nullptr;
        off = (off + bytes + 255) & ~(size_t)255;
        return r;
    };
    w.KS = KS;
    w.max_chunks = max_chunks_for(T, s->E);
    const size_t P = 2 * (size_t)T, MC = (size_t)w.max_chunks, VB = (size_t)vec_bytes(s->group);
    w.status = (int32_t *)take(256);
    w.idx = (int32_t *)take(P * 4);
    w.w = (float *)take(P * 4);
    w.pruned = take((size_t)T);
    w.offsets = (int32_t *)take(4 * (kMaxE + 1));
    w.perm = (int32_t *)take(P * 4);
    w.inv = (int32_t *)take(P * 4);
    w.chunks = (ChunkInfo *)take(MC * sizeof(ChunkInfo));
    w.nchunks = (int32_t *)take(4);
    w.counters = (int32_t *)take(16);
    w.xvec = take(MC * 2 * (s->H / kTileK) * VB);
    w.hvec = take(MC * 2 * (s->F / kTileK) * VB);
    w.opart = (float *)take((size_t)w.KS * P * s->H * 4);
    w.total = off;
    return w;
}

}  // namespace mc

using namespace mc;

extern "C" int mc_moe_forward_static(const void *x, const void *gate_w, int T, const mc_shape *shape,
                                     const int8_t *bits_host, const void *packed_dev, float mu,
                                     const uint8_t *protect, void *y, int32_t *status_dev, void *stream)
{
    clear_error();
    int rc = check_bits(shape, bits_host);
    if (rc) return rc;
    if (!(mu == mu) || mu < 0.f || isinf(mu))
        return set_error(MC_ERR_INVALID_ARG, "mu=%g: need a finite mu >= 0", (double)mu);
    if (T < 0) return set_error(MC_ERR_INVALID_ARG, "T=%d < 0", T);
    if (T == 0) return MC_OK;
    if (!x || !gate_w || !packed_dev || !y) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    if (!aligned(x, 16) || !aligned(gate_w, 16) || !aligned(y, 16) || !aligned(packed_dev, 256) ||
        (status_dev && !aligned(status_dev, 4)))
        return set_error(MC_ERR_INVALID_ARG, "x, gate_w, y need 16-byte and packed_dev 256-byte alignment");
    // W2 column splits: mc_moe_forward's choice when its partial outputs fit in
    // the scratch, else a single split (the limit below is the single split's)
    int dev = 0, nsm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return set_error(MC_ERR_CUDA, "device query failed");
    int KS = choose_ks(shape, T, nsm);
    size_t need = carve_static(shape, T, KS, nullptr).total;
    if (need > kStaticScratchBytes && KS > 1) {
        KS = 1;
        need = carve_static(shape, T, KS, nullptr).total;
    }
    if (need > kStaticScratchBytes)
        return set_error(MC_ERR_INVALID_ARG,
                         "T=%d needs %zu bytes of scratch, more than the %zu-byte static scratch of "
                         "mc_moe_forward_static; use mc_moe_forward with a workspace",
                         T, need, kStaticScratchBytes);
    void *base = nullptr;
    if ((rc = static_scratch(&base))) return rc;
    const StaticWs ws = carve_static(shape, T, KS, (uint8_t *)base);
    cudaStream_t st = (cudaStream_t)stream;
    int32_t *status = status_dev ? status_dev : ws.status;
    if (!status_dev) {
        cudaError_t err = cudaMemsetAsync(ws.status, 0, 4, st);
        if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaMemsetAsync: %s", cudaGetErrorString(err));
    }

    RouteParams rp{};
    memset(&rp, 0, sizeof rp);
    rp.x = (const __nv_bfloat16 *)x;
    rp.gate = (const __nv_bfloat16 *)gate_w;
    rp.T = T;
    rp.H = shape->H;
    rp.E = shape->E;
    rp.neg_log_mu = mu <= 0.f ? INFINITY : (float)(-log((double)mu));
    rp.protect = protect;
    rp.idx = ws.idx;
    rp.w = ws.w;
    rp.pruned = ws.pruned;
    PermuteParams pp{};
    memset(&pp, 0, sizeof pp);
    pp.idx = ws.idx;
    pp.pruned = ws.pruned;
    pp.T = T;
    pp.E = shape->E;
    for (int e = 0; e < shape->E; ++e) pp.bits[e] = bits_host[e];
    pp.offsets = ws.offsets;
    pp.perm = ws.perm;
    pp.inv = ws.inv;
    pp.chunks = ws.chunks;
    pp.nchunks = ws.nchunks;
    pp.counters = ws.counters;
    pp.chunk = kChunk;
    if ((rc = launch_route(rp, pp, st))) return rc;

    ExpertParams ep{};
    memset(&ep, 0, sizeof ep);  // the tensor-core path's buffers stay NULL: not used here
    ep.packed = (const uint8_t *)packed_dev;
    uint64_t total;
    layout_offsets(shape, bits_host, ep.mat_off, &total);
    for (int e = 0; e < shape->E; ++e) ep.bits[e] = bits_host[e];
    ep.E = shape->E;
    ep.H = shape->H;
    ep.F = shape->F;
    ep.group = shape->group;
    ep.chunks = ws.chunks;
    ep.nchunks = ws.nchunks;
    ep.counters = ws.counters;
    ep.x = (const __nv_bfloat16 *)x;
    ep.perm = ws.perm;
    ep.xvec = ws.xvec;
    ep.hvec = ws.hvec;
    ep.opart = ws.opart;
    ep.KS = ws.KS;
    ep.Pmax = 2 * T;
    ep.max_chunks = ws.max_chunks;
    ep.status = status;
    ep.hdr_ok = ws.status + kHdrOkWord;
    ep.timeout_ns = wait_bound_ns();  // the mc_set_debug hooks apply here as well
    ep.debug = debug_flags();
    if ((rc = launch_gemv(ep, st))) return rc;

    CombineParams cp{};
    cp.opart = ws.opart;
    cp.w = ws.w;
    cp.inv = ws.inv;
    cp.T = T;
    cp.H = shape->H;
    cp.KS = ws.KS;
    cp.Pmax = 2 * T;
    cp.y = (__nv_bfloat16 *)y;
    return launch_combine(cp, st);
}
