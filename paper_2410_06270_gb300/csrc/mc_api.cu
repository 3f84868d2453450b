// mc_api.cu -- the extern "C" entry points of include/mc.h: argument checks,
// workspace carving and kernel launches.  No entry point here allocates device
// memory or synchronises, except the ones documented as synchronous.
#include <math.h>
#include <string.h>

#include <atomic>
#include <vector>

#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"

namespace mc {

// expert paths of mc_moe_forward (mc_set_path)
constexpr int kPathAuto = 0, kPathGemv = 1, kPathGemm = 2;
static std::atomic<int> g_path{kPathAuto};
// pairs (2 T) from which mc_moe_forward's automatic choice is the prefill GEMM:
// measured on the Mixtral-8x7b layer, the GEMV path (each weight tile decoded
// once per 16-pair chunk) is faster up to ~96 tokens, the GEMM (once per
// 128-pair token block) from ~128 tokens on
constexpr int kPrefillPairs = 240;
static std::atomic<int> g_debug{0};
static std::atomic<unsigned long long> g_timeout_ns{1000000000ull};  // 1 s

#define MC_CUDA(call)                                                                         \
    do {                                                                                      \
        cudaError_t err_ = (call);                                                            \
        if (err_ != cudaSuccess)                                                              \
            return set_error(MC_ERR_CUDA, "%s failed: %s", #call, cudaGetErrorString(err_)); \
    } while (0)

static inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

// Column splits of the W2 GEMV pass.  The workspace holds up to kMaxKS splits
// (decode sizes); the forward picks, among the divisors of F/128 that leave each
// item at least two ring stages, the split count whose work items (estimated
// chunks x 256-row block pairs x splits) fill the SMs' last wave best, the
// smaller one on ties.

int max_ks(const mc_shape *s, int T) { return T > 64 ? 1 : kMaxKS; }

int choose_ks(const mc_shape *s, int T, int nsm)
{
    const int nt = s->F / kTileK, npairs = (s->H / kBlockRows + 1) / 2;
    const int chunks = 2 * T < s->E ? 2 * T : s->E;  // pairs land on distinct experts at small T
    int best = 1;
    double best_eff = -1.0;
    for (int ks = 1; ks <= max_ks(s, T); ++ks) {
        if (nt % ks || nt / ks < 8) continue;
        const long items = (long)chunks * npairs * ks, waves = (items + nsm - 1) / nsm;
        const double eff = (double)items / (double)(waves * nsm);
        if (eff > best_eff + 1e-9) {
            best_eff = eff;
            best = ks;
        }
    }
    return best;
}

struct Workspace {
    int32_t *status;
    int32_t *idx;
    float *w;
    uint8_t *pruned;
    int32_t *offsets, *perm, *inv;
    ChunkInfo *chunks;
    int32_t *nchunks, *counters;
    int32_t *route_done;  // zero between calls: single-launch routing for small T
    uint8_t *xvec, *hvec;
    uint8_t *ximg, *himg;
    float *opart;
    int max_chunks, max_blocks, KS;
    size_t total;
};

static Workspace carve(const mc_shape *s, int T, void *base)
{
    Workspace w;
    uint8_t *p = (uint8_t *)base;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t *r = p ? p + off : nullptr;
        off = align256(off + bytes);
        return r;
    };
    w.KS = max_ks(s, T);  // room for the largest split count the forward may pick
    w.max_chunks = max_chunks_for(T, s->E);
    const size_t P = 2 * (size_t)T, MC = (size_t)w.max_chunks;
    // The words that must be zero when a call starts (and that every call leaves
    // at zero) come first, at offsets that do not depend on T, so one workspace
    // serves calls with any T up to the T it was sized for.
    w.status = (int32_t *)take(256);
    w.route_done = (int32_t *)take(4);
    w.idx = (int32_t *)take(P * 4);
    w.w = (float *)take(P * 4);
    w.pruned = (uint8_t *)take((size_t)T);
    w.offsets = (int32_t *)take(4 * (kMaxE + 1));
    w.perm = (int32_t *)take(P * 4);
    w.inv = (int32_t *)take(P * 4);
    w.chunks = (ChunkInfo *)take(MC * sizeof(ChunkInfo));
    w.nchunks = (int32_t *)take(4);
    w.counters = (int32_t *)take(16);
    w.xvec = (uint8_t *)take(MC * 2 * (s->H / kTileK) * (size_t)vec_bytes(s->group));
    w.hvec = (uint8_t *)take(MC * 2 * (s->F / kTileK) * (size_t)vec_bytes(s->group));
    w.max_blocks = max_blocks_for(T, s->E);
    w.ximg = (uint8_t *)take(img_buffer_bytes(w.max_blocks, s->H));
    w.himg = (uint8_t *)take(img_buffer_bytes(w.max_blocks, s->F));
    w.opart = (float *)take((size_t)w.KS * P * s->H * 4);
    w.total = off;
    return w;
}

static int check_mu(float mu)
{
    if (!(mu == mu) || mu < 0.f || isinf(mu))
        return set_error(MC_ERR_INVALID_ARG, "mu=%g: need a finite mu >= 0", (double)mu);
    return MC_OK;
}

static float neg_log_mu(float mu)
{
    if (mu <= 0.f) return INFINITY;
    return (float)(-log((double)mu));
}

bool pdl_enabled() { return !(g_debug.load() & kDebugNoPdl); }
int debug_flags() { return g_debug.load(); }
uint64_t wait_bound_ns() { return g_timeout_ns.load(); }

}  // namespace mc

using namespace mc;

extern "C" {

int mc_set_path(int path)
{
    if (path != kPathAuto && path != kPathGemv && path != kPathGemm) {
        clear_error();
        return set_error(MC_ERR_INVALID_ARG, "path %d: 0 (automatic), 1 (GEMV) or 2 (GEMM)", path);
    }
    return g_path.exchange(path);
}

// Test hook (not in the public header's main API): debug flags and the bound on
// device waits.  flags = 1 makes the weight producer issue nothing, so every
// consumer wait runs into the bound and the status word reports MC_ERR_TIMEOUT.
int mc_set_debug(int flags, unsigned long long timeout_ns)
{
    g_debug = flags;
    if (timeout_ns) g_timeout_ns = timeout_ns;
    return MC_OK;
}

size_t mc_moe_workspace_size(const mc_shape *shape, int T_max)
{
    if (check_shape(shape) || T_max < 0) return 0;
    return carve(shape, T_max, nullptr).total;
}

int mc_route(const void *x, const void *gate_w, int T, const mc_shape *shape, float mu, const uint8_t *protect,
             int32_t *topk_idx, float *topk_w, uint8_t *pruned, int32_t *expert_offsets, int32_t *perm, void *stream)
{
    clear_error();
    int rc = check_shape(shape);
    if (rc) return rc;
    if ((rc = check_mu(mu))) return rc;
    if (T < 0) return set_error(MC_ERR_INVALID_ARG, "T=%d < 0", T);
    if (T == 0) return MC_OK;
    if (!x || !gate_w || !topk_idx || !topk_w || !pruned || !expert_offsets || !perm)
        return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    if (!aligned(x, 16) || !aligned(gate_w, 16))
        return set_error(MC_ERR_INVALID_ARG, "x and gate_w must be 16-byte aligned");
    RouteParams rp{};
    memset(&rp, 0, sizeof rp);
    rp.x = (const __nv_bfloat16 *)x;
    rp.gate = (const __nv_bfloat16 *)gate_w;
    rp.T = T;
    rp.H = shape->H;
    rp.E = shape->E;
    rp.neg_log_mu = neg_log_mu(mu);
    rp.protect = protect;
    rp.idx = topk_idx;
    rp.w = topk_w;
    rp.pruned = pruned;
    PermuteParams pp{};
    memset(&pp, 0, sizeof pp);
    pp.idx = topk_idx;
    pp.pruned = pruned;
    pp.T = T;
    pp.E = shape->E;
    pp.offsets = expert_offsets;
    pp.perm = perm;
    pp.chunk = kChunk;
    if (g_debug.load() & kDebugRouteFused) {
        int32_t *done = route_done_word();
        if (!done) return set_error(MC_ERR_CUDA, "routing arrival word not found");
        return launch_route(rp, pp, (cudaStream_t)stream, done);
    }
    return launch_route(rp, pp, (cudaStream_t)stream);
}

}  // extern "C"

// mc_moe_forward with the stack's pre-norm and residual folded into its first
// and last launches (LayerPrePost).
int mc::moe_forward_ex(const void *x, const void *gate_w, int T, const mc_shape *shape, const int8_t *bits_host,
                       const void *packed_dev, float mu, const uint8_t *protect, void *y, const LayerPrePost *lpp,
                       void *workspace, size_t ws_bytes, int32_t *topk_idx_out, float *topk_w_out,
                       uint8_t *pruned_out, void *stream)
{
    clear_error();
    int rc = check_bits(shape, bits_host);
    if (rc) return rc;
    if ((rc = check_mu(mu))) return rc;
    if (T < 0) return set_error(MC_ERR_INVALID_ARG, "T=%d < 0", T);
    if (T == 0) return MC_OK;
    if (!x || !gate_w || !packed_dev || !y || !workspace)
        return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    if (!aligned(x, 16) || !aligned(gate_w, 16) || !aligned(y, 16) || !aligned(packed_dev, 256) ||
        !aligned(workspace, 256))
        return set_error(MC_ERR_INVALID_ARG, "x, gate_w, y need 16-byte and packed_dev, workspace 256-byte alignment");
    Workspace ws = carve(shape, T, workspace);
    if (ws_bytes < ws.total)
        return set_error(MC_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu", ws_bytes, ws.total);
    cudaStream_t st = (cudaStream_t)stream;
    // expert path: many pairs per expert -> tensor-core grouped GEMM (prefill),
    // few -> mma.sync grouped GEMV (decode); mc_set_path overrides
    int path = g_path;
    // 16-bit (unquantised) experts have the mma.sync kernels only
    const bool dense = bits_host[0] == 16;
    if (path == kPathAuto) path = dense ? kPathGemv : 2 * T >= kPrefillPairs ? kPathGemm : kPathGemv;
    if (dense && path != kPathGemv)
        return set_error(MC_ERR_UNSUPPORTED, "16-bit experts run on the mma.sync path only (path %d requested)", path);

    RouteParams rp{};
    memset(&rp, 0, sizeof rp);
    rp.x = (const __nv_bfloat16 *)x;
    rp.gate = (const __nv_bfloat16 *)gate_w;
    rp.T = T;
    rp.H = shape->H;
    rp.E = shape->E;
    rp.neg_log_mu = neg_log_mu(mu);
    rp.protect = protect;
    rp.idx = ws.idx;
    rp.w = ws.w;
    rp.pruned = ws.pruned;
    rp.idx_out = topk_idx_out;
    rp.w_out = topk_w_out;
    rp.pruned_out = pruned_out;
    if (lpp && lpp->norm_in) {
        if (shape->H > 16384 || !aligned(lpp->norm_in, 16) || !aligned(lpp->gamma, 16))
            return set_error(MC_ERR_INVALID_ARG, "pre-norm input and gamma need 16-byte alignment, H <= 16384");
        rp.h_in = (const __nv_bfloat16 *)lpp->norm_in;
        rp.gamma = (const __nv_bfloat16 *)lpp->gamma;
        rp.eps = lpp->eps;
    }
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
    pp.chunk = path == kPathGemm ? 128 : kChunk;
    rc = launch_route(rp, pp, st, ws.route_done);
    if (rc) return rc;

    ExpertParams ep{};
    memset(&ep, 0, sizeof ep);
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
    ep.ximg = ws.ximg;
    ep.himg = ws.himg;
    ep.max_blocks = ws.max_blocks;
    ep.opart = ws.opart;
    int nsm = 0, dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return set_error(MC_ERR_CUDA, "device query failed");
    ep.KS = path == kPathGemm ? 1 : choose_ks(shape, T, nsm);  // the GEMM's W2 pass covers all of F at once
    ep.Pmax = 2 * T;
    ep.max_chunks = ws.max_chunks;
    ep.status = ws.status;
    ep.hdr_ok = ws.status + kHdrOkWord;
    ep.timeout_ns = g_timeout_ns;
    ep.debug = g_debug;
    rc = path == kPathGemm ? launch_gemm(ep, st) : launch_gemv(ep, st);
    if (rc) return rc;

    CombineParams cp{};
    cp.opart = ws.opart;
    cp.w = ws.w;
    cp.inv = ws.inv;
    cp.T = T;
    cp.H = shape->H;
    cp.KS = ep.KS;
    cp.Pmax = 2 * T;
    cp.y = (__nv_bfloat16 *)y;
    cp.resid = lpp ? (const __nv_bfloat16 *)lpp->resid : nullptr;
    return launch_combine(cp, st);
}

extern "C" {

int mc_moe_forward(const void *x, const void *gate_w, int T, const mc_shape *shape, const int8_t *bits_host,
                   const void *packed_dev, float mu, const uint8_t *protect, void *y, void *workspace,
                   size_t ws_bytes, int32_t *topk_idx_out, float *topk_w_out, uint8_t *pruned_out, void *stream)
{
    return moe_forward_ex(x, gate_w, T, shape, bits_host, packed_dev, mu, protect, y, nullptr, workspace, ws_bytes,
                          topk_idx_out, topk_w_out, pruned_out, stream);
}

int mc_check_status(void *workspace, void *stream)
{
    clear_error();
    if (!workspace) return set_error(MC_ERR_INVALID_ARG, "NULL workspace");
    cudaStream_t st = (cudaStream_t)stream;
    int32_t v = 0;
    MC_CUDA(cudaMemcpyAsync(&v, workspace, 4, cudaMemcpyDeviceToHost, st));
    MC_CUDA(cudaStreamSynchronize(st));
    if (v != 0) {
        int32_t z = 0;
        MC_CUDA(cudaMemcpyAsync(workspace, &z, 4, cudaMemcpyHostToDevice, st));
        MC_CUDA(cudaStreamSynchronize(st));
        return set_error(v, "device status word reported %d", v);
    }
    return MC_OK;
}

int mc_pack_experts(const mc_shape *shape, const int8_t *bits_host, const uint8_t *const *codes_host,
                    const uint16_t *const *scale_host, const uint16_t *const *zero_host, void *packed_dev,
                    size_t packed_bytes, void *stream)
{
    clear_error();
    size_t need = mc_packed_size(shape, bits_host);
    if (!need) return check_bits(shape, bits_host);
    if (!packed_dev) return set_error(MC_ERR_INVALID_ARG, "NULL packed_dev");
    if (!aligned(packed_dev, 256)) return set_error(MC_ERR_INVALID_ARG, "packed_dev must be 256-byte aligned");
    if (packed_bytes < need)
        return set_error(MC_ERR_INVALID_ARG, "packed buffer has %zu bytes, needs %zu", packed_bytes, need);
    void *stage = nullptr;
    MC_CUDA(cudaMallocHost(&stage, need));
    int rc = mc_pack_experts_host(shape, bits_host, codes_host, scale_host, zero_host, stage, need);
    if (rc == MC_OK) {
        cudaStream_t st = (cudaStream_t)stream;
        cudaError_t e1 = cudaMemcpyAsync(packed_dev, stage, need, cudaMemcpyHostToDevice, st);
        cudaError_t e2 = e1 == cudaSuccess ? cudaStreamSynchronize(st) : e1;
        if (e2 != cudaSuccess) rc = set_error(MC_ERR_CUDA, "upload failed: %s", cudaGetErrorString(e2));
    }
    cudaFreeHost(stage);
    return rc;
}

int mc_pack_verify(const mc_shape *shape, const int8_t *bits_host, const void *packed_dev, size_t packed_bytes)
{
    clear_error();
    int rc = check_bits(shape, bits_host);
    if (rc) return rc;
    if (!packed_dev) return set_error(MC_ERR_INVALID_ARG, "NULL packed_dev");
    size_t need = mc_packed_size(shape, bits_host);
    if (packed_bytes < need) return set_error(MC_ERR_BAD_PACK, "buffer has %zu bytes, needs %zu", packed_bytes, need);
    PackHeader hd;
    MC_CUDA(cudaMemcpy(&hd, packed_dev, sizeof hd, cudaMemcpyDeviceToHost));
    if (hd.magic != kMagic || hd.version != kFormatVersion)
        return set_error(MC_ERR_BAD_PACK, "bad magic/version (%08x/%u)", hd.magic, hd.version);
    if (hd.E != shape->E || hd.H != shape->H || hd.F != shape->F || hd.group != shape->group)
        return set_error(MC_ERR_BAD_PACK, "header shape (%d,%d,%d,%d) != (%d,%d,%d,%d)", hd.E, hd.H, hd.F, hd.group,
                         shape->E, shape->H, shape->F, shape->group);
    for (int e = 0; e < shape->E; ++e)
        if (hd.bits[e] != bits_host[e])
            return set_error(MC_ERR_BAD_PACK, "header bits[%d]=%d != %d", e, hd.bits[e], bits_host[e]);
    if (hd.total_bytes != need) return set_error(MC_ERR_BAD_PACK, "header total %llu != %zu",
                                                 (unsigned long long)hd.total_bytes, need);
    return MC_OK;
}

}  // extern "C"
