// mc_route.cu -- the gate of Eq. 1, top-2 selection with renormalised softmax
// weights, the ODP test of Eq. 5 with the token protection of Sec. 2.3.2 and the
// token drop of Sec. 3.2 (Fig. 9: mask byte 2 masks all of a token's experts),
// and the permutation of kept (token, slot) pairs by expert.
//
// route_kernel: one CTA of 16 warps per token; each thread takes 8 columns of
//   a 4096-column round and issues all of the round's loads (x and the E gate
//   rows, 16 bytes each) before it uses any, so a round costs one memory round
//   trip; the partial logits meet in shared memory, warp 0 adds them up and
//   thread 0 takes the decision in fp32.
// route_cluster_kernel (T <= 16): the same as one thread-block cluster, the
//   decisions gathered in CTA 0's shared memory and placed by its first warp.
// permute_kernel: one CTA; histogram, exclusive scan and a stable placement with
//   __match_any_sync ranks, so the permutation is unique (ascending token within
//   an expert) and identical run to run.  It also lists the work chunks of the
//   expert kernels (one thread per expert) and resets their work counters.
#include <cooperative_groups.h>

#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"

namespace mc {

constexpr int kRouteThreads = 512;

// The pre-norm of token t's row (the stack): h_in[t] staged in shared memory and
// its sum of squares accumulated in the order of rmsnorm_vec_kernel (256
// threads, thread i over the 16-byte chunks i + 256 j, j < 8; warp xor
// reductions; the 8 warp partials added in order), so that inv and every
// normalised element f * inv * g are bit for bit those of mc_rmsnorm.
__device__ __forceinline__ float route_row_inv(const RouteParams &p, int t, uint4 *row_s, float *red)
{
    const int tid = threadIdx.x, n8 = p.H >> 3;
    const uint4 *hr = reinterpret_cast<const uint4 *>(p.h_in + (size_t)t * p.H);
    for (int c = tid; c < n8; c += kRouteThreads) row_s[c] = hr[c];
    __syncthreads();
    if (tid < 256) {
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int c = tid + 256 * i;
            if (c >= n8) continue;
            const uint4 v = row_s[c];
            const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float2 f = __bfloat1622float2(b2[k]);
                ss = fmaf(f.x, f.x, ss);
                ss = fmaf(f.y, f.y, ss);
            }
        }
        for (int m = 16; m >= 1; m >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, m);
        if ((tid & 31) == 0) red[tid >> 5] = ss;
    }
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w];
    return rsqrtf(tot / p.H + p.eps);
}

// The logits of token t by the whole CTA; thread 0 takes the decision and writes
// the outputs.
template <bool NORM>
//   sink (optional): where thread 0 also leaves the decision (e0, e1, pruned) of
//   token t, three ints at 3 t (the cluster routing: CTA 0's shared memory).
__device__ __forceinline__ void route_token(const RouteParams &p, int t, int *sink = nullptr)
{
    __shared__ float part[kRouteThreads / 32][kMaxE];
    __shared__ float red[8];
    // the pre-norm row: dynamic shared memory, H * 2 bytes, given only with h_in
    extern __shared__ uint4 row_s[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int H = p.H, E = p.E;
    const __nv_bfloat16 *xr = p.x + (size_t)t * H;
    // the gate's first column round goes out before the pre-norm's reduction
    uint4 gr[kMaxE];
    if constexpr (NORM) {
        const int c0 = 8 * threadIdx.x;
#pragma unroll
        for (int e = 0; e < kMaxE; ++e)
            if (e < E && c0 < H) gr[e] = *reinterpret_cast<const uint4 *>(p.gate + (size_t)e * H + c0);
    }
    float inv = 0.f;
    if constexpr (NORM) inv = route_row_inv(p, t, row_s, red);
    // the mask byte is needed only by thread 0's decision; load it now
    // (0: prunable, 2: dropped, anything else: protected)
    const int mask = threadIdx.x == 0 && p.protect != nullptr ? p.protect[t] : 0;
    float acc[kMaxE];
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) acc[e] = 0.f;
    for (int c0 = 8 * threadIdx.x; c0 < H; c0 += 8 * kRouteThreads) {
        uint4 raw;
        if constexpr (NORM) {
            // x = h * inv * gamma rounded to bf16 (mc_rmsnorm's expression), written
            // for the expert kernels and routed on as written
            const uint4 hv = row_s[c0 >> 3], gv = *reinterpret_cast<const uint4 *>(p.gamma + c0);
            const __nv_bfloat162 *h2 = reinterpret_cast<const __nv_bfloat162 *>(&hv);
            const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gv);
            __nv_bfloat162 *o2 = reinterpret_cast<__nv_bfloat162 *>(&raw);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float2 f = __bfloat1622float2(h2[k]), g = __bfloat1622float2(g2[k]);
                o2[k] = __floats2bfloat162_rn(f.x * inv * g.x, f.y * inv * g.y);
            }
            *reinterpret_cast<uint4 *>(const_cast<__nv_bfloat16 *>(xr) + c0) = raw;
        } else {
            raw = *reinterpret_cast<const uint4 *>(xr + c0);
        }
        if (!NORM || c0 != 8 * (int)threadIdx.x) {
#pragma unroll
            for (int e = 0; e < kMaxE; ++e)
                if (e < E) gr[e] = *reinterpret_cast<const uint4 *>(p.gate + (size_t)e * H + c0);
        }
        const __nv_bfloat162 *x2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
        float xf[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float2 f = __bfloat1622float2(x2[i]);
            xf[2 * i] = f.x;
            xf[2 * i + 1] = f.y;
        }
#pragma unroll
        for (int e = 0; e < kMaxE; ++e) {
            if (e < E) {
                const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gr[e]);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const float2 gf = __bfloat1622float2(g2[i]);
                    acc[e] = fmaf(xf[2 * i], gf.x, acc[e]);
                    acc[e] = fmaf(xf[2 * i + 1], gf.y, acc[e]);
                }
            }
        }
    }
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) {
        if (e < E) {
            for (int m = 16; m >= 1; m >>= 1) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], m);
            if (lane == 0) part[warp][e] = acc[e];
        }
    }
    __syncthreads();
    if (warp != 0) return;  // (route_token returns to its caller; the CTA re-joins there)
    // lane e adds up expert e's partials (warps in order), then thread 0 gathers them
    float le = 0.f;
    if (lane < E)
        for (int w = 0; w < kRouteThreads / 32; ++w) le += part[w][lane];
    float l[kMaxE];
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) l[e] = __shfl_sync(0xffffffffu, le, e);
    if (lane != 0) return;
    // top-2 on fp32 logits, lower index wins ties
    int e0 = 0;
    float b0 = l[0];
#pragma unroll
    for (int e = 1; e < kMaxE; ++e)
        if (e < E && l[e] > b0) {
            b0 = l[e];
            e0 = e;
        }
    int e1 = -1;
    float b1 = 0.f;
#pragma unroll
    for (int e = 0; e < kMaxE; ++e)
        if (e < E && e != e0 && (e1 < 0 || l[e] > b1)) {
            b1 = l[e];
            e1 = e;
        }
    const float d = b0 - b1;  // >= 0
    const float r = __expf(-d);     // = p1 / p0
    float w0 = 1.f / (1.f + r), w1 = r / (1.f + r);
    const bool drop = mask == 2, prot = mask != 0 && !drop;
    int prune = !prot && (d > p.neg_log_mu);
    if (prune) {
        w0 = 1.f;
        w1 = 0.f;
    }
    if (drop) {  // no expert: weights (0, 0), pruned = 2
        w0 = w1 = 0.f;
        prune = 2;
    }
    if (sink) {
        sink[3 * t] = e0;
        sink[3 * t + 1] = e1;
        sink[3 * t + 2] = prune;
    }
    p.idx[2 * t] = e0;
    p.idx[2 * t + 1] = e1;
    p.w[2 * t] = w0;
    p.w[2 * t + 1] = w1;
    p.pruned[t] = (uint8_t)prune;
    if (p.idx_out) {
        p.idx_out[2 * t] = e0;
        p.idx_out[2 * t + 1] = e1;
    }
    if (p.w_out) {
        p.w_out[2 * t] = w0;
        p.w_out[2 * t + 1] = w1;
    }
    if (p.pruned_out) p.pruned_out[t] = (uint8_t)prune;
}

template <bool NORM>
__global__ void __launch_bounds__(kRouteThreads) route_kernel(RouteParams p)
{
    pdl_trigger();
    pdl_wait();
    route_token<NORM>(p, blockIdx.x);
}

// Histogram, scan, stable placement and work-chunk list by one CTA of any size
// (whole warps, at most 1024 threads).
__device__ __forceinline__ void permute_block(const PermuteParams &p)
{
    __shared__ int cnt[kMaxE];
    __shared__ int run[kMaxE];
    __shared__ int nbits[kMaxE];
    __shared__ int wcnt[32][kMaxE];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int NP = 2 * p.T;
    // expert of pair i, -1 when ODP pruned it or its token was dropped (both loads
    // in flight together)
    auto pair_key = [&](int i) {
        const uint8_t pr = __ldcg(p.pruned + (i >> 1));
        const int e = __ldcg(p.idx + i);
        return ((i & 1) && pr) || pr == 2 ? -1 : e;
    };
    const int key0 = tid < NP ? pair_key(tid) : -1;  // the first pass's pair, kept for the placement
    if (tid < kMaxE) {
        cnt[tid] = 0;
        run[tid] = 0;
        int b = 0;
#pragma unroll
        for (int f = 0; f < kMaxE; ++f)
            if (f == tid) b = p.bits[f];
        nbits[tid] = b;
    }
    __syncthreads();
    for (int i = tid; i < NP; i += blockDim.x) {
        const int key = i == tid ? key0 : pair_key(i);
        if (key >= 0) atomicAdd(&cnt[key], 1);
    }
    __syncthreads();
    if (tid < p.E) {
        // expert tid: its offset, and the index of its first work chunk in the
        // order the expert kernels take them (more bits first, then by expert)
        const int e = tid, be = nbits[e], ce = cnt[e];
        int off = 0, k0 = 0;
        for (int f = 0; f < p.E; ++f) {
            const int cf = cnt[f], bf = nbits[f];
            if (f < e) off += cf;
            if (bf > be || (bf == be && f < e)) k0 += (cf + p.chunk - 1) / p.chunk;
        }
        p.offsets[e] = off;
        run[e] = off;
        if (e == p.E - 1) p.offsets[p.E] = off + ce;
        if (p.chunks) {
            for (int c = 0, k = k0; c < ce; c += p.chunk, ++k) {
                ChunkInfo ci;
                ci.e = e;
                ci.pair_base = off + c;
                ci.nv = min(p.chunk, ce - c);
                ci.bits = be;
                p.chunks[k] = ci;
            }
            if (e == 0) {
                int n = 0;
                for (int f = 0; f < p.E; ++f) n += (cnt[f] + p.chunk - 1) / p.chunk;
                *p.nchunks = n;
                for (int i = 0; i < 4; ++i) p.counters[i] = 0;
            }
        }
    }
    __syncthreads();
    for (int base = 0; base < NP; base += blockDim.x) {
        int i = base + tid;
        const int key = i >= NP ? -1 : base == 0 ? key0 : pair_key(i);
        for (int e = lane; e < kMaxE; e += 32) wcnt[warp][e] = 0;
        __syncwarp();
        unsigned same = __match_any_sync(0xffffffffu, key);
        int rank = __popc(same & ((1u << lane) - 1));
        if (key >= 0 && rank == 0) wcnt[warp][key] = __popc(same);
        __syncthreads();
        if (tid < p.E) {
            int s = run[tid];
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
                int c = wcnt[w][tid];
                wcnt[w][tid] = s;
                s += c;
            }
            run[tid] = s;
        }
        __syncthreads();
        if (i < NP) {
            int pos = key >= 0 ? wcnt[warp][key] + rank : -1;
            if (key >= 0) p.perm[pos] = i;
            if (p.inv) p.inv[i] = pos;
        }
        __syncthreads();
    }
}

__global__ void __launch_bounds__(1024) permute_kernel(PermuteParams p)
{
    pdl_trigger();
    pdl_wait();
    permute_block(p);
}

// Placement of at most 128 pairs (T <= 64) by one warp, with no block barrier.
// Pair i = 32k + lane sits in slice k.  Lane e (< E) keeps, per slice, the ballot
// of the lanes whose pair goes to expert e; their population counts give the
// expert's count, a warp scan over the lanes gives the offsets, and a pair's
// place is its expert's start of the slice plus the lanes of that expert below
// it in the slice.  Same result as permute_block.
//   dec (optional): the tokens' decisions in shared memory (e0, e1, pruned at 3 t)
//   instead of the routing outputs in global memory.
__device__ __forceinline__ void permute_warp(const PermuteParams &p, const int *dec = nullptr)
{
    const unsigned full = 0xffffffffu, lt = (1u << (threadIdx.x & 31)) - 1;
    const int lane = threadIdx.x & 31, NP = 2 * p.T, nk = (NP + 31) / 32, E = p.E;
    int key[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int i = 32 * k + lane;
        key[k] = -1;
        if (i < NP) {
            const int pr = dec ? dec[3 * (i >> 1) + 2] : (int)__ldcg(p.pruned + (i >> 1));
            const int e = dec ? dec[3 * (i >> 1) + (i & 1)] : __ldcg(p.idx + i);
            key[k] = ((i & 1) && pr) || pr == 2 ? -1 : e;
        }
    }
    unsigned mine[4] = {0u, 0u, 0u, 0u};  // lane e: ballot of expert e per slice
#pragma unroll
    for (int k = 0; k < 4; ++k)
        if (k < nk)
            for (int e = 0; e < E; ++e) {
                const unsigned b = __ballot_sync(full, key[k] == e);
                if (lane == e) mine[k] = b;
            }
    int cnt = 0, bits = 0;
#pragma unroll
    for (int k = 0; k < 4; ++k) cnt += __popc(mine[k]);
#pragma unroll
    for (int f = 0; f < kMaxE; ++f)
        if (f == lane) bits = p.bits[f];
    int incl = cnt;  // inclusive scan of the counts over the lanes (experts)
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
        const int v = __shfl_up_sync(full, incl, d);
        if (lane >= d) incl += v;
    }
    const int off = incl - cnt;
    // the index of expert `lane`'s first work chunk in the order the expert
    // kernels take them (more bits first, then by expert), and the chunk total
    const int nch = (cnt + p.chunk - 1) / p.chunk;
    int k0 = 0, nchunks = 0;
    for (int f = 0; f < E; ++f) {
        const int nf = __shfl_sync(full, nch, f), bf = __shfl_sync(full, bits, f);
        nchunks += nf;
        if (bf > bits || (bf == bits && f < lane)) k0 += nf;
    }
    if (lane < E) {
        p.offsets[lane] = off;
        if (lane == E - 1) p.offsets[E] = incl;
        if (p.chunks)
            for (int c = 0, k = k0; c < cnt; c += p.chunk, ++k) {
                ChunkInfo ci;
                ci.e = lane;
                ci.pair_base = off + c;
                ci.nv = min(p.chunk, cnt - c);
                ci.bits = bits;
                p.chunks[k] = ci;
            }
    }
    if (lane == 0 && p.chunks) {
        *p.nchunks = nchunks;
        for (int i = 0; i < 4; ++i) p.counters[i] = 0;
    }
    int start = off;  // lane e: where expert e's pairs of the current slice begin
#pragma unroll
    for (int k = 0; k < 4; ++k)
        if (k < nk) {
            const int e = key[k], src = e >= 0 ? e : 0;
            const int s0 = __shfl_sync(full, start, src);
            const unsigned b = __shfl_sync(full, mine[k], src);
            const int i = 32 * k + lane, pos = e >= 0 ? s0 + __popc(b & lt) : -1;
            if (e >= 0) p.perm[pos] = i;
            if (p.inv && i < NP) p.inv[i] = pos;
            start += __popc(mine[k]);
        }
}

// Routing of token blockIdx.x, then the last CTA to finish (counted on *done,
// which it resets) places the pairs: one launch instead of two for small T.
template <bool NORM>
__global__ void __launch_bounds__(kRouteThreads) route_permute_kernel(RouteParams rp, PermuteParams pp, int32_t *done)
{
    __shared__ int last;
    pdl_trigger();
    pdl_wait();
    route_token<NORM>(rp, blockIdx.x);
    __syncthreads();
    if (threadIdx.x == 0) {
        // thread 0 wrote this CTA's routing outputs: the release orders them before
        // the count, the acquire makes the other CTAs' outputs visible to the last
        int prev;
        asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(prev) : "l"(done) : "memory");
        last = prev == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (!last || threadIdx.x >= 32) return;
    permute_warp(pp);  // T <= 64 here
    if (threadIdx.x == 0) *done = 0;
}

// Routing and placement of up to kClusterMaxT tokens as one thread-block cluster
// (one CTA per token): each CTA's decision also goes into CTA 0's shared memory,
// a cluster barrier (release / acquire) replaces the global arrival count, and
// CTA 0 places the pairs from its shared memory.
constexpr int kClusterMaxT = 16;

template <bool NORM>
__global__ void __launch_bounds__(kRouteThreads) route_cluster_kernel(RouteParams rp, PermuteParams pp)
{
    __shared__ int dec_s[3 * kClusterMaxT];
    namespace cg = cooperative_groups;
    cg::cluster_group cl = cg::this_cluster();
    int *sink = cl.map_shared_rank(dec_s, 0);
    pdl_trigger();
    pdl_wait();
    route_token<NORM>(rp, blockIdx.x, sink);
    cl.sync();
    if (cl.block_rank() != 0 || threadIdx.x >= 32) return;
    permute_warp(pp, dec_s);
}

// The arrival count of mc_route's single-launch routing (kDebugRouteFused): one
// word owned by the library, zero between launches (the last CTA resets it), so
// such calls must not overlap in time on one device.
__device__ int32_t g_route_done;

int32_t *route_done_word()
{
    void *p = nullptr;
    return cudaGetSymbolAddress(&p, g_route_done) == cudaSuccess ? (int32_t *)p : nullptr;
}

int max_chunks_for(int T, int E) { return (2 * T + kChunk - 1) / kChunk + E; }

// One cluster of T CTAs (T <= kClusterMaxT; above 8 a non-portable cluster size).
template <bool NORM>
static cudaError_t launch_route_cluster(const RouteParams &rp, const PermuteParams &pp, size_t smem, cudaStream_t st)
{
    cudaError_t err = cudaFuncSetAttribute(route_cluster_kernel<NORM>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (err != cudaSuccess) return err;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(rp.T);
    cfg.blockDim = dim3(kRouteThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)rp.T;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, route_cluster_kernel<NORM>, rp, pp);
}

int launch_route(const RouteParams &rp, const PermuteParams &pp, cudaStream_t st, int32_t *done)
{
    // the pre-norm row (mc_stack_forward's layers) in dynamic shared memory
    const size_t norm_smem = rp.h_in ? (size_t)rp.H * 2 : 0;
    cudaError_t err;
    if (done && rp.T <= kClusterMaxT) {
        profile_begin(kKRoute, st);
        err = rp.h_in ? launch_route_cluster<true>(rp, pp, norm_smem, st) : launch_route_cluster<false>(rp, pp, 0, st);
        profile_end(kKRoute, st);
        if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "route launch: %s", cudaGetErrorString(err));
        return MC_OK;
    }
    if (done && rp.T <= 64) {
        profile_begin(kKRoute, st);
        err = rp.h_in ? launch_k(route_permute_kernel<true>, dim3(rp.T), dim3(kRouteThreads), norm_smem, st, rp, pp, done)
                      : launch_k(route_permute_kernel<false>, dim3(rp.T), dim3(kRouteThreads), 0, st, rp, pp, done);
        profile_end(kKRoute, st);
        if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "route launch: %s", cudaGetErrorString(err));
        return MC_OK;
    }
    profile_begin(kKRoute, st);
    err = rp.h_in ? launch_k(route_kernel<true>, dim3(rp.T), dim3(kRouteThreads), norm_smem, st, rp)
                  : launch_k(route_kernel<false>, dim3(rp.T), dim3(kRouteThreads), 0, st, rp);
    profile_end(kKRoute, st);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "route launch: %s", cudaGetErrorString(err));
    profile_begin(kKPermute, st);
    // one thread per pair (whole warps), at most 1024: fewer threads to synchronise for small T
    const int nt = min(1024, max(32, (2 * pp.T + 31) / 32 * 32));
    err = launch_k(permute_kernel, dim3(1), dim3(nt), 0, st, pp);
    profile_end(kKPermute, st);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "permute launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

}  // namespace mc
