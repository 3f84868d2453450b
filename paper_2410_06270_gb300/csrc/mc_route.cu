// mc_route.cu -- the gate of Eq. 1, top-2 selection with renormalised softmax
// weights, the ODP test of Eq. 5 with the token protection of Sec. 2.3.2, and the
// permutation of kept (token, slot) pairs by expert.
//
// route_kernel: one CTA of 4 warps per token; each warp takes a quarter of the
//   row (16-byte loads of x and of the gate rows), the partial logits meet in
//   shared memory and thread 0 takes the decision in fp32.
// permute_kernel: one CTA; histogram, exclusive scan and a stable placement with
//   __match_any_sync ranks, so the permutation is unique (ascending token within
//   an expert) and identical run to run.  It also lists the work chunks of the
//   expert kernels and resets their work counters.
#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"

namespace mc {

constexpr int kRouteWarps = 4;

// The logits of token t by the whole CTA; thread 0 takes the decision and writes
// the outputs.
__device__ __forceinline__ void route_token(const RouteParams &p, int t)
{
    __shared__ float part[kRouteWarps][kMaxE];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int H = p.H, E = p.E;
    const __nv_bfloat16 *xr = p.x + (size_t)t * H;
    float acc[kMaxE];
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) acc[e] = 0.f;
    // unrolled so that the loads of several 1024-column steps are in flight together
#pragma unroll 4
    for (int c0 = 8 * (threadIdx.x); c0 < H; c0 += 8 * 32 * kRouteWarps) {
        uint4 raw = *reinterpret_cast<const uint4 *>(xr + c0);
        const __nv_bfloat162 *x2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
        float xf[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float2 f = __bfloat1622float2(x2[i]);
            xf[2 * i] = f.x;
            xf[2 * i + 1] = f.y;
        }
#pragma unroll
        for (int e = 0; e < kMaxE; ++e) {
            if (e < E) {
                uint4 gr = *reinterpret_cast<const uint4 *>(p.gate + (size_t)e * H + c0);
                const __nv_bfloat162 *g2 = reinterpret_cast<const __nv_bfloat162 *>(&gr);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    float2 gf = __bfloat1622float2(g2[i]);
                    acc[e] = fmaf(xf[2 * i], gf.x, acc[e]);
                    acc[e] = fmaf(xf[2 * i + 1], gf.y, acc[e]);
                }
            }
        }
    }
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) {
        for (int m = 16; m >= 1; m >>= 1) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], m);
        if (lane == 0) part[warp][e] = acc[e];
    }
    __syncthreads();
    if (threadIdx.x != 0) return;  // (route_token returns to its caller; the CTA re-joins there)
    float l[kMaxE];
    for (int e = 0; e < E; ++e) {
        float s = 0.f;
        for (int w = 0; w < kRouteWarps; ++w) s += part[w][e];
        l[e] = s;
    }
    // top-2 on fp32 logits, lower index wins ties
    int e0 = 0;
    for (int e = 1; e < E; ++e)
        if (l[e] > l[e0]) e0 = e;
    int e1 = e0 == 0 ? 1 : 0;
    for (int e = 0; e < E; ++e)
        if (e != e0 && l[e] > l[e1]) e1 = e;
    const float d = l[e0] - l[e1];  // >= 0
    const float r = __expf(-d);     // = p1 / p0
    float w0 = 1.f / (1.f + r), w1 = r / (1.f + r);
    const bool prot = p.protect != nullptr && p.protect[t] != 0;
    const bool prune = !prot && (d > p.neg_log_mu);
    if (prune) {
        w0 = 1.f;
        w1 = 0.f;
    }
    p.idx[2 * t] = e0;
    p.idx[2 * t + 1] = e1;
    p.w[2 * t] = w0;
    p.w[2 * t + 1] = w1;
    p.pruned[t] = prune ? 1 : 0;
    if (p.idx_out) {
        p.idx_out[2 * t] = e0;
        p.idx_out[2 * t + 1] = e1;
    }
    if (p.w_out) {
        p.w_out[2 * t] = w0;
        p.w_out[2 * t + 1] = w1;
    }
    if (p.pruned_out) p.pruned_out[t] = prune ? 1 : 0;
}

__global__ void __launch_bounds__(kRouteWarps * 32) route_kernel(RouteParams p) { route_token(p, blockIdx.x); }

// Histogram, scan, stable placement and work-chunk list by one CTA of any size
// (whole warps).
__device__ __forceinline__ void permute_block(const PermuteParams &p)
{
    __shared__ int cnt[kMaxE];
    __shared__ int run[kMaxE];
    __shared__ int wcnt[32][kMaxE];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int NP = 2 * p.T;
    if (tid < kMaxE) {
        cnt[tid] = 0;
        run[tid] = 0;
    }
    __syncthreads();
    for (int i = tid; i < NP; i += blockDim.x) {
        bool kept = !((i & 1) && __ldcg(p.pruned + (i >> 1)));
        if (kept) atomicAdd(&cnt[__ldcg(p.idx + i)], 1);
    }
    __syncthreads();
    if (tid == 0) {
        int s = 0;
        for (int e = 0; e < p.E; ++e) {
            p.offsets[e] = s;
            run[e] = s;
            s += cnt[e];
        }
        p.offsets[p.E] = s;
        if (p.chunks) {
            // work chunks of <= p.chunk pairs, experts with more bits first
            int k = 0;
            for (int b = 3; b >= 1; --b)
                for (int e = 0; e < p.E; ++e) {
                    if (p.bits[e] != b) continue;
                    for (int c = 0; c < cnt[e]; c += p.chunk) {
                        ChunkInfo ci;
                        ci.e = e;
                        ci.pair_base = run[e] + c;
                        ci.nv = min(p.chunk, cnt[e] - c);
                        ci.bits = b;
                        p.chunks[k++] = ci;
                    }
                }
            *p.nchunks = k;
            for (int i = 0; i < 4; ++i) p.counters[i] = 0;
        }
    }
    __syncthreads();
    for (int base = 0; base < NP; base += blockDim.x) {
        int i = base + tid;
        int key = -1;
        if (i < NP) {
            bool kept = !((i & 1) && __ldcg(p.pruned + (i >> 1)));
            key = kept ? __ldcg(p.idx + i) : -1;
        }
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

__global__ void __launch_bounds__(1024) permute_kernel(PermuteParams p) { permute_block(p); }

// Routing of token blockIdx.x, then the last CTA to finish (counted on *done,
// which it resets) places the pairs: one launch instead of two for small T.
__global__ void __launch_bounds__(kRouteWarps * 32) route_permute_kernel(RouteParams rp, PermuteParams pp, int32_t *done)
{
    __shared__ int last;
    route_token(rp, blockIdx.x);
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();  // this CTA's routing outputs before the count
        last = atomicAdd(done, 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    permute_block(pp);
    if (threadIdx.x == 0) *done = 0;
}

int max_chunks_for(int T, int E) { return (2 * T + kChunk - 1) / kChunk + E; }

int launch_route(const RouteParams &rp, const PermuteParams &pp, cudaStream_t st, int32_t *done)
{
    if (done && rp.T <= 64) {
        profile_begin(kKRoute, st);
        route_permute_kernel<<<rp.T, kRouteWarps * 32, 0, st>>>(rp, pp, done);
        profile_end(kKRoute, st);
        cudaError_t err = cudaGetLastError();
        if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "route launch: %s", cudaGetErrorString(err));
        return MC_OK;
    }
    profile_begin(kKRoute, st);
    route_kernel<<<rp.T, kRouteWarps * 32, 0, st>>>(rp);
    profile_end(kKRoute, st);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "route launch: %s", cudaGetErrorString(err));
    profile_begin(kKPermute, st);
    // one thread per pair (whole warps), at most 1024: fewer threads to synchronise for small T
    const int nt = min(1024, max(32, (2 * pp.T + 31) / 32 * 32));
    permute_kernel<<<1, nt, 0, st>>>(pp);
    profile_end(kKPermute, st);
    err = cudaGetLastError();
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "permute launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

}  // namespace mc
