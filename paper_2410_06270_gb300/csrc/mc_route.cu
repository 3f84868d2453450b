// mc_route.cu -- the gate of Eq. 1, top-2 selection with renormalised softmax
// weights, the ODP test of Eq. 5 with the token protection of Sec. 2.3.2, and the
// permutation of kept (token, slot) pairs by expert.
//
// route_kernel: one warp per token.  The warp streams the token's bf16 row once
// (16-byte loads) and, in the same pass, writes the fp16 copy the expert kernels
// consume plus the per-group offset tables of mc_layout.h.
// permute_kernel: one CTA; histogram, exclusive scan and a stable placement with
// __match_any_sync ranks, so the permutation is unique (ascending token within an
// expert) and identical run to run.
#include "mc_kernels.h"

namespace mc {

__global__ void __launch_bounds__(256) route_kernel(RouteParams p)
{
    const int lane = threadIdx.x & 31;
    const int t = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (t >= p.T) return;
    const int H = p.H, E = p.E;
    const __nv_bfloat16 *xr = p.x + (size_t)t * H;
    float acc[kMaxE];
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) acc[e] = 0.f;
    bool bad = false;
    // lanes of one half-warp cover 128 consecutive columns per iteration; every
    // lane runs every iteration (H is a multiple of 128, not always of 256)
    for (int it = 0; it < (H + 255) / 256; ++it) {
        const int c0 = it * 256 + 8 * lane;
        const bool act = c0 < H;
        uint4 raw = act ? *reinterpret_cast<const uint4 *>(xr + c0) : make_uint4(0, 0, 0, 0);
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
            if (e < E && act) {
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
        if (p.xh) {
            // fp16 copy for the tensor-core expert kernels + offset tables
            __half hv[8];
            float tab[7] = {0, 0, 0, 0, 0, 0, 0};
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (!(fabsf(xf[i]) <= 65504.f)) bad = true;
                hv[i] = __float2half_rn(xf[i]);
                float v = __half2float(hv[i]);
                int col = (c0 + i) & (kTileK - 1);
                int j0 = pair_of_col(col, 0), j1 = pair_of_col(col, 1);
                tab[0] += v;
                tab[1] = fmaf(off1(j0), v, tab[1]);
                tab[2] = fmaf(off1(j1), v, tab[2]);
                tab[3] = fmaf(off2(j0), v, tab[3]);
                tab[4] = fmaf(off2(j1), v, tab[4]);
            }
            if (act) *reinterpret_cast<uint4 *>(p.xh + (size_t)t * H + c0) = *reinterpret_cast<uint4 *>(hv);
            // reduce over the lanes sharing a quantisation group (8 cols per lane)
            const int lanes_per_group = p.group / 8;  // 8 or 16
#pragma unroll
            for (int k = 0; k < 5; ++k)
                for (int m = 1; m < lanes_per_group; m <<= 1) tab[k] += __shfl_xor_sync(0xffffffffu, tab[k], m);
            if (act && (lane & (lanes_per_group - 1)) == 0) {
                int G = c0 / p.group, ng = H / p.group;
                float4 *dst = reinterpret_cast<float4 *>(p.xtab + ((size_t)t * ng + G) * kTabFloats);
                dst[0] = make_float4(tab[0], tab[1], tab[2], tab[3]);
                dst[1] = make_float4(tab[4], tab[3] + 4.f * tab[1], tab[4] + 4.f * tab[2], 0.f);
            }
        }
    }
#pragma unroll
    for (int e = 0; e < kMaxE; ++e)
        for (int m = 16; m >= 1; m >>= 1) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], m);
    if (p.xh && __any_sync(0xffffffffu, bad) && lane == 0) set_status(p.status, MC_ERR_RANGE);
    if (lane != 0) return;
    // top-2 on fp32 logits, lower index wins ties
    int e0 = 0;
    for (int e = 1; e < E; ++e)
        if (acc[e] > acc[e0]) e0 = e;
    int e1 = e0 == 0 ? 1 : 0;
    for (int e = 0; e < E; ++e)
        if (e != e0 && acc[e] > acc[e1]) e1 = e;
    float d = acc[e0] - acc[e1];  // >= 0
    float r = __expf(-d);         // = p1 / p0
    float w0 = 1.f / (1.f + r), w1 = r / (1.f + r);
    bool prot = p.protect != nullptr && p.protect[t] != 0;
    bool prune = !prot && (d > p.neg_log_mu);
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

__global__ void __launch_bounds__(1024) permute_kernel(PermuteParams p)
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
        bool kept = !((i & 1) && p.pruned[i >> 1]);
        if (kept) atomicAdd(&cnt[p.idx[i]], 1);
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
    }
    __syncthreads();
    for (int base = 0; base < NP; base += blockDim.x) {
        int i = base + tid;
        int key = -1;
        if (i < NP) {
            bool kept = !((i & 1) && p.pruned[i >> 1]);
            key = kept ? p.idx[i] : -1;
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

}  // namespace mc
