// mc_gemv.cu -- decode-path expert kernels: mixed-bit (1/2/3-bit) grouped
// dequant-GEMV over the SwiGLU experts (Eq. 1's E_i on PMQ weights, Sec. 2.2).
//
// gemv_w13_kernel: one CTA per (expert, 128 rows of W1 and the same 128 rows of
//   W3); h = silu(W1 x) * (W3 x) for every pair routed to the expert, written in
//   fp16 (pair order) together with the per-group offset tables of h for W2.
// gemv_w2_kernel: one CTA per (expert, 256 rows of W2, column split); writes the
//   fp32 expert outputs of its split.
//
// Work per CTA: a producer warp streams the packed 128x128 supertiles of both
// row streams with cp.async.bulk into a 4-stage shared-memory ring (mbarrier
// completion, L2 evict-first).  Eight consumer warps each own one 16-row tile of
// every supertile: the lane's code words become fp16 mma.sync A fragments with
// one LOP3 per register (mc_layout.h), multiply fp16 activations held in shared
// memory in fragment order, and are folded per quantisation group:
//   y += s * (acc - O - z * X)
// where acc = sum_k (off_k + q_k) x_k, O = sum_k off_k x_k and X = sum_k x_k,
// which equals s * sum_k (q_k - z) x_k, the group-wise dequantised product.
// The decode path is bound by HBM bandwidth on the packed weight bytes.
#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"

namespace mc {

constexpr int kStages = 4;
constexpr int kConsumerWarps = 8;
constexpr int kGemvThreads = (kConsumerWarps + 1) * 32;

struct GemvLayout {
    int st_max;       // bytes of one stream buffer in a stage
    int nkt;          // column tiles handled by the CTA
    int ng_loc;       // quantisation groups handled by the CTA
    size_t off_stage, off_bfrag, off_tab, off_hs, total;
};

template <int NT>
__host__ __device__ inline GemvLayout gemv_layout(int group, int nkt)
{
    GemvLayout L;
    L.st_max = supertile_bytes(3, group);
    L.nkt = nkt;
    L.ng_loc = nkt * (kTileK / group);
    L.off_stage = 256;
    L.off_bfrag = L.off_stage + (size_t)kStages * 2 * L.st_max;
    L.off_tab = L.off_bfrag + (size_t)nkt * 8 * NT * 32 * sizeof(uint2);
    L.off_hs = L.off_tab + (size_t)8 * NT * L.ng_loc * kTabFloats * sizeof(float);
    L.total = L.off_hs + (size_t)8 * NT * kTileK * sizeof(__half);
    return L;
}

__host__ __device__ inline int w2_split_tiles(const ExpertParams &p) { return (p.F / kTileK) / p.KS; }

size_t gemv_smem_bytes(int NT, bool w13, const ExpertParams &p)
{
    int nkt = w13 ? p.H / kTileK : w2_split_tiles(p);
    return NT == 1 ? gemv_layout<1>(p.group, nkt).total : gemv_layout<2>(p.group, nkt).total;
}

struct Shared {
    volatile int abort;
    volatile int issued;
    int tok[16];
};

// Bounded wait that also gives up as soon as another thread of the CTA aborted.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, const ExpertParams &p, Shared *sh)
{
    if (mbar_try_wait(bar, parity)) return true;
    uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (sh->abort) return false;
        if (globaltimer_ns() - t0 > p.timeout_ns) {
            set_status(p.status, MC_ERR_TIMEOUT);
            sh->abort = 1;
            return false;
        }
    }
}

// One pair of row streams (A, B) of one expert over column tiles [kt0, kt0+nkt).
// W13: A = W1 rows, B = W3 rows of 128-row block blkA (== blkB); vectors are the
//      routed tokens' fp16 activations.
// W2:  A, B = W2 row blocks blkA, blkB (blkB < 0: none); vectors are h.
template <int NT, int BITS, bool W13>
__device__ __forceinline__ void gemv_body(const ExpertParams &p, uint8_t *smem, int e, int blkA, int blkB,
                                          int kt0, int nkt, int ks)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int group = p.group, gpt = kTileK / group;
    const GemvLayout L = gemv_layout<NT>(group, nkt);
    const int TB = tile_bytes(BITS, group), STB = kTilesPerBlock * TB;
    const int KTtot = W13 ? p.H / kTileK : p.F / kTileK;
    const int ng_vec = (W13 ? p.H : p.F) / group;  // groups per vector row
    const uint8_t *matA = p.packed + p.mat_off[e][W13 ? 0 : 2];
    const uint8_t *matB = p.packed + p.mat_off[e][W13 ? 1 : 2];
    const bool hasB = blkB >= 0;

    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    uint64_t *empty = full + kStages;
    Shared *sh = reinterpret_cast<Shared *>(smem + 128);
    uint8_t *stage = smem + L.off_stage;
    uint2 *bfrag = reinterpret_cast<uint2 *>(smem + L.off_bfrag);
    float *tab = reinterpret_cast<float *>(smem + L.off_tab);
    __half *hs = reinterpret_cast<__half *>(smem + L.off_hs);

    const int base = p.offsets[e];
    const int Te = p.offsets[e + 1] - base;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kConsumerWarps);
        }
        sh->abort = 0;
        sh->issued = 0;
        fence_mbar_init();
    }
    __syncthreads();

    int itbase = 0;
    for (int c0 = 0; c0 < Te; c0 += 8 * NT, itbase += nkt) {
        const int nv = min(8 * NT, Te - c0);
        if (warp == kConsumerWarps) {
            // ------------------------------------------------------ producer --
            if (lane == 0 && !(p.debug & kDebugNoProducer)) {
                const uint64_t pol = policy_evict_first();
                for (int i = 0; i < nkt; ++i) {
                    const int it = itbase + i, s = it % kStages;
                    if (it >= kStages && !wait_or_abort(&empty[s], ((it / kStages) - 1) & 1, p, sh)) break;
                    const int kt = kt0 + i;
                    mbar_arrive_expect_tx(&full[s], hasB ? 2 * STB : STB);
                    bulk_g2s_stream(stage + (size_t)s * 2 * L.st_max,
                                    matA + ((size_t)blkA * KTtot + kt) * STB, STB, &full[s], pol);
                    if (hasB)
                        bulk_g2s_stream(stage + (size_t)s * 2 * L.st_max + L.st_max,
                                        matB + ((size_t)blkB * KTtot + kt) * STB, STB, &full[s], pol);
                    sh->issued = it + 1;
                }
            }
        } else {
            // ------------------------------------------------------ consumers --
            const int ctid = threadIdx.x;
            if (ctid < 8 * NT) {
                int q = base + c0 + ctid;
                sh->tok[ctid] = ctid < nv ? (W13 ? (p.perm[q] >> 1) : q) : -1;
            }
            named_bar_sync(1, kConsumerWarps * 32);
            // activations in mma B-fragment order: [i][s][j][lane] -> 4 fp16
            const int nfrag = nkt * 8 * NT * 32;
            for (int f = ctid; f < nfrag; f += kConsumerWarps * 32) {
                const int ln = f & 31, j = (f >> 5) % NT, s = ((f >> 5) / NT) & 7, i = ((f >> 5) / NT) >> 3;
                const int n = 8 * j + (ln >> 2), t = ln & 3;
                const int col = (kt0 + i) * kTileK + 64 * (s >> 2) + 16 * t + 4 * (s & 3);
                const int v = sh->tok[n];
                uint2 val = make_uint2(0, 0);
                if (v >= 0) {
                    const __half *row = W13 ? p.xh + (size_t)v * p.H : p.h + (size_t)v * p.F;
                    val = *reinterpret_cast<const uint2 *>(row + col);
                }
                bfrag[f] = val;
            }
            for (int f = ctid; f < 8 * NT * L.ng_loc; f += kConsumerWarps * 32) {
                const int n = f / L.ng_loc, gl = f % L.ng_loc;
                const int v = sh->tok[n];
                float4 a = make_float4(0, 0, 0, 0), b = a;
                if (v >= 0) {
                    const float *src = (W13 ? p.xtab : p.htab) + ((size_t)v * ng_vec + kt0 * gpt + gl) * kTabFloats;
                    a = *reinterpret_cast<const float4 *>(src);
                    b = *reinterpret_cast<const float4 *>(src + 4);
                }
                reinterpret_cast<float4 *>(tab + (size_t)f * kTabFloats)[0] = a;
                reinterpret_cast<float4 *>(tab + (size_t)f * kTabFloats)[1] = b;
            }
            named_bar_sync(1, kConsumerWarps * 32);

            float y[2][NT][4], acc[2][NT][4];
#pragma unroll
            for (int x = 0; x < 2; ++x)
#pragma unroll
                for (int j = 0; j < NT; ++j)
#pragma unroll
                    for (int c = 0; c < 4; ++c) y[x][j][c] = acc[x][j][c] = 0.f;

            const int oa = 2 * BITS - 1;  // offset-table index for row half 0 (half 1: oa + 1)
            for (int i = 0; i < nkt; ++i) {
                const int it = itbase + i, s = it % kStages;
                if (!wait_or_abort(&full[s], (it / kStages) & 1, p, sh)) break;
                const uint8_t *tA = stage + (size_t)s * 2 * L.st_max + warp * TB;
                const uint8_t *tB = tA + L.st_max;
                uint32_t c2[2][4], c1[2][2];
                uint2 meta[2][2];
#pragma unroll
                for (int x = 0; x < 2; ++x) {
                    const uint8_t *tt = x ? tB : tA;
                    if (BITS >= 2) {
                        uint4 v = *reinterpret_cast<const uint4 *>(tt + 16 * lane);
                        c2[x][0] = v.x; c2[x][1] = v.y; c2[x][2] = v.z; c2[x][3] = v.w;
                    }
                    if (BITS != 2) {
                        uint2 v = *reinterpret_cast<const uint2 *>(tt + (BITS == 3 ? 512 : 0) + 8 * lane);
                        c1[x][0] = v.x; c1[x][1] = v.y;
                    }
                    const uint8_t *mt = tt + tile_code_bytes(BITS);
                    meta[x][0] = *reinterpret_cast<const uint2 *>(mt + (lane >> 2) * 8);
                    meta[x][1] = gpt == 2 ? *reinterpret_cast<const uint2 *>(mt + 64 + (lane >> 2) * 8) : meta[x][0];
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&empty[s]);

#pragma unroll
                for (int qd = 0; qd < 4; ++qd) {
                    uint32_t r[2][8], rh[2][8];
#pragma unroll
                    for (int x = 0; x < 2; ++x) {
                        if (BITS == 1) cvt1_half<false>(c1[x][qd >> 1], 8 * (qd & 1), r[x]);
                        if (BITS >= 2) cvt2(c2[x][qd], r[x]);
                        if (BITS == 3) cvt1_half<true>(c1[x][qd >> 1], 8 * (qd & 1), rh[x]);
                    }
#pragma unroll
                    for (int kk = 0; kk < 2; ++kk) {
                        const int sidx = 2 * qd + kk;
#pragma unroll
                        for (int j = 0; j < NT; ++j) {
                            const uint2 b = bfrag[((i * 8 + sidx) * NT + j) * 32 + lane];
#pragma unroll
                            for (int x = 0; x < 2; ++x) {
                                if (x == 1 && !hasB) continue;
                                mma16816(acc[x][j], r[x][4 * kk], r[x][4 * kk + 1], r[x][4 * kk + 2],
                                         r[x][4 * kk + 3], b.x, b.y);
                                if (BITS == 3)
                                    mma16816(acc[x][j], rh[x][4 * kk], rh[x][4 * kk + 1], rh[x][4 * kk + 2],
                                             rh[x][4 * kk + 3], b.x, b.y);
                            }
                        }
                        // group boundary: fold the accumulators (see file header)
                        if ((sidx == 3 && gpt == 2) || sidx == 7) {
                            const int gi = sidx == 3 ? 0 : gpt - 1;
                            const int gl = i * gpt + gi;
#pragma unroll
                            for (int x = 0; x < 2; ++x) {
                                const __half2 *m2 = reinterpret_cast<const __half2 *>(&meta[x][gi]);
                                const float2 sz0 = __half22float2(m2[0]), sz1 = __half22float2(m2[1]);
#pragma unroll
                                for (int j = 0; j < NT; ++j) {
                                    const int n0 = 8 * j + 2 * (lane & 3);
                                    const float *T0 = tab + ((size_t)n0 * L.ng_loc + gl) * kTabFloats;
                                    const float *T1 = T0 + (size_t)L.ng_loc * kTabFloats;
                                    const float X0 = T0[0], X1 = T1[0];
                                    y[x][j][0] += sz0.x * (acc[x][j][0] - T0[oa] - sz0.y * X0);
                                    y[x][j][1] += sz0.x * (acc[x][j][1] - T1[oa] - sz0.y * X1);
                                    y[x][j][2] += sz1.x * (acc[x][j][2] - T0[oa + 1] - sz1.y * X0);
                                    y[x][j][3] += sz1.x * (acc[x][j][3] - T1[oa + 1] - sz1.y * X1);
#pragma unroll
                                    for (int c = 0; c < 4; ++c) acc[x][j][c] = 0.f;
                                }
                            }
                        }
                    }
                }
            }

            // ------------------------------------------------------ epilogue --
            const int g8 = lane >> 2, t2 = 2 * (lane & 3);
            if (W13) {
                const int F = p.F;
#pragma unroll
                for (int j = 0; j < NT; ++j)
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const int n = 8 * j + t2 + (c & 1);
                        const int r = warp * 16 + g8 + 8 * (c >> 1);
                        const __half hv = __float2half_rn(silu(y[0][j][c]) * y[1][j][c]);
                        hs[n * kTileK + r] = hv;
                        if (n < nv) p.h[(size_t)(base + c0 + n) * F + (size_t)blkA * kTileK + r] = hv;
                    }
                named_bar_sync(1, kConsumerWarps * 32);
                // offset tables of h for the W2 pass (same definitions as for x)
                for (int item = warp; item < nv * gpt; item += kConsumerWarps) {
                    const int n = item / gpt, gi = item % gpt;
                    float tb[5] = {0, 0, 0, 0, 0};
                    for (int c = gi * group + lane; c < (gi + 1) * group; c += 32) {
                        const float v = __half2float(hs[n * kTileK + c]);
                        const int j0 = pair_of_col(c, 0), j1 = pair_of_col(c, 1);
                        tb[0] += v;
                        tb[1] = fmaf(off1(j0), v, tb[1]);
                        tb[2] = fmaf(off1(j1), v, tb[2]);
                        tb[3] = fmaf(off2(j0), v, tb[3]);
                        tb[4] = fmaf(off2(j1), v, tb[4]);
                    }
#pragma unroll
                    for (int k = 0; k < 5; ++k)
#pragma unroll
                        for (int m = 16; m >= 1; m >>= 1) tb[k] += __shfl_xor_sync(0xffffffffu, tb[k], m);
                    if (lane == 0) {
                        float4 *dst = reinterpret_cast<float4 *>(
                            p.htab + ((size_t)(base + c0 + n) * (F / group) + (size_t)blkA * gpt + gi) * kTabFloats);
                        dst[0] = make_float4(tb[0], tb[1], tb[2], tb[3]);
                        dst[1] = make_float4(tb[4], tb[3] + 4.f * tb[1], tb[4] + 4.f * tb[2], 0.f);
                    }
                }
            } else {
                const int H = p.H;
                float *out = p.opart + (size_t)ks * p.Pmax * H;
#pragma unroll
                for (int x = 0; x < 2; ++x) {
                    if (x == 1 && !hasB) continue;
                    const int blk = x ? blkB : blkA;
#pragma unroll
                    for (int j = 0; j < NT; ++j)
#pragma unroll
                        for (int c = 0; c < 4; ++c) {
                            const int n = 8 * j + t2 + (c & 1);
                            const int r = blk * kTileK + warp * 16 + g8 + 8 * (c >> 1);
                            if (n < nv) out[(size_t)(base + c0 + n) * H + r] = y[x][j][c];
                        }
                }
            }
        }
        __syncthreads();
        if (sh->abort) break;
    }
    // On an abort, let copies that were issued but never consumed land before the
    // CTA's shared memory is released (bounded).
    if (threadIdx.x == 0 && sh->abort) {
        const int total_it = itbase;
        for (int it = max(0, sh->issued - kStages); it < sh->issued && it < total_it; ++it) {
            uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(&full[it % kStages], (it / kStages) & 1))
                if (globaltimer_ns() - t0 > p.timeout_ns) break;
        }
    }
}

// The packed buffer must carry the header written for this shape and bit table:
// the expert's bit width and the byte offsets of its matrices (which depend on
// every earlier expert's width) must match what the host computed, so a CTA never
// reads outside the region the buffer was packed with.
__device__ __forceinline__ bool header_ok(const ExpertParams &p, int e)
{
    const PackHeader *hd = reinterpret_cast<const PackHeader *>(p.packed);
    const bool ok = hd->magic == kMagic && hd->version == kFormatVersion && hd->E == p.E && hd->H == p.H &&
                    hd->F == p.F && hd->group == p.group && hd->bits[e] == p.bits[e] &&
                    hd->mat_off[e][0] == p.mat_off[e][0] && hd->mat_off[e][1] == p.mat_off[e][1] &&
                    hd->mat_off[e][2] == p.mat_off[e][2];
    if (!ok && threadIdx.x == 0) set_status(p.status, MC_ERR_BAD_PACK);
    return ok;
}

template <int NT>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_w13_kernel(ExpertParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    const int RBF = p.F / kBlockRows;
    const int e = blockIdx.x / RBF, rb = blockIdx.x % RBF;
    if (p.offsets[e + 1] == p.offsets[e]) return;
    if (!header_ok(p, e)) return;
    const int nkt = p.H / kTileK;
    switch (p.bits[e]) {
    case 1: gemv_body<NT, 1, true>(p, smem, e, rb, rb, 0, nkt, 0); break;
    case 2: gemv_body<NT, 2, true>(p, smem, e, rb, rb, 0, nkt, 0); break;
    case 3: gemv_body<NT, 3, true>(p, smem, e, rb, rb, 0, nkt, 0); break;
    default: set_status(p.status, MC_ERR_BAD_PACK);
    }
}

template <int NT>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_w2_kernel(ExpertParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    const int nrb = p.H / kBlockRows, npair = (nrb + 1) / 2;
    const int per_e = npair * p.KS;
    const int e = blockIdx.x / per_e, rem = blockIdx.x % per_e;
    const int pr = rem / p.KS, ks = rem % p.KS;
    if (p.offsets[e + 1] == p.offsets[e]) return;
    if (!header_ok(p, e)) return;
    const int blkA = 2 * pr, blkB = 2 * pr + 1 < nrb ? 2 * pr + 1 : -1;
    const int nkt = w2_split_tiles(p);
    switch (p.bits[e]) {
    case 1: gemv_body<NT, 1, false>(p, smem, e, blkA, blkB, ks * nkt, nkt, ks); break;
    case 2: gemv_body<NT, 2, false>(p, smem, e, blkA, blkB, ks * nkt, nkt, ks); break;
    case 3: gemv_body<NT, 3, false>(p, smem, e, blkA, blkB, ks * nkt, nkt, ks); break;
    default: set_status(p.status, MC_ERR_BAD_PACK);
    }
}

template <int NT>
static int launch_gemv_nt(const ExpertParams &ep, cudaStream_t st)
{
    const size_t sm13 = gemv_smem_bytes(NT, true, ep), sm2 = gemv_smem_bytes(NT, false, ep);
    int dev = 0, maxsm = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&maxsm, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "device query: %s", cudaGetErrorString(err));
    if (sm13 > (size_t)maxsm || sm2 > (size_t)maxsm)
        return set_error(MC_ERR_UNSUPPORTED, "GEMV path needs %zu/%zu bytes of shared memory (device: %d)", sm13,
                         sm2, maxsm);
    err = cudaFuncSetAttribute(gemv_w13_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm13);
    if (err == cudaSuccess)
        err = cudaFuncSetAttribute(gemv_w2_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm2);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(err));
    const int g13 = ep.E * (ep.F / kBlockRows);
    const int g2 = ep.E * (((ep.H / kBlockRows) + 1) / 2) * ep.KS;
    profile_begin(kKGemvW13, st);
    gemv_w13_kernel<NT><<<g13, kGemvThreads, sm13, st>>>(ep);
    profile_end(kKGemvW13, st);
    err = cudaGetLastError();
    if (err == cudaSuccess) {
        profile_begin(kKGemvW2, st);
        gemv_w2_kernel<NT><<<g2, kGemvThreads, sm2, st>>>(ep);
        profile_end(kKGemvW2, st);
        err = cudaGetLastError();
    }
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "GEMV launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

int launch_gemv(const ExpertParams &ep, int NT, cudaStream_t st)
{
    return NT == 1 ? launch_gemv_nt<1>(ep, st) : launch_gemv_nt<2>(ep, st);
}

int launch_combine(const CombineParams &cp, cudaStream_t st)
{
    const int n = cp.T * (cp.H / 8);
    profile_begin(kKCombine, st);
    combine_kernel<<<(n + 255) / 256, 256, 0, st>>>(cp);
    profile_end(kKCombine, st);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "combine launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

// ---------------------------------------------------------------- combine --
// y[t] = w0 * o[p(t,0)] + w1 * o[p(t,1)] (second term absent when pruned),
// summing the column splits of the W2 pass in a fixed order (Eq. 1 with Eq. 5).
__global__ void __launch_bounds__(256) combine_kernel(CombineParams p)
{
    const int H8 = p.H / 8;
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= p.T * H8) return;
    const int t = idx / H8, c = (idx % H8) * 8;
    float out[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int slot = 0; slot < 2; ++slot) {
        const int q = p.inv[2 * t + slot];
        if (q < 0) continue;
        const float wt = p.w[2 * t + slot];
        float o[8] = {0, 0, 0, 0, 0, 0, 0, 0};
        for (int ks = 0; ks < p.KS; ++ks) {
            const float4 *src = reinterpret_cast<const float4 *>(p.opart + ((size_t)ks * p.Pmax + q) * p.H + c);
            float4 a = src[0], b = src[1];
            o[0] += a.x; o[1] += a.y; o[2] += a.z; o[3] += a.w;
            o[4] += b.x; o[5] += b.y; o[6] += b.z; o[7] += b.w;
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) out[k] = fmaf(wt, o[k], out[k]);
    }
    __nv_bfloat16 r[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) r[k] = __float2bfloat16_rn(out[k]);
    *reinterpret_cast<uint4 *>(p.y + (size_t)t * p.H + c) = *reinterpret_cast<uint4 *>(r);
}

}  // namespace mc
