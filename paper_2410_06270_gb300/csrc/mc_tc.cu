// mc_tc.cu -- expert kernels on the 5th-generation tensor cores (tcgen05):
// mixed-bit (1/2/3-bit) grouped dequant-GEMV/GEMM over the SwiGLU experts
// (Eq. 1's E_i on PMQ weights, Sec. 2.2), for chunks of up to 16 pairs.
//
// Per work item (a chunk of <= 16 pairs of one expert x 128 rows of one matrix,
// over a column range) a persistent CTA streams 128-column steps:
//   producer warp   cp.async.bulk of one ring stage:
//                   [activation tile: 16 pairs x 128 cols, fp16, SW128 image]
//                   [offset tables of the 16 pairs][packed 128x128 supertile]
//   8 converter warps  packed words -> fp16 (2^E + q) with one LOP3 per two
//                   weights, stored as SW128 A tiles (64-column atoms); the
//                   third bit of 3-bit codes goes to a second A tile weighted x4
//   MMA thread      tcgen05.mma kind::f16, M = 128 rows, N = 16 pairs, K = 16,
//                   one TMEM accumulator per quantisation group
//   4 epilogue warps   thread = row: tcgen05.ld of the group accumulator and
//                   y += s * (acc - O - z * X)   (= s * sum_k (q_k - z) x_k)
// At the end of an item the rows' 16 results go to global memory: W1 / W3 gate
// and up values (SwiGLU is applied by frag_h_kernel), or W2 outputs.
#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"
#include "mc_umma.cuh"

namespace mc {

constexpr int kTcConv = 8;                    // converter warps  (0..7)
constexpr int kTcEpi0 = 8;                    // epilogue warps   (8..11)
constexpr int kTcProd = 12;                   // producer warp
constexpr int kTcMma = 13;                    // MMA warp
constexpr int kTcThreads = 14 * 32;
constexpr int kTcMaxSlots = 16;
constexpr int kTcNA = 3;                      // A atom buffers (16 KB each)
constexpr int kTcND = 8;                      // TMEM accumulators of 16 columns
constexpr int kABufBytes = 16384;
constexpr int kSlotBImg = 0;                  // 4096 B
constexpr int kSlotTab = 4096;                // <= 1024 B
constexpr int kSlotPack = 5120;               // <= 7168 B
constexpr int kTcSlotBytes = 12288;
constexpr int kTcHdr = 1024;                  // barriers + bookkeeping
constexpr int kTcABase = kTcHdr;              // A buffers (1024-aligned)
constexpr int kTcRingBase = kTcABase + kTcNA * kABufBytes;

__host__ __device__ inline size_t tc_smem(int nslots) { return (size_t)kTcRingBase + (size_t)nslots * kTcSlotBytes; }

struct TcShared {
    uint64_t full[kTcMaxSlots], empty[kTcMaxSlots];
    uint64_t a_full[kTcNA], a_empty[kTcNA];
    uint64_t d_full[kTcND], d_empty[kTcND];
    uint64_t drain;
    uint32_t tmem_base;
    volatile int abort;
    volatile int issued;
    int slot_item[kTcMaxSlots];
    int slot_i[kTcMaxSlots];
};
static_assert(sizeof(TcShared) <= kTcHdr, "header");

__device__ __forceinline__ bool tc_wait(uint64_t *bar, uint32_t parity, const ExpertParams &p, TcShared *sh)
{
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait_sleep(bar, parity, kWaitHintNs)) return true;
        if (sh->abort) return false;
        if (globaltimer_ns() - t0 > p.timeout_ns) {
            set_status(p.status, MC_ERR_TIMEOUT);
            sh->abort = 1;
            return false;
        }
    }
}

__device__ __forceinline__ bool tc_header_ok(const ExpertParams &p, int e)
{
    const PackHeader *hd = reinterpret_cast<const PackHeader *>(p.packed);
    return hd->magic == kMagic && hd->version == kFormatVersion && hd->E == p.E && hd->H == p.H &&
           hd->F == p.F && hd->group == p.group && hd->bits[e] == p.bits[e] &&
           hd->mat_off[e][0] == p.mat_off[e][0] && hd->mat_off[e][1] == p.mat_off[e][1] &&
           hd->mat_off[e][2] == p.mat_off[e][2];
}

// ------------------------------------------------ activation tiles + tables --

// Offset tables (mc_layout.h) of `ntok` rows of 128 fp16 columns held in shared
// memory, one warp per (row, group): dst[(n * gpt + gi) * 8] =
// [X, 0, O1 half0, O1 half1, O2 half0, O2 half1, O3 half0, O3 half1].
__device__ __forceinline__ void tc_tables(const __half *rows, int ntok, int group, float *dst, int warp, int nwarps,
                                          int lane)
{
    const int gpt = kTileK / group;
    for (int item = warp; item < ntok * gpt; item += nwarps) {
        const int n = item / gpt, gi = item % gpt;
        float tb[7] = {0, 0, 0, 0, 0, 0, 0};
        for (int c = gi * group + lane; c < (gi + 1) * group; c += 32) {
            const float v = __half2float(rows[n * kTileK + c]);
            const int j0 = pair_of_col(c, 0), j1 = pair_of_col(c, 1);
            tb[0] += v;
            tb[1] = fmaf(off1(j0), v, tb[1]);
            tb[2] = fmaf(off1(j1), v, tb[2]);
            tb[3] = fmaf(off2(j0), v, tb[3]);
            tb[4] = fmaf(off2(j1), v, tb[4]);
            tb[5] = fmaf(off3(j0), v, tb[5]);
            tb[6] = fmaf(off3(j1), v, tb[6]);
        }
#pragma unroll
        for (int k = 0; k < 7; ++k)
#pragma unroll
            for (int m = 16; m >= 1; m >>= 1) tb[k] += __shfl_xor_sync(0xffffffffu, tb[k], m);
        if (lane == 0) {
            float4 *d = reinterpret_cast<float4 *>(dst + (size_t)item * kTabFloats);
            d[0] = make_float4(tb[0], 0.f, tb[1], tb[2]);
            d[1] = make_float4(tb[3], tb[4], tb[5], tb[6]);
        }
    }
}

// SW128 image of a [16 rows][128 cols] fp16 tile: two 64-column atoms of
// 16 rows x 128 bytes; one 16-byte chunk per thread-iteration.
__device__ __forceinline__ void tc_bimage(const __half *rows, uint8_t *dst, int tid, int nthreads)
{
    for (int idx = tid; idx < 16 * 16; idx += nthreads) {
        const int n = idx >> 4, c = idx & 15;  // row, 16-byte chunk along the 128 columns
        const uint4 v = *reinterpret_cast<const uint4 *>(rows + n * kTileK + c * 8);
        *reinterpret_cast<uint4 *>(dst + (c >> 3) * 2048 + sw128_offset(n, (c & 7) * 8)) = v;
    }
}

// x of the routed pairs -> fp16 activation tiles + tables, per (chunk, 128 cols)
__global__ void __launch_bounds__(256) frag_x_tc_kernel(ExpertParams p)
{
    __shared__ __align__(16) __half xs[kChunk * kTileK];
    const int k = blockIdx.x, kt = blockIdx.y, KT = p.H / kTileK;
    if (k >= *p.nchunks) return;
    const ChunkInfo ci = p.chunks[k];
    const int tid = threadIdx.x;
    {
        const int n = tid >> 4, c8 = (tid & 15) * 8;
        uint4 out = make_uint4(0, 0, 0, 0);
        if (n < ci.nv) {
            const int tok = p.perm[ci.pair_base + n] >> 1;
            const uint4 raw = *reinterpret_cast<const uint4 *>(p.x + (size_t)tok * p.H + kt * kTileK + c8);
            const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
            __half2 *h2 = reinterpret_cast<__half2 *>(&out);
            bool bad = false;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 f = __bfloat1622float2(b2[i]);
                bad |= !(fabsf(f.x) <= 65504.f) || !(fabsf(f.y) <= 65504.f);
                h2[i] = __floats2half2_rn(f.x, f.y);
            }
            if (bad) set_status(p.status, MC_ERR_RANGE);
        }
        *reinterpret_cast<uint4 *>(xs + n * kTileK + c8) = out;
    }
    __syncthreads();
    const size_t tile = (size_t)k * KT + kt;
    tc_bimage(xs, p.xfrag + tile * kFragBytes, tid, 256);
    tc_tables(xs, kChunk, p.group, p.xtab + tile * (tab_bytes(p.group) / 4), tid >> 5, 8, tid & 31);
}

// h = silu(g) * u of the chunk's pairs -> fp16 activation tiles + tables for W2
__global__ void __launch_bounds__(256) frag_h_tc_kernel(ExpertParams p)
{
    __shared__ __align__(16) __half hs[kChunk * kTileK];
    const int k = blockIdx.x, kt = blockIdx.y, KT = p.F / kTileK;
    if (k >= *p.nchunks) return;
    const ChunkInfo ci = p.chunks[k];
    const int tid = threadIdx.x;
    // gu layout: [chunk][m (0: gate, 1: up)][F rows][16 pairs] fp32
    const float *g = p.gu + ((size_t)k * 2 + 0) * p.F * kChunk;
    const float *u = p.gu + ((size_t)k * 2 + 1) * p.F * kChunk;
    for (int idx = tid; idx < kTileK * kChunk; idx += 256) {
        const int f = idx >> 4, n = idx & 15;
        const size_t o = (size_t)(kt * kTileK + f) * kChunk + n;
        const float hv = n < ci.nv ? silu(g[o]) * u[o] : 0.f;
        hs[n * kTileK + f] = __float2half_rn(hv);
    }
    __syncthreads();
    const size_t tile = (size_t)k * KT + kt;
    tc_bimage(hs, p.hfrag + tile * kFragBytes, tid, 256);
    tc_tables(hs, kChunk, p.group, p.htab + tile * (tab_bytes(p.group) / 4), tid >> 5, 8, tid & 31);
}

// ------------------------------------------------------------------- items --

struct TcItem {
    int k;              // chunk
    ChunkInfo ci;
    int mat;            // 0 = W1, 1 = W3, 2 = W2
    int blk;            // 128-row block
    int kt0, nkt, ks;   // column tiles [kt0, kt0 + nkt), split index
};

template <bool W13>
__device__ __forceinline__ TcItem tc_item(const ExpertParams &p, int item, int U)
{
    TcItem it;
    it.k = item / U;
    const int u = item % U;
    it.ci = p.chunks[it.k];
    if (W13) {
        const int nrb = p.F / kBlockRows;
        it.mat = u / nrb;
        it.blk = u % nrb;
        it.kt0 = 0;
        it.nkt = p.H / kTileK;
        it.ks = 0;
    } else {
        const int nrb = p.H / kBlockRows;
        it.mat = 2;
        it.ks = u / nrb;
        it.blk = u % nrb;
        it.nkt = (p.F / kTileK) / p.KS;
        it.kt0 = it.ks * it.nkt;
    }
    return it;
}

// ------------------------------------------------------------ conversion --

// One converter lane, one 128-column step of its 16-row tile: packed words ->
// fp16 A values written into the two 64-column atoms' SW128 tiles.
template <int BITS>
__device__ __forceinline__ void tc_convert(const uint8_t *tile, int lane, int rbase, uint8_t *abuf0, uint8_t *abuf1)
{
    uint32_t c2[4], c1[2];
    if (BITS >= 2) {
        const uint4 v = *reinterpret_cast<const uint4 *>(tile + 16 * lane);
        c2[0] = v.x; c2[1] = v.y; c2[2] = v.z; c2[3] = v.w;
    }
    if (BITS != 2) {
        const uint2 v = *reinterpret_cast<const uint2 *>(tile + (BITS == 3 ? 512 : 0) + 8 * lane);
        c1[0] = v.x; c1[1] = v.y;
    }
    const int g8 = lane >> 2, t = lane & 3;
    const int r0 = rbase + g8, r1 = r0 + 8;
#pragma unroll
    for (int qd = 0; qd < 4; ++qd) {
        uint32_t r[8];
        if (BITS == 1) cvt1_half(c1[qd >> 1], 8 * (qd & 1), r);
        if (BITS == 2) cvt2(c2[qd], r);
        if (BITS == 3) {
            const uint32_t w[6] = {c2[0], c2[1], c2[2], c2[3], c1[0], c1[1]};
            cvt3(w, qd, r);
        }
        uint8_t *ab = (qd >> 1) ? abuf1 : abuf0;
        const int chunk = 2 * t + (qd & 1);
        const uint32_t o0 = r0 * 128u + ((uint32_t)(chunk ^ (r0 & 7)) << 4);
        const uint32_t o1 = r1 * 128u + ((uint32_t)(chunk ^ (r1 & 7)) << 4);
        *reinterpret_cast<uint4 *>(ab + o0) = make_uint4(r[0], r[2], r[4], r[6]);
        *reinterpret_cast<uint4 *>(ab + o1) = make_uint4(r[1], r[3], r[5], r[7]);
    }
}

// ------------------------------------------------------------------ fold --

template <int NC>
__device__ __forceinline__ void tc_fold(float (&y)[16], const float (&d)[16], float s, float z, const float *tab,
                                        int gpt, int gi, int oidx)
{
#pragma unroll
    for (int n = 0; n < NC; ++n) {
        const float *T = tab + (n * gpt + gi) * kTabFloats;
        y[n] += s * (d[n] - T[oidx] - z * T[0]);
    }
}

// End of an item: the 16 results of this thread's row.  W13: gate / up values
// [chunk][mat][F][16] for frag_h_tc_kernel; W2: expert outputs of the split.
template <bool W13>
__device__ __forceinline__ void tc_flush(const ExpertParams &p, const TcItem &I, const float (&y)[16], int row)
{
    if (W13) {
        float4 *dst = reinterpret_cast<float4 *>(
            p.gu + (((size_t)I.k * 2 + I.mat) * p.F + (size_t)I.blk * kBlockRows + row) * kChunk);
#pragma unroll
        for (int q = 0; q < 4; ++q) dst[q] = make_float4(y[4 * q], y[4 * q + 1], y[4 * q + 2], y[4 * q + 3]);
    } else {
        float *out = p.opart + (size_t)I.ks * p.Pmax * p.H + (size_t)I.blk * kBlockRows + row;
#pragma unroll
        for (int n = 0; n < 16; ++n)
            if (n < I.ci.nv) out[(size_t)(I.ci.pair_base + n) * p.H] = y[n];
    }
}

// ----------------------------------------------------------------- kernel --

template <bool W13>
__global__ void __launch_bounds__(kTcThreads, 1) tc_kernel(ExpertParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    TcShared *sh = reinterpret_cast<TcShared *>(smem);
    uint8_t *abase = smem + kTcABase;
    uint8_t *ring = smem + kTcRingBase;
    const int S = p.nslots, group = p.group, gpt = kTileK / group;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int U = W13 ? 2 * (p.F / kBlockRows) : (p.H / kBlockRows) * p.KS;
    const int KTv = W13 ? p.H / kTileK : p.F / kTileK;  // column tiles of the activations
    const uint8_t *vimg = W13 ? p.xfrag : p.hfrag;
    const float *vtab = W13 ? p.xtab : p.htab;
    const int tabf = tab_bytes(group) / 4;
    const int fpt = gpt;  // fold units (quantisation groups) per 128-column step

    if (threadIdx.x == 0) {
        for (int s = 0; s < kTcMaxSlots; ++s) {
            mbar_init(&sh->full[s], 1);
            mbar_init(&sh->empty[s], kTcConv + 1 + 4);
        }
        for (int a = 0; a < kTcNA; ++a) {
            mbar_init(&sh->a_full[a], kTcConv);
            mbar_init(&sh->a_empty[a], 1);
        }
        for (int d = 0; d < kTcND; ++d) {
            mbar_init(&sh->d_full[d], 1);
            mbar_init(&sh->d_empty[d], 4);
        }
        mbar_init(&sh->drain, 1);
        sh->abort = 0;
        sh->issued = 0;
        fence_mbar_init();
    }
    if (warp == kTcMma) tmem_alloc(&sh->tmem_base, kTcND * 16);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = sh->tmem_base;

    if (warp == kTcProd) {
        // ------------------------------------------------------------ producer --
        if (lane == 0 && !(p.debug & kDebugNoProducer)) {
            const uint64_t pol = policy_evict_first();
            const int total = *p.nchunks * U;
            int it = 0;
            bool ok = true;
            while (ok) {
                const int item = atomicAdd(&p.counters[W13 ? 0 : 1], 1);
                if (item >= total) break;
                const TcItem I = tc_item<W13>(p, item, U);
                const int e = I.ci.e;
                if (!tc_header_ok(p, e)) {
                    set_status(p.status, MC_ERR_BAD_PACK);
                    sh->abort = 1;
                    ok = false;
                    break;
                }
                const int STB = supertile_bytes(I.ci.bits, group);
                const int KTm = W13 ? p.H / kTileK : p.F / kTileK;
                const uint8_t *mat = p.packed + p.mat_off[e][I.mat];
                for (int i = 0; i < I.nkt; ++i, ++it) {
                    const int slot = it % S;
                    if (it >= S && !tc_wait(&sh->empty[slot], ((it / S) - 1) & 1, p, sh)) {
                        ok = false;
                        break;
                    }
                    const int kt = I.kt0 + i;
                    sh->slot_item[slot] = item;
                    sh->slot_i[slot] = i;
                    uint8_t *dst = ring + (size_t)slot * kTcSlotBytes;
                    const size_t vt = (size_t)I.k * KTv + kt;
                    mbar_arrive_expect_tx(&sh->full[slot], kFragBytes + tabf * 4 + STB);
                    bulk_g2s(dst + kSlotBImg, vimg + vt * kFragBytes, kFragBytes, &sh->full[slot]);
                    bulk_g2s(dst + kSlotTab, vtab + vt * tabf, tabf * 4, &sh->full[slot]);
                    bulk_g2s_stream(dst + kSlotPack,
                                    mat + supertile_off(I.mat, I.blk, kt, KTm,
                                                        (I.mat < 2 ? p.F : p.H) / kBlockRows, STB),
                                    STB, &sh->full[slot],
                                    pol);
                    sh->issued = it + 1;
                }
            }
            if (ok) {
                const int slot = it % S;
                if (it < S || tc_wait(&sh->empty[slot], ((it / S) - 1) & 1, p, sh)) {
                    sh->slot_item[slot] = -1;
                    mbar_arrive(&sh->full[slot]);
                }
            }
        }
    } else if (warp < kTcConv) {
        // ---------------------------------------------------------- converters --
        int cur = -1, bits = 1;
        for (int it = 0;; ++it) {
            const int slot = it % S;
            if (!tc_wait(&sh->full[slot], (it / S) & 1, p, sh)) break;
            const int item = sh->slot_item[slot];
            if (item < 0) break;
            if (item != cur) {
                cur = item;
                bits = p.chunks[item / U].bits;
            }
            const int ga = 2 * it;  // global atom index of this step's first atom
            const int a0 = ga % kTcNA, a1 = (ga + 1) % kTcNA;
            bool ok = true;
            if (ga >= kTcNA) ok = tc_wait(&sh->a_empty[a0], ((ga / kTcNA) - 1) & 1, p, sh);
            if (ok && ga + 1 >= kTcNA) ok = tc_wait(&sh->a_empty[a1], (((ga + 1) / kTcNA) - 1) & 1, p, sh);
            if (!ok) break;
            const uint8_t *tile = ring + (size_t)slot * kTcSlotBytes + kSlotPack + warp * tile_bytes(bits, group);
            uint8_t *ab0 = abase + a0 * kABufBytes, *ab1 = abase + a1 * kABufBytes;
            if (bits == 1) tc_convert<1>(tile, lane, warp * 16, ab0, ab1);
            else if (bits == 2) tc_convert<2>(tile, lane, warp * 16, ab0, ab1);
            else tc_convert<3>(tile, lane, warp * 16, ab0, ab1);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&sh->a_full[a0]);
                mbar_arrive(&sh->a_full[a1]);
                mbar_arrive(&sh->empty[slot]);
            }
        }
    } else if (warp == kTcMma) {
        // ------------------------------------------------------------- MMA --
        if (lane == 0) {
            const uint32_t idesc = umma_idesc_f16(128, kChunk);
            int cur = -1, bits = 1;
            for (int it = 0;; ++it) {
                const int slot = it % S;
                if (!tc_wait(&sh->full[slot], (it / S) & 1, p, sh)) break;
                const int item = sh->slot_item[slot];
                if (item < 0) break;
                if (item != cur) {
                    cur = item;
                    bits = p.chunks[item / U].bits;
                }
                const uint8_t *bimg = ring + (size_t)slot * kTcSlotBytes + kSlotBImg;
                bool ok = true;
                for (int h = 0; h < 2 && ok; ++h) {
                    const int ga = 2 * it + h, ai = ga % kTcNA;
                    const int fu = gpt == 2 ? ga : it;  // fold unit
                    const int ds = fu % kTcND;
                    const bool first = gpt == 2 || h == 0;
                    if (first && fu >= kTcND) ok = tc_wait(&sh->d_empty[ds], ((fu / kTcND) - 1) & 1, p, sh);
                    if (ok) ok = tc_wait(&sh->a_full[ai], (ga / kTcNA) & 1, p, sh);
                    if (!ok) break;
                    tc_fence_after();
                    const uint8_t *ab = abase + ai * kABufBytes;
                    const uint32_t dt = tbase + (uint32_t)(ds * 16);
#pragma unroll
                    for (int sub = 0; sub < 4; ++sub) {
                        const uint64_t bd = umma_desc_sw128(bimg + h * 2048 + sub * 32);
                        umma_f16(dt, umma_desc_sw128(ab + sub * 32), bd, idesc, !(first && sub == 0));
                    }
                    umma_commit(&sh->a_empty[ai]);
                    if (gpt == 2 || h == 1) umma_commit(&sh->d_full[ds]);
                }
                if (!ok) break;
                umma_commit(&sh->empty[slot]);
            }
            // every MMA this thread issued has completed before TMEM is released
            umma_commit(&sh->drain);
            const uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(&sh->drain, 0))
                if (globaltimer_ns() - t0 > p.timeout_ns) break;
        }
    } else {
        // --------------------------------------------------------- epilogue --
        const int ew = warp - kTcEpi0;  // TMEM lanes 32 ew .. 32 ew + 31
        const int row = 32 * ew + lane;  // 0..127 within the item's row block
        float y[16];
#pragma unroll
        for (int n = 0; n < 16; ++n) y[n] = 0.f;
        int cur = -1;
        TcItem I;
        I.k = 0;
        I.ci.nv = 0;
        for (int it = 0;; ++it) {
            const int slot = it % S;
            if (!tc_wait(&sh->full[slot], (it / S) & 1, p, sh)) break;
            const int item = sh->slot_item[slot];
            if (item < 0) break;
            if (item != cur) {
                if (cur >= 0) tc_flush<W13>(p, I, y, row);
                cur = item;
                I = tc_item<W13>(p, item, U);
#pragma unroll
                for (int n = 0; n < 16; ++n) y[n] = 0.f;
            }
            const uint8_t *sl = ring + (size_t)slot * kTcSlotBytes;
            const float *tab = reinterpret_cast<const float *>(sl + kSlotTab);
            const int bits = I.ci.bits, TB = tile_bytes(bits, group);
            const uint8_t *meta = sl + kSlotPack + (row >> 4) * TB + tile_code_bytes(bits);
            const int oidx = 2 * bits + ((row >> 3) & 1);
            bool ok = true;
            for (int f = 0; f < fpt; ++f) {
                const int fu = fpt * it + f, ds = fu % kTcND;
                if (!tc_wait(&sh->d_full[ds], (fu / kTcND) & 1, p, sh)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                float d[16];
                tmem_ld16(tbase + ((uint32_t)(32 * ew) << 16) + (uint32_t)(ds * 16), d);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sh->d_empty[ds]);
                const __half2 sz = *reinterpret_cast<const __half2 *>(meta + (f * 8 + (row & 7)) * 8 +
                                                                       ((row >> 3) & 1) * 4);
                const float2 szf = __half22float2(sz);
                if (I.ci.nv <= 4) tc_fold<4>(y, d, szf.x, szf.y, tab, gpt, f, oidx);
                else if (I.ci.nv <= 8) tc_fold<8>(y, d, szf.x, szf.y, tab, gpt, f, oidx);
                else tc_fold<16>(y, d, szf.x, szf.y, tab, gpt, f, oidx);
            }
            if (!ok) break;
            __syncwarp();
            if (lane == 0) mbar_arrive(&sh->empty[slot]);
        }
        if (cur >= 0 && !sh->abort) tc_flush<W13>(p, I, y, row);
    }

    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && sh->abort) {
        for (int it = max(0, sh->issued - S); it < sh->issued; ++it) {
            const uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(&sh->full[it % S], (it / S) & 1))
                if (globaltimer_ns() - t0 > p.timeout_ns) break;
        }
    }
    if (warp == kTcMma) {
        tc_fence_after();
        tmem_dealloc(tbase, kTcND * 16);
    }
}

// --------------------------------------------------------------- launcher --

int launch_tc(ExpertParams ep, cudaStream_t st)
{
    int dev = 0, maxsm = 0, nsm = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&maxsm, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "device query: %s", cudaGetErrorString(err));
    int nslots = (int)((maxsm - tc_smem(0)) / kTcSlotBytes);
    nslots = nslots > kTcMaxSlots ? kTcMaxSlots : nslots;
    if (nslots < 2) return set_error(MC_ERR_UNSUPPORTED, "not enough shared memory for the expert ring");
    ep.nslots = nslots;
    const size_t sm = tc_smem(nslots);
    err = cudaFuncSetAttribute(tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (err == cudaSuccess) err = cudaFuncSetAttribute(tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(err));

    profile_begin(kKGemmGather, st);
    frag_x_tc_kernel<<<dim3(ep.max_chunks, ep.H / kTileK), 256, 0, st>>>(ep);
    profile_end(kKGemmGather, st);
    err = cudaGetLastError();
    if (err == cudaSuccess) {
        profile_begin(kKGemvW13, st);
        tc_kernel<true><<<nsm, kTcThreads, sm, st>>>(ep);
        profile_end(kKGemvW13, st);
        err = cudaGetLastError();
    }
    if (err == cudaSuccess) {
        profile_begin(kKGlu, st);
        frag_h_tc_kernel<<<dim3(ep.max_chunks, ep.F / kTileK), 256, 0, st>>>(ep);
        profile_end(kKGlu, st);
        err = cudaGetLastError();
    }
    if (err == cudaSuccess) {
        profile_begin(kKGemvW2, st);
        tc_kernel<false><<<nsm, kTcThreads, sm, st>>>(ep);
        profile_end(kKGemvW2, st);
        err = cudaGetLastError();
    }
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "expert kernel launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

}  // namespace mc
