// mc_gemv.cu -- decode-path expert kernels: mixed-bit (1/2/3-bit) grouped
// dequant-GEMV over the SwiGLU experts (Eq. 1's E_i on PMQ weights, Sec. 2.2).
//
// frag_x_kernel: gathers the routed tokens' activations per work chunk (<= 16
//   pairs of one expert) into mma B-fragment order, fp16, with the per-group
//   offset tables, one 128-column tile at a time.
// gemv_kernel<W13>: persistent, one CTA per SM.  A producer warp claims work
//   items from an atomic counter (chunks of experts with more bits first) and
//   streams, for every 128-column step of an item, one ring stage holding
//     [row stream A supertile][row stream B supertile][B fragments][tables]
//   with cp.async.bulk (mbarrier transaction counts, L2 evict-first for the
//   weights), never pausing between items.  Sixteen consumer warps each own one
//   16-row tile of one stream: its code words become fp16 mma.sync A fragments
//   with one LOP3 per register (mc_layout.h), and every quantisation group is
//   folded as
//       y += s * (acc - O - z * X)
//   where acc = sum_k (off_k + q_k) x_k, O = sum_k off_k x_k, X = sum_k x_k, i.e.
//   y += s * sum_k (q_k - z) x_k, the group-wise dequantised product.
//   W13: streams = W1 and W3 rows of a 128-row block; the epilogue forms
//        h = silu(W1 x) * (W3 x) and writes it straight into W2's fragment order
//        with its tables.
//   W2:  streams = two 128-row blocks of W2 over one column split; the epilogue
//        writes fp32 expert outputs.
// The decode path is bound by HBM bandwidth on the packed weight bytes.
#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"

namespace mc {

constexpr int kCW = 16;                     // consumer warps
constexpr int kGemvThreads = (kCW + 1) * 32;
constexpr int kMaxSlots = 16;
constexpr int kRingOff = 1024;

struct RingShared {
    uint64_t cbar;  // consumer-warp barrier of the W13 epilogue (bounded waits)
    volatile int abort;
    volatile int issued;
    int slot_item[kMaxSlots];
    int slot_i[kMaxSlots];
};

__host__ __device__ inline int slot_bytes(int group)
{
    return 2 * supertile_bytes(3, group) + kFragBytes + tab_bytes(group);
}

__host__ __device__ inline size_t epi_off(int nslots, int group) { return kRingOff + (size_t)nslots * slot_bytes(group); }
constexpr int kXbufBytes = 8 * 32 * 8 * 4;   // stream-B results handed to stream A
constexpr int kHsBytes = kChunk * kTileK * 2;  // h tile [16][128] fp16

__host__ __device__ inline size_t gemv_smem(int nslots, int group)
{
    return epi_off(nslots, group) + kXbufBytes + kHsBytes;
}

// Bounded wait that gives up as soon as another thread of the CTA aborted.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, const ExpertParams &p, RingShared *sh)
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

// The packed buffer must carry the header written for this shape and bit table:
// the expert's bit width and the byte offsets of its matrices (which depend on
// every earlier expert's width) must match what the host computed, so no copy
// ever reads outside the region the buffer was packed with.
__device__ __forceinline__ bool header_ok(const ExpertParams &p, int e)
{
    const PackHeader *hd = reinterpret_cast<const PackHeader *>(p.packed);
    return hd->magic == kMagic && hd->version == kFormatVersion && hd->E == p.E && hd->H == p.H &&
           hd->F == p.F && hd->group == p.group && hd->bits[e] == p.bits[e] &&
           hd->mat_off[e][0] == p.mat_off[e][0] && hd->mat_off[e][1] == p.mat_off[e][1] &&
           hd->mat_off[e][2] == p.mat_off[e][2];
}

// Offset tables (mc_layout.h) of `ntok` rows of 128 fp16 columns held in shared
// memory; one warp per (row, group) item, written to dst[(n * gpt + gi) * 8].
__device__ __forceinline__ void write_tables(const __half *rows, int ntok, int group, float *dst, int warp, int nwarps,
                                             int lane)
{
    const int gpt = kTileK / group;
    for (int item = warp; item < ntok * gpt; item += nwarps) {
        const int n = item / gpt, gi = item % gpt;
        float tb[5] = {0, 0, 0, 0, 0};
        for (int c = gi * group + lane; c < (gi + 1) * group; c += 32) {
            const float v = __half2float(rows[n * kTileK + c]);
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
            float4 *d = reinterpret_cast<float4 *>(dst + (size_t)item * kTabFloats);
            d[0] = make_float4(tb[0], 0.f, tb[1], tb[2]);
            d[1] = make_float4(tb[3], tb[4], tb[3] + 4.f * tb[1], tb[4] + 4.f * tb[2]);
        }
    }
}

// Fragment entries (j < NT) of a [16][128] fp16 tile held in shared memory,
// 8 bytes each, ordered [j][s/2][lane][s%2] so that one 16-byte load gives a
// lane its B fragments of k-steps 2q and 2q+1.
__device__ __forceinline__ void write_frags(const __half *rows, int NT, uint8_t *dst, int tid, int nthreads)
{
    for (int idx = tid; idx < NT * 256; idx += nthreads) {
        const int j = idx >> 8, s = 2 * ((idx >> 6) & 3) + (idx & 1), ln = (idx >> 1) & 31;
        const int n = 8 * j + (ln >> 2), t = ln & 3;
        const int col = 64 * (s >> 2) + 16 * t + 4 * (s & 3);
        reinterpret_cast<uint2 *>(dst)[idx] = *reinterpret_cast<const uint2 *>(rows + n * kTileK + col);
    }
}

// ------------------------------------------------------------------ frag_x --
__global__ void __launch_bounds__(256) frag_x_kernel(ExpertParams p)
{
    __shared__ __align__(16) __half xs[kChunk * kTileK];
    const int k = blockIdx.x, kt = blockIdx.y, KT = p.H / kTileK;
    if (k >= *p.nchunks) return;
    const ChunkInfo ci = p.chunks[k];
    const int NT = ci.nv > 8 ? 2 : 1;
    const int tid = threadIdx.x;
    {
        const int n = tid >> 4, c8 = (tid & 15) * 8;
        uint4 out = make_uint4(0, 0, 0, 0);
        if (n < ci.nv) {
            const int tok = p.perm[ci.pair_base + n] >> 1;
            uint4 raw = *reinterpret_cast<const uint4 *>(p.x + (size_t)tok * p.H + kt * kTileK + c8);
            const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&raw);
            __half2 *h2 = reinterpret_cast<__half2 *>(&out);
            bool bad = false;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float2 f = __bfloat1622float2(b2[i]);
                bad |= !(fabsf(f.x) <= 65504.f) || !(fabsf(f.y) <= 65504.f);
                h2[i] = __floats2half2_rn(f.x, f.y);
            }
            if (bad) set_status(p.status, MC_ERR_RANGE);
        }
        *reinterpret_cast<uint4 *>(xs + n * kTileK + c8) = out;
    }
    __syncthreads();
    const size_t tile = (size_t)k * KT + kt;
    write_frags(xs, NT, p.xfrag + tile * kFragBytes, tid, 256);
    write_tables(xs, 8 * NT, p.group, p.xtab + tile * (tab_bytes(p.group) / 4), tid >> 5, 8, tid & 31);
}

// -------------------------------------------------------------- one stage --
// One consumer warp, one 128-column step of its 16-row tile: decode, mma and
// fold.  Accumulates into y[j][c] (C-fragment layout, rows g8 / g8+8, pairs
// 8j + 2t + {0,1}).
template <int NT, int BITS>
__device__ __forceinline__ void stage_compute(const uint8_t *tile, const uint4 *frag, const float *tab, int group,
                                              int lane, float (&y)[2][4])
{
    const int gpt = kTileK / group;
    uint32_t c2[4], c1[2];
    if (BITS >= 2) {
        const uint4 v = *reinterpret_cast<const uint4 *>(tile + 16 * lane);
        c2[0] = v.x; c2[1] = v.y; c2[2] = v.z; c2[3] = v.w;
    }
    if (BITS != 2) {
        const uint2 v = *reinterpret_cast<const uint2 *>(tile + (BITS == 3 ? 512 : 0) + 8 * lane);
        c1[0] = v.x; c1[1] = v.y;
    }
    const uint8_t *mt = tile + tile_code_bytes(BITS);
    uint2 meta[2];
    meta[0] = *reinterpret_cast<const uint2 *>(mt + (lane >> 2) * 8);
    meta[1] = gpt == 2 ? *reinterpret_cast<const uint2 *>(mt + 64 + (lane >> 2) * 8) : meta[0];
    // two independent accumulators halve the dependent mma chain: 1/2-bit by
    // k-step parity, 3-bit low plane / high plane
    float acc[2][NT][4];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int c = 0; c < 4; ++c) acc[a][j][c] = 0.f;
#pragma unroll
    for (int qd = 0; qd < 4; ++qd) {
        uint32_t r[8], rh[8];
        if (BITS == 1) cvt1_half<false>(c1[qd >> 1], 8 * (qd & 1), r);
        if (BITS >= 2) cvt2(c2[qd], r);
        if (BITS == 3) cvt1_half<true>(c1[qd >> 1], 8 * (qd & 1), rh);
        uint4 bq[NT];
#pragma unroll
        for (int j = 0; j < NT; ++j) bq[j] = frag[(j * 4 + qd) * 32 + lane];
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const int s = 2 * qd + kk;
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                const uint32_t b0 = kk ? bq[j].z : bq[j].x, b1 = kk ? bq[j].w : bq[j].y;
                if (BITS == 3) {
                    mma16816(acc[0][j], r[4 * kk], r[4 * kk + 1], r[4 * kk + 2], r[4 * kk + 3], b0, b1);
                    mma16816(acc[1][j], rh[4 * kk], rh[4 * kk + 1], rh[4 * kk + 2], rh[4 * kk + 3], b0, b1);
                } else {
                    mma16816(acc[kk][j], r[4 * kk], r[4 * kk + 1], r[4 * kk + 2], r[4 * kk + 3], b0, b1);
                }
            }
            if ((s == 3 && gpt == 2) || s == 7) {
                const int gi = s == 3 ? 0 : gpt - 1;
                const uint2 mg = gi == 0 ? meta[0] : meta[1];  // no dynamic index: keeps meta in registers
                const __half2 *m2 = reinterpret_cast<const __half2 *>(&mg);
                const float2 sz0 = __half22float2(m2[0]), sz1 = __half22float2(m2[1]);
#pragma unroll
                for (int j = 0; j < NT; ++j) {
                    const int n0 = 8 * j + 2 * (lane & 3);
                    const float *T0 = tab + (size_t)(n0 * gpt + gi) * kTabFloats;
                    const float *T1 = T0 + gpt * kTabFloats;
                    const float X0 = T0[0], X1 = T1[0];
                    const float2 O0 = *reinterpret_cast<const float2 *>(T0 + 2 * BITS);
                    const float2 O1 = *reinterpret_cast<const float2 *>(T1 + 2 * BITS);
                    y[j][0] += sz0.x * (acc[0][j][0] + acc[1][j][0] - O0.x - sz0.y * X0);
                    y[j][1] += sz0.x * (acc[0][j][1] + acc[1][j][1] - O1.x - sz0.y * X1);
                    y[j][2] += sz1.x * (acc[0][j][2] + acc[1][j][2] - O0.y - sz1.y * X0);
                    y[j][3] += sz1.x * (acc[0][j][3] + acc[1][j][3] - O1.y - sz1.y * X1);
#pragma unroll
                    for (int a = 0; a < 2; ++a)
#pragma unroll
                        for (int c = 0; c < 4; ++c) acc[a][j][c] = 0.f;
                }
            }
        }
    }
}

template <int NT>
__device__ __forceinline__ void stage_dispatch(int bits, const uint8_t *tile, const uint4 *frag, const float *tab,
                                               int group, int lane, float (&y)[2][4])
{
    if (bits == 1) stage_compute<NT, 1>(tile, frag, tab, group, lane, y);
    else if (bits == 2) stage_compute<NT, 2>(tile, frag, tab, group, lane, y);
    else stage_compute<NT, 3>(tile, frag, tab, group, lane, y);
}

struct Item {
    int k, u;          // chunk, unit
    ChunkInfo ci;
    int blkA, blkB;    // 128-row blocks of the two streams (blkB < 0: none)
    int kt0, nkt, ks;
};

template <bool W13>
__device__ __forceinline__ Item decode_item(const ExpertParams &p, int item, int U)
{
    Item it;
    it.k = item / U;
    it.u = item % U;
    it.ci = p.chunks[it.k];
    if (W13) {
        it.blkA = it.blkB = it.u;
        it.kt0 = 0;
        it.nkt = p.H / kTileK;
        it.ks = 0;
    } else {
        const int nrb = p.H / kBlockRows, npair = (nrb + 1) / 2;
        it.ks = it.u / npair;
        const int pr = it.u % npair;
        it.blkA = 2 * pr;
        it.blkB = 2 * pr + 1 < nrb ? 2 * pr + 1 : -1;
        it.nkt = (p.F / kTileK) / p.KS;
        it.kt0 = it.ks * it.nkt;
    }
    return it;
}

// All consumer warps meet at the CTA's consumer barrier; false once the CTA
// aborted (bounded like every other wait).
__device__ __forceinline__ bool consumer_sync(const ExpertParams &p, RingShared *sh, int lane, int &uses)
{
    __syncwarp();
    if (lane == 0) mbar_arrive(&sh->cbar);
    return wait_or_abort(&sh->cbar, (uses++) & 1, p, sh);
}

// End of an item.  W13: h = silu(W1 x) * (W3 x) for the item's 128 rows, written
// in W2's fragment order with its tables.  W2: fp32 outputs of the split.
template <bool W13>
__device__ __forceinline__ void epilogue(const ExpertParams &p, const Item &J, const float (&y)[2][4], int x, int tl,
                                         int lane, int warp, float *xbuf, __half *hs, RingShared *sh, int &cbar_uses)
{
    const int NT = J.ci.nv > 8 ? 2 : 1;
    const int g8 = lane >> 2, t2 = 2 * (lane & 3);
    if (W13) {
        if (x == 1) {
            float4 *d = reinterpret_cast<float4 *>(xbuf + (tl * 32 + lane) * 8);
            d[0] = make_float4(y[0][0], y[0][1], y[0][2], y[0][3]);
            d[1] = make_float4(y[1][0], y[1][1], y[1][2], y[1][3]);
        }
        if (!consumer_sync(p, sh, lane, cbar_uses)) return;
        if (x == 0) {
            const float4 *u4 = reinterpret_cast<const float4 *>(xbuf + (tl * 32 + lane) * 8);
            const float4 ua = u4[0], ub = u4[1];
            const float u[2][4] = {{ua.x, ua.y, ua.z, ua.w}, {ub.x, ub.y, ub.z, ub.w}};
#pragma unroll
            for (int j = 0; j < 2; ++j)
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int n = 8 * j + t2 + (c & 1);
                    const int r = tl * 16 + g8 + 8 * (c >> 1);
                    const float hv = (j < NT && n < J.ci.nv) ? silu(y[j][c]) * u[j][c] : 0.f;
                    hs[n * kTileK + r] = __float2half_rn(hv);
                }
        }
        if (!consumer_sync(p, sh, lane, cbar_uses)) return;
        const int tabf = tab_bytes(p.group) / 4;
        const size_t vt = (size_t)J.k * (p.F / kTileK) + J.u;  // W2 column tile = this row block
        write_frags(hs, NT, p.hfrag + vt * kFragBytes, threadIdx.x, kCW * 32);
        write_tables(hs, 8 * NT, p.group, p.htab + vt * tabf, warp, kCW, lane);
    } else {
        if (x == 1 && J.blkB < 0) return;
        const int blk = x ? J.blkB : J.blkA;
        float *out = p.opart + (size_t)J.ks * p.Pmax * p.H;
#pragma unroll
        for (int j = 0; j < 2; ++j)
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int n = 8 * j + t2 + (c & 1);
                const int r = blk * kBlockRows + tl * 16 + g8 + 8 * (c >> 1);
                if (j < NT && n < J.ci.nv) out[(size_t)(J.ci.pair_base + n) * p.H + r] = y[j][c];
            }
    }
}

template <bool W13>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_kernel(ExpertParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    uint64_t *empty = full + kMaxSlots;
    RingShared *sh = reinterpret_cast<RingShared *>(smem + 256);
    uint8_t *ring = smem + kRingOff;
    const int S = p.nslots, group = p.group;
    const int SB = slot_bytes(group), stmax = supertile_bytes(3, group);
    float *xbuf = reinterpret_cast<float *>(smem + epi_off(S, group));
    __half *hs = reinterpret_cast<__half *>(smem + epi_off(S, group) + kXbufBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int U = W13 ? p.F / kBlockRows : ((p.H / kBlockRows + 1) / 2) * p.KS;
    const int KTv = W13 ? p.H / kTileK : p.F / kTileK;  // column tiles of the activation vectors
    const uint8_t *vfrag = W13 ? p.xfrag : p.hfrag;
    const float *vtab = W13 ? p.xtab : p.htab;
    const int tabf = tab_bytes(group) / 4;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kMaxSlots; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kCW);
        }
        mbar_init(&sh->cbar, kCW);
        sh->abort = 0;
        sh->issued = 0;
        fence_mbar_init();
    }
    __syncthreads();

    if (warp == kCW) {
        // ---------------------------------------------------------- producer --
        if (lane == 0 && !(p.debug & kDebugNoProducer)) {
            const uint64_t pol = policy_evict_first();
            const int total = *p.nchunks * U;
            int it = 0;
            bool ok = true;
            while (ok) {
                const int item = atomicAdd(&p.counters[W13 ? 0 : 1], 1);
                if (item >= total) break;
                const Item I = decode_item<W13>(p, item, U);
                const int e = I.ci.e, bits = I.ci.bits, NT = I.ci.nv > 8 ? 2 : 1;
                if (!header_ok(p, e)) {
                    set_status(p.status, MC_ERR_BAD_PACK);
                    sh->abort = 1;
                    ok = false;
                    break;
                }
                const int TB = tile_bytes(bits, group), STB = kTilesPerBlock * TB;
                const int KTm = W13 ? p.H / kTileK : p.F / kTileK;
                const uint8_t *matA = p.packed + p.mat_off[e][W13 ? 0 : 2];
                const uint8_t *matB = p.packed + p.mat_off[e][W13 ? 1 : 2];
                const uint32_t fbytes = NT * (kFragBytes / 2), tbytes = NT * (tabf * 4 / 2);
                for (int i = 0; i < I.nkt; ++i, ++it) {
                    const int slot = it % S;
                    if (it >= S && !wait_or_abort(&empty[slot], ((it / S) - 1) & 1, p, sh)) {
                        ok = false;
                        break;
                    }
                    const int kt = I.kt0 + i;
                    sh->slot_item[slot] = item;
                    sh->slot_i[slot] = i;
                    uint8_t *dst = ring + (size_t)slot * SB;
                    const size_t vt = (size_t)I.k * KTv + kt;
                    mbar_arrive_expect_tx(&full[slot], (I.blkB >= 0 ? 2 * STB : STB) + fbytes + tbytes);
                    bulk_g2s_stream(dst, matA + ((size_t)I.blkA * KTm + kt) * STB, STB, &full[slot], pol);
                    if (I.blkB >= 0)
                        bulk_g2s_stream(dst + stmax, matB + ((size_t)I.blkB * KTm + kt) * STB, STB, &full[slot], pol);
                    bulk_g2s(dst + 2 * stmax, vfrag + vt * kFragBytes, fbytes, &full[slot]);
                    bulk_g2s(dst + 2 * stmax + kFragBytes, vtab + vt * tabf, tbytes, &full[slot]);
                    sh->issued = it + 1;
                }
            }
            if (ok) {
                // end marker: one more stage with item -1 and no data
                const int slot = it % S;
                if (it < S || wait_or_abort(&empty[slot], ((it / S) - 1) & 1, p, sh)) {
                    sh->slot_item[slot] = -1;
                    mbar_arrive(&full[slot]);
                }
            }
        }
    } else {
        // --------------------------------------------------------- consumers --
        const int x = warp >> 3, tl = warp & 7;
        float y[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
        int cur = -1, cbar_uses = 0;
        Item I;
        I.k = 0;
        for (int it = 0;; ++it) {
            const int slot = it % S;
            if (!wait_or_abort(&full[slot], (it / S) & 1, p, sh)) break;
            const int item = sh->slot_item[slot];
            if (item < 0) break;
            if (item != cur) {
                if (cur >= 0) epilogue<W13>(p, I, y, x, tl, lane, warp, xbuf, hs, sh, cbar_uses);
                cur = item;
                I = decode_item<W13>(p, item, U);
#pragma unroll
                for (int j = 0; j < 2; ++j)
#pragma unroll
                    for (int c = 0; c < 4; ++c) y[j][c] = 0.f;
            }
            const uint8_t *base = ring + (size_t)slot * SB;
            if (!(x == 1 && I.blkB < 0)) {
                const int TB = tile_bytes(I.ci.bits, group);
                const uint8_t *tile = base + x * stmax + tl * TB;
                const uint4 *frag = reinterpret_cast<const uint4 *>(base + 2 * stmax);
                const float *tab = reinterpret_cast<const float *>(base + 2 * stmax + kFragBytes);
                if (I.ci.nv > 8) stage_dispatch<2>(I.ci.bits, tile, frag, tab, group, lane, y);
                else stage_dispatch<1>(I.ci.bits, tile, frag, tab, group, lane, y);
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty[slot]);
        }
        if (cur >= 0 && !sh->abort) epilogue<W13>(p, I, y, x, tl, lane, warp, xbuf, hs, sh, cbar_uses);
    }
    __syncthreads();
    // On an abort, let copies that were issued but never consumed land before the
    // CTA's shared memory is released (bounded).
    if (threadIdx.x == 0 && sh->abort) {
        for (int it = max(0, sh->issued - S); it < sh->issued; ++it) {
            const uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(&full[it % S], (it / S) & 1))
                if (globaltimer_ns() - t0 > p.timeout_ns) break;
        }
    }
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
            const float4 a = src[0], b = src[1];
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

// -------------------------------------------------------------- launchers --

int launch_gemv(ExpertParams ep, cudaStream_t st)
{
    int dev = 0, maxsm = 0, nsm = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&maxsm, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "device query: %s", cudaGetErrorString(err));
    int nslots = (int)((maxsm - gemv_smem(0, ep.group)) / slot_bytes(ep.group));
    nslots = nslots > kMaxSlots ? kMaxSlots : nslots;
    if (nslots < 2) return set_error(MC_ERR_UNSUPPORTED, "not enough shared memory for the GEMV ring");
    ep.nslots = nslots;
    const size_t sm = gemv_smem(nslots, ep.group);
    err = cudaFuncSetAttribute(gemv_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (err == cudaSuccess)
        err = cudaFuncSetAttribute(gemv_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(err));

    profile_begin(kKGemmGather, st);
    frag_x_kernel<<<dim3(ep.max_chunks, ep.H / kTileK), 256, 0, st>>>(ep);
    profile_end(kKGemmGather, st);
    err = cudaGetLastError();
    if (err == cudaSuccess) {
        profile_begin(kKGemvW13, st);
        gemv_kernel<true><<<nsm, kGemvThreads, sm, st>>>(ep);
        profile_end(kKGemvW13, st);
        err = cudaGetLastError();
    }
    if (err == cudaSuccess) {
        profile_begin(kKGemvW2, st);
        gemv_kernel<false><<<nsm, kGemvThreads, sm, st>>>(ep);
        profile_end(kKGemvW2, st);
        err = cudaGetLastError();
    }
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "GEMV launch: %s", cudaGetErrorString(err));
    return MC_OK;
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

}  // namespace mc
