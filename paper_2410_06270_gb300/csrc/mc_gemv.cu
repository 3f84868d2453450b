// mc_gemv.cu -- decode-path expert kernels: mixed-bit (1/2/3-bit) grouped
// dequant-GEMV over the SwiGLU experts (Eq. 1's E_i on PMQ weights, Sec. 2.2).
//
// frag_x_kernel: gathers the routed tokens' activations per work chunk (<= 16
//   pairs of one expert) into mma B-fragment order, fp16, with the per-group
//   offset tables: one "vector block" per (chunk, n-tile, 128-column step).
// gemv_kernel<W13>: persistent, one CTA per SM.  A producer warp claims work
//   items (a chunk x a 128-row block of W1|W3, or a chunk x a 256-row block pair
//   of W2 over one column split) from an atomic counter, experts with more bits
//   first, and streams each item as ring stages of kKPS 128-column steps:
//     [weights of both row streams, kKPS steps]   one cp.async.bulk copy
//     [vector blocks of n-tile 0][of n-tile 1]      one copy each
//   The packed layout interleaves the two streams step by step (mc_layout.h), so
//   a stage is a few large copies: small copies cap the streaming bandwidth well
//   below the HBM peak.  Eight consumer warps own 16-row tile tl of BOTH streams
//   (the B fragments and tables are loaded once for the two).  Code
//   words become fp16 mma.sync A fragments with one LOP3 per register
//   (mc_layout.h), and every quantisation group is accumulated from
//       acc = -(O + z X) + sum_k (off_k + q_k) x_k = sum_k (q_k - z) x_k
//   (O = sum_k off_k x_k, X = sum_k x_k from the vector block's tables) and
//   folded as y += s * acc, the group-wise dequantised product.
//   W13: streams = W1 and W3 rows of a 128-row block; each warp forms
//        h = silu(W1 x) * (W3 x) in registers and the CTA writes W2's vector
//        blocks.
//   W2:  streams = two 128-row blocks of W2; the epilogue writes fp32 outputs.
// Decoding costs about one ALU instruction per two weights, so the
// consumers are kept lean: this path is bound by HBM bandwidth on the packed
// weight bytes only while the decode keeps up with it.
#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"

namespace mc {

constexpr int kTPW = 2;                     // 16-row tiles per consumer warp: tile tl of both streams
constexpr int kCW = 16 / kTPW;              // consumer warps
constexpr int kGemvThreads = (kCW + 1) * 32;
constexpr int kMaxSlots = 16;
constexpr int kRingOff = 1024;
#ifndef MC_GEMV_KPS
#define MC_GEMV_KPS 4
#endif
constexpr int kKPS = MC_GEMV_KPS;           // 128-column steps per ring stage

struct RingShared {
    uint64_t cbar;  // consumer-warp barrier of the W13 epilogue (bounded waits)
    volatile int abort;
    volatile int issued;
    int slot_item[kMaxSlots];
    int slot_kc[kMaxSlots];  // column steps held by the stage (1..kKPS)
    ChunkInfo slot_ci[kMaxSlots];  // the stage's chunk
};
static_assert(256 + sizeof(RingShared) <= 1024, "ring header");

constexpr int kVecMax = kVecFragBytes + 8 * 2 * kTabFloats * 4;  // vec_bytes(64), the largest

// Column steps per ring stage: kKPS for quantised experts; one for 16-bit experts,
// whose two supertiles per step are already 64 KB.
__host__ __device__ inline int stage_steps(bool dense) { return dense ? 1 : kKPS; }
__host__ __device__ inline int slot_bytes(int group, bool dense)
{
    const int kps = stage_steps(dense);
    return kps * 2 * supertile_bytes(dense ? 16 : 3, group) + 2 * kps * kVecMax;
}
constexpr int kHsBytes = kChunk * kTileK * 2;           // h tile [16][128] fp16 (two of them)

__host__ __device__ inline size_t gemv_smem(int nslots, int group, bool dense)
{
    return kRingOff + (size_t)nslots * slot_bytes(group, dense) + 2 * kHsBytes + 8 * 32 * sizeof(uint2);
}

// Bounded wait that gives up as soon as another thread of the CTA aborted
// (*abort, the CTA's abort flag).
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, const ExpertParams &p,
                                              volatile int *abort)
{
    if (mbar_try_wait(bar, parity)) return true;
    uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait_sleep(bar, parity, kWaitHintNs)) return true;
        if (*abort) return false;
        if (globaltimer_ns() - t0 > p.timeout_ns) {
            set_status(p.status, MC_ERR_TIMEOUT);
            *abort = 1;
            return false;
        }
    }
}
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, const ExpertParams &p, RingShared *sh)
{
    return wait_or_abort(bar, parity, p, &sh->abort);
}

// The packed buffer must carry the header written for this shape and bit table:
// every expert's bit width and the byte offsets of its matrices (which depend on
// every earlier expert's width) must match what the host computed, so that no
// copy ever reads outside the region the buffer was packed with.  Checked once per
// call by frag_x_kernel (all loads in flight together); the expert kernels read
// its verdict.
__device__ __forceinline__ bool header_ok(const ExpertParams &p)
{
    const PackHeader *hd = reinterpret_cast<const PackHeader *>(p.packed);
    bool ok = hd->magic == kMagic && hd->version == kFormatVersion && hd->E == p.E && hd->H == p.H &&
              hd->F == p.F && hd->group == p.group;
#pragma unroll
    for (int e = 0; e < kMaxE; ++e)
        if (e < p.E)
            ok &= hd->bits[e] == p.bits[e] && hd->mat_off[e][0] == p.mat_off[e][0] &&
                  hd->mat_off[e][1] == p.mat_off[e][1] && hd->mat_off[e][2] == p.mat_off[e][2];
    return ok;
}

// D += A * B, m16n8k16, fp16 inputs, fp32 accumulate (not volatile, so the
// compiler may schedule it).
__device__ __forceinline__ void mma_acc(float (&d)[4], const uint32_t *a, uint32_t b0, uint32_t b1)
{
    asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Offset tables as a matrix product.  For pairs n of a vector block and one
// quantisation group, the table slots are
//     T[r][n] = sum_c M[r][c] x_n[c],   r = 0..7,
// with the rows of M the coefficients of the table layout below: off2(half 0),
// off2(half 1), 1, off1(half 0), off3(half 0), off3(half 1), 1, off1(half 1)
// (off_b(half) of column c = the b-bit field offset of the pair holding column
// c in that row half, mc_layout.h).  M is a constant fp16 matrix (powers of
// two), so one m16n8k16 mma per k-step forms the tables of eight pairs, with
// the B fragments of the main product.  tab_afrag[s][lane] holds the A
// fragment registers a0, a2 of k-step s (rows 8..15 of M are zero).
__device__ __forceinline__ float tab_coef(int r, int col)
{
    const int jp = pair_of_col(col, (r == 1 || r == 5 || r == 7) ? 1 : 0);
    if (r == 2 || r == 6) return 1.f;
    if (r == 0 || r == 1) return off2(jp);
    if (r == 3 || r == 7) return off1(jp);
    return off3(jp);
}

__device__ __forceinline__ void build_tab_afrag(uint2 *afr, int tid, int nthreads)
{
    for (int idx = tid; idx < 8 * 32; idx += nthreads) {
        const int s = idx >> 5, lane = idx & 31, g8 = lane >> 2, t = lane & 3;
        const int col0 = 64 * (s >> 2) + 16 * t + 4 * (s & 3);
        const __half2 lo = __floats2half2_rn(tab_coef(g8, col0), tab_coef(g8, col0 + 1));
        const __half2 hi = __floats2half2_rn(tab_coef(g8, col0 + 2), tab_coef(g8, col0 + 3));
        afr[idx] = make_uint2(*reinterpret_cast<const uint32_t *>(&lo), *reinterpret_cast<const uint32_t *>(&hi));
    }
}

// Vector blocks (n-tiles j < NT) built from a [16][128] fp16 tile in shared
// memory; block j at dst + j * jstride:
//   fragments, 256 entries of 8 bytes ordered [s/2][lane][s%2] (one 16-byte load
//     gives a lane its B fragments of k-steps 2q and 2q+1); an entry holds the
//     4 fp16 values at columns 64(s/4) + 16t + 4(s%4) .. +3 of pair 8j + lane/4;
//   then the offset tables of pairs 8j .. 8j+7, [n][group][8 floats]:
//     [O2 half 0, O2 half 1, X, O1 half 0, O3 half 0, O3 half 1, X, O1 half 1]
//   (X = sum of the group's inputs, O_b = sum of the b-bit field offsets times
//   the inputs for the rows of one half; mc_layout.h), so that a 2- or 3-bit
//   fold reads its O pair and X with one 16-byte load.
// All threads copy fragment entries; warp j forms block j's tables.
__device__ __forceinline__ void write_vec_blocks(const __half *rows, int NT, int group, uint8_t *dst, size_t jstride,
                                                 const uint2 *afr, int tid, int nthreads)
{
    for (int idx = tid; idx < NT * 256; idx += nthreads) {
        const int j = idx >> 8, s = 2 * ((idx >> 6) & 3) + (idx & 1), ln = (idx >> 1) & 31;
        const int n = 8 * j + (ln >> 2), t = ln & 3;
        const int col = 64 * (s >> 2) + 16 * t + 4 * (s & 3);
        reinterpret_cast<uint2 *>(dst + j * jstride)[idx & 255] =
            *reinterpret_cast<const uint2 *>(rows + n * kTileK + col);
    }
    const int warp = tid >> 5, lane = tid & 31;
    if (warp < NT) {
        const int j = warp, g8 = lane >> 2, t = lane & 3, gpt = kTileK / group;
        float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
        for (int s = 0; s < 8; ++s) {
            const int col0 = 64 * (s >> 2) + 16 * t + 4 * (s & 3);
            const uint2 b = *reinterpret_cast<const uint2 *>(rows + (8 * j + g8) * kTileK + col0);
            const uint2 a = afr[s * 32 + lane];
            const uint32_t af[4] = {a.x, 0u, a.y, 0u};
            mma_acc(acc[gpt == 2 ? (s >> 2) : 0], af, b.x, b.y);
        }
        float *tab = reinterpret_cast<float *>(dst + j * jstride + kVecFragBytes);
        for (int gi = 0; gi < gpt; ++gi) {
            tab[((2 * t) * gpt + gi) * kTabFloats + g8] = acc[gi][0];
            tab[((2 * t + 1) * gpt + gi) * kTabFloats + g8] = acc[gi][1];
        }
    }
}

// ------------------------------------------------------------------ frag_x --
__global__ void __launch_bounds__(256) frag_x_kernel(ExpertParams p)
{
    __shared__ __align__(16) __half xs[kChunk * kTileK];
    __shared__ uint2 afr[8 * 32];
    const int k = blockIdx.x, kt = blockIdx.y, KT = p.H / kTileK;
    // CTA (0, 0) checks the packed header for the expert kernels that follow (they
    // read only its verdict): the header's loads go out before the wait (the packed
    // buffer is complete before the layer starts), the verdict is written after it,
    // when the expert kernels of the call before have completed
    const bool hdr_thread = k == 0 && kt == 0 && threadIdx.x == 0;
    const bool hok = hdr_thread ? header_ok(p) : true;
    build_tab_afrag(afr, threadIdx.x, 256);
    // trigger only after the routing launch has completed: the expert kernel that
    // follows reads the routing outputs before its own wait
    pdl_wait();
    pdl_trigger();
    if (hdr_thread) {
        *p.hdr_ok = hok ? 1 : 0;
        if (!hok) set_status(p.status, MC_ERR_BAD_PACK);
    }
    // both loads in flight together (entry k < max_chunks exists even when unused)
    const int nchunks = *p.nchunks;
    const ChunkInfo ci = p.chunks[k];
    if (k >= nchunks) return;
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
    write_vec_blocks(xs, NT, p.group, p.xvec + vec_off(k, 0, kt, KT, p.group),
                     vec_off(0, 1, 0, KT, p.group), afr, tid, 256);
}

// --------------------------------------------------------------- one step --

// The code words and fp16 (scale, zero) pairs one lane needs from a tile.
template <int BITS, int GPT>
struct TileRegs {
    uint32_t c2[4], c1[2];
    uint2 meta[GPT];
};

template <int BITS, int GPT>
__device__ __forceinline__ void load_tile(const uint8_t *tile, int lane, TileRegs<BITS, GPT> &t)
{
    if (BITS >= 2) {
        const uint4 v = *reinterpret_cast<const uint4 *>(tile + 16 * lane);
        t.c2[0] = v.x; t.c2[1] = v.y; t.c2[2] = v.z; t.c2[3] = v.w;
    }
    if (BITS != 2) {
        const uint2 v = *reinterpret_cast<const uint2 *>(tile + (BITS == 3 ? 512 : 0) + 8 * lane);
        t.c1[0] = v.x; t.c1[1] = v.y;
    }
    const uint8_t *mt = tile + tile_code_bytes(BITS);
#pragma unroll
    for (int g = 0; g < GPT; ++g) t.meta[g] = *reinterpret_cast<const uint2 *>(mt + 64 * g + (lane >> 2) * 8);
}

// A-fragment registers of k-steps 2qd, 2qd+1 (pairs 8qd .. 8qd+7).
template <int BITS, int GPT>
__device__ __forceinline__ void decode_qd(const TileRegs<BITS, GPT> &t, int qd, uint32_t (&r)[8])
{
    if (BITS == 1) cvt1_half(t.c1[qd >> 1], 8 * (qd & 1), r);
    if (BITS == 2) cvt2(t.c2[qd], r);
    if (BITS == 3) {
        const uint32_t w[6] = {t.c2[0], t.c2[1], t.c2[2], t.c2[3], t.c1[0], t.c1[1]};
        cvt3(w, qd, r);
    }
}

// One consumer warp, one 128-column step of its NTL 16-row tiles: decode, mma
// and fold.  y[u][j][c]: tile u, C-fragment layout (rows g8 / g8+8 of the tile,
// pairs 8j + 2t + {0,1}).  vec0 / vec1: the step's vector blocks of n-tiles
// 0 / 1, shared by the tiles.  Each group's accumulator starts at
// -(O + z X), so after the group's mma chain it holds sum_k (q_k - z) x_k and
// the fold is a single y += s * acc.
template <int NT, int BITS, int GPT, int NTL>
__device__ __forceinline__ void step_tiles(const uint8_t *const (&tile)[NTL], const uint8_t *vec0,
                                           const uint8_t *vec1, int lane, float (&y)[NTL][NT][4])
{
    constexpr int SPG = 8 / GPT;  // k-steps per quantisation group
    TileRegs<BITS, GPT> R[NTL];
#pragma unroll
    for (int u = 0; u < NTL; ++u) load_tile<BITS, GPT>(tile[u], lane, R[u]);
    float acc[NTL][NT][4];
#pragma unroll
    for (int qd = 0; qd < 4; ++qd) {
        uint32_t r[NTL][8];
#pragma unroll
        for (int u = 0; u < NTL; ++u) decode_qd<BITS, GPT>(R[u], qd, r[u]);
        uint4 bq[NT];
#pragma unroll
        for (int j = 0; j < NT; ++j) bq[j] = reinterpret_cast<const uint4 *>(j ? vec1 : vec0)[qd * 32 + lane];
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const int s = 2 * qd + kk, gi = s / SPG;
            if (s % SPG == 0) {
#pragma unroll
                for (int j = 0; j < NT; ++j) {
                    const float *T0 = reinterpret_cast<const float *>((j ? vec1 : vec0) + kVecFragBytes) +
                                      (size_t)((2 * (lane & 3)) * GPT + gi) * kTabFloats;
                    const float *T1 = T0 + GPT * kTabFloats;
                    float2 O0, O1;
                    float X0, X1;
                    if (BITS == 1) {
                        const float4 u0 = *reinterpret_cast<const float4 *>(T0);
                        const float4 u1 = *reinterpret_cast<const float4 *>(T1);
                        O0 = make_float2(u0.w, T0[7]);
                        O1 = make_float2(u1.w, T1[7]);
                        X0 = u0.z;
                        X1 = u1.z;
                    } else {
                        const float4 u0 = *reinterpret_cast<const float4 *>(T0 + (BITS == 3 ? 4 : 0));
                        const float4 u1 = *reinterpret_cast<const float4 *>(T1 + (BITS == 3 ? 4 : 0));
                        O0 = make_float2(u0.x, u0.y);
                        O1 = make_float2(u1.x, u1.y);
                        X0 = u0.z;
                        X1 = u1.z;
                    }
#pragma unroll
                    for (int u = 0; u < NTL; ++u) {
                        const __half2 *m2 = reinterpret_cast<const __half2 *>(&R[u].meta[gi]);
                        const float z0 = __high2float(m2[0]), z1 = __high2float(m2[1]);
                        acc[u][j][0] = fmaf(-z0, X0, -O0.x);
                        acc[u][j][1] = fmaf(-z0, X1, -O1.x);
                        acc[u][j][2] = fmaf(-z1, X0, -O0.y);
                        acc[u][j][3] = fmaf(-z1, X1, -O1.y);
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                const uint32_t b0 = kk ? bq[j].z : bq[j].x, b1 = kk ? bq[j].w : bq[j].y;
#pragma unroll
                for (int u = 0; u < NTL; ++u) mma_acc(acc[u][j], r[u] + 4 * kk, b0, b1);
            }
            if (s % SPG == SPG - 1) {
#pragma unroll
                for (int u = 0; u < NTL; ++u) {
                    const __half2 *m2 = reinterpret_cast<const __half2 *>(&R[u].meta[gi]);
                    const float s0 = __low2float(m2[0]), s1 = __low2float(m2[1]);
#pragma unroll
                    for (int j = 0; j < NT; ++j) {
                        y[u][j][0] = fmaf(s0, acc[u][j][0], y[u][j][0]);
                        y[u][j][1] = fmaf(s0, acc[u][j][1], y[u][j][1]);
                        y[u][j][2] = fmaf(s1, acc[u][j][2], y[u][j][2]);
                        y[u][j][3] = fmaf(s1, acc[u][j][3], y[u][j][3]);
                    }
                }
            }
        }
    }
}

// One 128-column step of 16-bit (unquantised fp16) tiles: the A fragments are
// loaded as stored (one 16-byte load per k-step) and multiplied straight into y;
// there is no quantisation group to fold.
template <int NT, int NTL>
__device__ __forceinline__ void step_dense(const uint8_t *const (&tile)[NTL], const uint8_t *vec0,
                                           const uint8_t *vec1, int lane, float (&y)[NTL][NT][4])
{
#pragma unroll
    for (int qd = 0; qd < 4; ++qd) {
        uint4 a[NTL][2];
#pragma unroll
        for (int u = 0; u < NTL; ++u) {
            const uint4 *t4 = reinterpret_cast<const uint4 *>(tile[u] + 128 * lane) + 2 * qd;
            a[u][0] = t4[0];
            a[u][1] = t4[1];
        }
        uint4 bq[NT];
#pragma unroll
        for (int j = 0; j < NT; ++j) bq[j] = reinterpret_cast<const uint4 *>(j ? vec1 : vec0)[qd * 32 + lane];
#pragma unroll
        for (int kk = 0; kk < 2; ++kk)
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                const uint32_t b0 = kk ? bq[j].z : bq[j].x, b1 = kk ? bq[j].w : bq[j].y;
#pragma unroll
                for (int u = 0; u < NTL; ++u)
                    mma_acc(y[u][j], reinterpret_cast<const uint32_t *>(&a[u][kk]), b0, b1);
            }
    }
}

struct Item {
    int k, u;          // chunk, unit
    ChunkInfo ci;
    int blkA, blkB;    // 128-row blocks of the two streams (blkB < 0: none)
    int kt0, nkt, ks;  // column steps [kt0, kt0 + nkt) of split ks
};

template <bool W13>
__device__ __forceinline__ Item decode_item(const ExpertParams &p, int item, int U, const ChunkInfo &ci)
{
    Item it;
    it.k = item / U;
    it.u = item % U;
    it.ci = ci;
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

// Ring geometry shared by the consumer warps.
struct Ring {
    uint64_t *full, *empty;
    const uint8_t *base;
    int S, SB, vec_off0, VB;
    const uint2 *afr;  // A fragments of the table matrix
};

// What one group of consumer warps shares: the CTA's abort flag, the group's
// epilogue barrier, the column steps of each of its ring's stages, and the
// thread's index within the group.
struct GroupCtx {
    volatile int *abort;
    uint64_t *cbar;
    const int *slot_kc;
    int gtid;
};

// All consumer warps of a group meet at its barrier (bounded); false once the
// CTA aborted.
__device__ __forceinline__ bool consumer_sync(const ExpertParams &p, const GroupCtx &G, int lane, int &uses)
{
    __syncwarp();
    if (lane == 0) mbar_arrive(G.cbar);
    return wait_or_abort(G.cbar, (uses++) & 1, p, G.abort);
}

// One work item for one consumer warp: all its stages, then the epilogue.  The
// first stage's full barrier has already been waited for; the ring position
// (slot, phase) advances by one per stage.
//   The warp owns tile tl of both streams.
//   W13: h = silu(W1 x) * (W3 x) for the item's rows goes to the h tile
//        (double-buffered by item parity), then the consumer warps together
//        write W2's vector blocks of this 128-row block.
//   W2:  fp32 outputs of the split.
template <bool W13, int NT, int BITS, int GPT, int KPS>
__device__ __forceinline__ bool run_item(const ExpertParams &p, const GroupCtx &G, const Ring &R, const Item &I,
                                         int nrb, int tl, int lane, int &slot, uint32_t &phase, __half *hs2,
                                         int &items, int &cbar_uses)
{
    constexpr int group = kTileK / GPT;
    const int STB = supertile_bytes(BITS, group), TB = tile_bytes(BITS, group);
    const int pw = W13 ? 2 : w2_pair_width(I.blkA >> 1, nrb);
    const int step_bytes = pw * STB;
    // a lone W2 block (odd row-block count): stream B repeats stream A, unused
    const int offB = (pw == 2 ? STB : 0) + tl * TB;
    const int off[2] = {tl * TB, offB};
    float y[kTPW][NT][4];
#pragma unroll
    for (int u = 0; u < kTPW; ++u)
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int c = 0; c < 4; ++c) y[u][j][c] = 0.f;
    for (int i = 0; i < I.nkt; i += KPS) {
        if (i > 0 && !wait_or_abort(&R.full[slot], phase, p, G.abort)) return false;
        const uint8_t *base = R.base + (size_t)slot * R.SB;
        const int kc = G.slot_kc[slot];
        const uint8_t *v0 = base + R.vec_off0, *v1 = v0 + KPS * R.VB;
        auto step = [&](int kk) {
            const uint8_t *st = base + kk * step_bytes;
            const uint8_t *t[kTPW];
#pragma unroll
            for (int u = 0; u < kTPW; ++u) t[u] = st + off[u];
            if constexpr (BITS == 16)
                step_dense<NT, kTPW>(t, v0 + kk * R.VB, v1 + kk * R.VB, lane, y);
            else
                step_tiles<NT, BITS, GPT, kTPW>(t, v0 + kk * R.VB, v1 + kk * R.VB, lane, y);
        };
        if (GPT == 1 && kc == KPS) {
            // a full stage as straight-line code, so consecutive steps' loads and
            // decodes overlap (one group per tile keeps it within the registers)
#pragma unroll
            for (int kk = 0; kk < KPS; ++kk) step(kk);
        } else {
#pragma unroll
            for (int kk = 0; kk < KPS; ++kk)
                if (kk < kc) step(kk);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&R.empty[slot]);
        if (++slot == R.S) {
            slot = 0;
            phase ^= 1u;
        }
    }
    const int g8 = lane >> 2, t2 = 2 * (lane & 3);
    if (W13) {
        __half *hs = hs2 + (items & 1) * (kChunk * kTileK);
        ++items;
        // y[0]: W1 x, y[1]: W3 x of the warp's rows; h is W2's fp16 input, so a
        // value outside the fp16 range (or not finite) is reported, as for x
        bool bad = false;
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int n = 8 * j + t2 + (c & 1);
                const int r = tl * 16 + g8 + 8 * (c >> 1);
                const float hv = n < I.ci.nv ? silu(y[0][j][c]) * y[1][j][c] : 0.f;
                bad |= !(fabsf(hv) <= 65504.f);
                hs[n * kTileK + r] = __float2half_rn(hv);
            }
        if (bad) set_status(p.status, MC_ERR_RANGE);
        // every warp finished the previous item's vector blocks before it got
        // here, so after this barrier the other h buffer is free again
        if (!consumer_sync(p, G, lane, cbar_uses)) return false;
        // the item's 128 rows are W2's column step I.u
        const int KT2 = p.F / kTileK;
        write_vec_blocks(hs, NT, group, p.hvec + vec_off(I.k, 0, I.u, KT2, group), vec_off(0, 1, 0, KT2, group),
                         R.afr, G.gtid, kCW * 32);
    } else {
        float *out = p.opart + (size_t)I.ks * p.Pmax * p.H;
#pragma unroll
        for (int j = 0; j < NT; ++j)
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                const int n = 8 * j + t2 + (c & 1);
                const int r = tl * 16 + g8 + 8 * (c >> 1);
                if (n < I.ci.nv) {
                    float *o = out + (size_t)(I.ci.pair_base + n) * p.H;
                    o[I.blkA * kBlockRows + r] = y[0][j][c];
                    if (I.blkB >= 0) o[I.blkB * kBlockRows + r] = y[1][j][c];
                }
            }
    }
    return true;
}

template <bool W13, int GPT, bool DENSE>
__global__ void __launch_bounds__(kGemvThreads, 1) gemv_kernel(ExpertParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    uint64_t *empty = full + kMaxSlots;
    RingShared *sh = reinterpret_cast<RingShared *>(smem + 256);
    uint8_t *ring = smem + kRingOff;
    const int S = p.nslots, group = p.group;
    constexpr int KPS = DENSE ? 1 : kKPS;  // stage_steps(DENSE)
    const int SB = slot_bytes(group, DENSE), VB = vec_bytes(group);
    const int vec_off0 = KPS * 2 * supertile_bytes(DENSE ? 16 : 3, group);
    __half *hs2 = reinterpret_cast<__half *>(smem + kRingOff + (size_t)S * SB);
    uint2 *afr = reinterpret_cast<uint2 *>(smem + kRingOff + (size_t)S * SB + 2 * kHsBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nrb = W13 ? p.F / kBlockRows : p.H / kBlockRows;  // 128-row blocks of the matrix
    const int U = W13 ? nrb : ((nrb + 1) / 2) * p.KS;
    const int KTm = W13 ? p.H / kTileK : p.F / kTileK;  // column steps of the matrix and its vectors
    const uint8_t *vbase = W13 ? p.xvec : p.hvec;

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
    if (W13) build_tab_afrag(afr, threadIdx.x, kGemvThreads);
    __syncthreads();

    // The producer's first claim reads only the routing outputs: the routing launch
    // completed before the launch before this one triggered this kernel, so it
    // overlaps that launch's end.  Everything after the wait may read what that
    // launch wrote (the packed header's verdict among it).
    const bool producer = warp == kCW && lane == 0 && !(p.debug & kDebugNoProducer);
    int *counter = &p.counters[W13 ? 0 : 1];
    int item = 0, total = 0;
    bool ok = true;
    ChunkInfo ci{};
    if (producer) {
        const int nchunks = *p.nchunks;
        item = atomicAdd(counter, 1);
        total = nchunks * U;
        if (item < total) ci = p.chunks[item / U];
    }
    pdl_wait();

    if (warp == kCW) {
        // ---------------------------------------------------------- producer --
        if (producer) {
            // no copy before the packed header's verdict (published by frag_x_kernel,
            // which completed before this wait returned)
            ok = __ldcg(p.hdr_ok) == 1;
            const uint64_t pol = policy_evict_first();
            int it = 0, pslot = 0;
            uint32_t pphase = 0;  // phase of the ring round being filled
            if (!ok) {
                set_status(p.status, MC_ERR_BAD_PACK);
                sh->abort = 1;
            }
            if (item >= total) pdl_trigger();
            while (ok && item < total) {
                // the next item is claimed with this item's second-to-last stage and
                // its chunk read with the last one: both round trips overlap copies
                // already in flight, and a CTA holds at most one unstarted item
                int next = total;
                ChunkInfo next_ci = ci;
                bool have_ci = false;
                const Item I = decode_item<W13>(p, item, U, ci);
                const int nst = (I.nkt + KPS - 1) / KPS, claim_at = nst > 1 ? nst - 2 : 0;
                const int bits = I.ci.bits, NT = I.ci.nv > 8 ? 2 : 1;
                const int e = I.ci.e;
                const int STB = supertile_bytes(bits, group);
                // one column step of both streams is pw contiguous supertiles
                const int pw = W13 ? 2 : w2_pair_width(I.blkA >> 1, nrb);
                const uint8_t *wsrc =
                    p.packed + p.mat_off[e][W13 ? 0 : 2] + supertile_off(W13 ? 0 : 2, I.blkA, I.kt0, KTm, nrb, STB);
                for (int i = 0, st = 0; i < I.nkt; i += KPS, ++it, ++st) {
                    const int slot = pslot;
                    if (it >= S && !wait_or_abort(&empty[slot], pphase ^ 1u, p, sh)) {
                        ok = false;
                        break;
                    }
                    if (++pslot == S) {
                        pslot = 0;
                        pphase ^= 1u;
                    }
                    const int kc = min(KPS, I.nkt - i);
                    sh->slot_item[slot] = item;
                    sh->slot_ci[slot] = I.ci;
                    sh->slot_kc[slot] = kc;
                    uint8_t *dst = ring + (size_t)slot * SB;
                    const uint32_t wb = (uint32_t)(kc * pw * STB), vb = (uint32_t)(kc * VB);
                    mbar_arrive_expect_tx(&full[slot], wb + NT * vb);
                    bulk_g2s_stream(dst, wsrc + (size_t)i * pw * STB, wb, &full[slot], pol);
                    for (int j = 0; j < NT; ++j)
                        bulk_g2s(dst + vec_off0 + j * KPS * VB, vbase + vec_off(I.k, j, I.kt0 + i, KTm, group), vb,
                                 &full[slot]);
                    sh->issued = it + 1;
                    if (st == claim_at) {
                        next = atomicAdd(counter, 1);
                    } else if (st == nst - 1 && next < total) {
                        next_ci = p.chunks[next / U];
                        have_ci = true;
                    }
                }
                if (!ok) break;
                if (!have_ci && next < total) next_ci = p.chunks[next / U];
                // the CTA takes no item after this one: the next kernel may launch
                if (next >= total) pdl_trigger();
                item = next;
                ci = next_ci;
            }
            if (ok) {
                // end marker: one more stage with item -1 and no data
                const int slot = pslot;
                if (it < S || wait_or_abort(&empty[slot], pphase ^ 1u, p, sh)) {
                    sh->slot_item[slot] = -1;
                    mbar_arrive(&full[slot]);
                }
            }
        }
    } else {
        // --------------------------------------------------------- consumers --
        const Ring R{full, empty, ring, S, SB, vec_off0, VB, afr};
        const GroupCtx G{&sh->abort, &sh->cbar, sh->slot_kc, (int)threadIdx.x};
        const int tl = warp;
        int slot = 0, items = 0, cbar_uses = 0;
        uint32_t phase = 0;
        while (true) {
            if (!wait_or_abort(&full[slot], phase, p, sh)) break;
            const int item = sh->slot_item[slot];
            if (item < 0) break;
            const Item I = decode_item<W13>(p, item, U, sh->slot_ci[slot]);
            const int sel = (I.ci.bits - 1) * 2 + (I.ci.nv > 8 ? 1 : 0);
            bool ok;
#define MC_RUN(NT_, B_) \
    run_item<W13, NT_, B_, GPT, (B_ == 16 ? 1 : kKPS)>(p, G, R, I, nrb, tl, lane, slot, phase, hs2, items, cbar_uses)
            if constexpr (DENSE) {
                ok = I.ci.nv > 8 ? MC_RUN(2, 16) : MC_RUN(1, 16);
            } else switch (sel) {
            case 0: ok = MC_RUN(1, 1); break;
            case 1: ok = MC_RUN(2, 1); break;
            case 2: ok = MC_RUN(1, 2); break;
            case 3: ok = MC_RUN(2, 2); break;
            case 4: ok = MC_RUN(1, 3); break;
            default: ok = MC_RUN(2, 3); break;
            }
#undef MC_RUN
            if (!ok) break;
        }
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

// -------------------------------------------------------------- ping-pong --
// gemv_pp_kernel: the quantised-expert GEMV with two consumer groups per CTA.
// Each group (8 consumer warps owning tile tl of both streams, as above, and a
// producer warp) has its own ring of two-step stages and its own epilogue
// barrier and h tiles; both producers claim whole items from the same counter.
// The two groups' warps share the SM's schedulers, so while one group's warps
// drain at a stage boundary or run an item's epilogue, the other group's decode
// and mma keep the pipes issuing.
constexpr int kPPKPS = 2;                  // 128-column steps per stage
constexpr int kPPSlots = 2;                // ring slots per group
constexpr int kPPThreads = 2 * (kCW + 1) * 32;
constexpr int kPPMinPairs = 32;            // 2 T from which a quantised layer takes this kernel

struct PPGroup {
    uint64_t full[kPPSlots], empty[kPPSlots];
    uint64_t cbar;
    volatile int issued;
    int slot_item[kPPSlots], slot_kc[kPPSlots];
    ChunkInfo slot_ci[kPPSlots];
};
struct PPShared {
    PPGroup g[2];
    volatile int abort;
    int producers_done;
};
static_assert(sizeof(PPShared) <= kRingOff, "ping-pong header");

__host__ __device__ inline int pp_slot_bytes(int group)
{
    return kPPKPS * 2 * supertile_bytes(3, group) + 2 * kPPKPS * vec_bytes(group);
}
__host__ __device__ inline size_t pp_smem(int group)
{
    return kRingOff + (size_t)2 * kPPSlots * pp_slot_bytes(group) + 2 * 2 * kHsBytes + 8 * 32 * sizeof(uint2);
}

// One group's producer: claims items from the shared counter (the first one
// already claimed by the caller) and streams them into the group's ring, then
// one end-marker stage.  Counts itself done on the CTA's counter when it takes
// no further item; the second producer to do so lets the next kernel launch.
template <bool W13>
__device__ __forceinline__ void pp_produce(const ExpertParams &p, PPShared *sh, PPGroup &G, uint8_t *ring, int SB,
                                           int VB, int vec_off0, int item, ChunkInfo ci, int total, int U, int nrb,
                                           int KTm, const uint8_t *vbase, int *counter)
{
    const int group = p.group;
    const uint64_t pol = policy_evict_first();
    int it = 0, pslot = 0;
    uint32_t pphase = 0;  // phase of the ring round being filled
    bool ok = true, done = false;
    auto signal_done = [&]() {
        if (!done) {
            done = true;
            if (atomicAdd(&sh->producers_done, 1) == 1) pdl_trigger();
        }
    };
    if (item >= total) signal_done();
    while (item < total) {
        // the next item is claimed with this item's second-to-last stage and its
        // chunk read with the last one (both round trips overlap copies in flight)
        int next = total;
        ChunkInfo next_ci = ci;
        bool have_ci = false;
        const Item I = decode_item<W13>(p, item, U, ci);
        const int nst = (I.nkt + kPPKPS - 1) / kPPKPS, claim_at = nst > 1 ? nst - 2 : 0;
        const int bits = I.ci.bits, NT = I.ci.nv > 8 ? 2 : 1;
        const int STB = supertile_bytes(bits, group);
        const int pw = W13 ? 2 : w2_pair_width(I.blkA >> 1, nrb);
        const uint8_t *wsrc =
            p.packed + p.mat_off[I.ci.e][W13 ? 0 : 2] + supertile_off(W13 ? 0 : 2, I.blkA, I.kt0, KTm, nrb, STB);
        for (int i = 0, st = 0; i < I.nkt; i += kPPKPS, ++it, ++st) {
            const int slot = pslot;
            if (it >= kPPSlots && !wait_or_abort(&G.empty[slot], pphase ^ 1u, p, &sh->abort)) {
                ok = false;
                break;
            }
            if (++pslot == kPPSlots) {
                pslot = 0;
                pphase ^= 1u;
            }
            const int kc = min(kPPKPS, I.nkt - i);
            G.slot_item[slot] = item;
            G.slot_ci[slot] = I.ci;
            G.slot_kc[slot] = kc;
            uint8_t *dst = ring + (size_t)slot * SB;
            const uint32_t wb = (uint32_t)(kc * pw * STB), vb = (uint32_t)(kc * VB);
            mbar_arrive_expect_tx(&G.full[slot], wb + NT * vb);
            bulk_g2s_stream(dst, wsrc + (size_t)i * pw * STB, wb, &G.full[slot], pol);
            for (int j = 0; j < NT; ++j)
                bulk_g2s(dst + vec_off0 + j * kPPKPS * VB, vbase + vec_off(I.k, j, I.kt0 + i, KTm, group), vb,
                         &G.full[slot]);
            G.issued = it + 1;
            if (st == claim_at) {
                next = atomicAdd(counter, 1);
            } else if (st == nst - 1 && next < total) {
                next_ci = p.chunks[next / U];
                have_ci = true;
            }
        }
        if (!ok) return;
        if (!have_ci && next < total) next_ci = p.chunks[next / U];
        if (next >= total) signal_done();
        item = next;
        ci = next_ci;
    }
    // end marker: one more stage with item -1 and no data
    const int slot = pslot;
    if (it < kPPSlots || wait_or_abort(&G.empty[slot], pphase ^ 1u, p, &sh->abort)) {
        G.slot_item[slot] = -1;
        mbar_arrive(&G.full[slot]);
    }
}

template <bool W13, int GPT>
__global__ void __launch_bounds__(kPPThreads, 1) gemv_pp_kernel(ExpertParams p)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    PPShared *sh = reinterpret_cast<PPShared *>(smem);
    const int group = p.group;
    const int SB = pp_slot_bytes(group), VB = vec_bytes(group);
    const int vec_off0 = kPPKPS * 2 * supertile_bytes(3, group);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = warp / (kCW + 1), lw = warp % (kCW + 1);  // group, warp within the group (kCW: producer)
    PPGroup &G = sh->g[g];
    uint8_t *ring = smem + kRingOff + (size_t)g * kPPSlots * SB;
    __half *hs2 = reinterpret_cast<__half *>(smem + kRingOff + (size_t)2 * kPPSlots * SB + (size_t)g * 2 * kHsBytes);
    uint2 *afr = reinterpret_cast<uint2 *>(smem + kRingOff + (size_t)2 * kPPSlots * SB + 4 * kHsBytes);
    const int nrb = W13 ? p.F / kBlockRows : p.H / kBlockRows;  // 128-row blocks of the matrix
    const int U = W13 ? nrb : ((nrb + 1) / 2) * p.KS;
    const int KTm = W13 ? p.H / kTileK : p.F / kTileK;  // column steps of the matrix and its vectors
    const uint8_t *vbase = W13 ? p.xvec : p.hvec;

    if (threadIdx.x == 0) {
        for (int gg = 0; gg < 2; ++gg) {
            for (int s = 0; s < kPPSlots; ++s) {
                mbar_init(&sh->g[gg].full[s], 1);
                mbar_init(&sh->g[gg].empty[s], kCW);
            }
            mbar_init(&sh->g[gg].cbar, kCW);
            sh->g[gg].issued = 0;
        }
        sh->abort = 0;
        sh->producers_done = 0;
        fence_mbar_init();
    }
    if (W13) build_tab_afrag(afr, threadIdx.x, kPPThreads);
    __syncthreads();

    // Each producer's first claim reads only the routing outputs (complete before
    // this kernel was let launch), so it overlaps the end of the launch before.
    const bool producer = lw == kCW && lane == 0 && !(p.debug & kDebugNoProducer);
    int *counter = &p.counters[W13 ? 0 : 1];
    int item = 0, total = 0;
    bool ok = true;
    ChunkInfo ci{};
    if (producer) {
        const int nchunks = *p.nchunks;
        item = atomicAdd(counter, 1);
        total = nchunks * U;
        if (item < total) ci = p.chunks[item / U];
    }
    pdl_wait();

    if (lw == kCW) {
        // ---------------------------------------------------------- producer --
        if (producer) {
            // no copy before the packed header's verdict (published by frag_x_kernel,
            // which completed before this wait returned)
            ok = __ldcg(p.hdr_ok) == 1;
            if (!ok) {
                set_status(p.status, MC_ERR_BAD_PACK);
                sh->abort = 1;
            } else {
                pp_produce<W13>(p, sh, G, ring, SB, VB, vec_off0, item, ci, total, U, nrb, KTm, vbase, counter);
            }
        }
    } else {
        // --------------------------------------------------------- consumers --
        const Ring R{G.full, G.empty, ring, kPPSlots, SB, vec_off0, VB, afr};
        const GroupCtx Gc{&sh->abort, &G.cbar, G.slot_kc, lw * 32 + lane};
        const int tl = lw;
        int slot = 0, items = 0, cbar_uses = 0;
        uint32_t phase = 0;
        while (true) {
            if (!wait_or_abort(&G.full[slot], phase, p, &sh->abort)) break;
            const int it_id = G.slot_item[slot];
            if (it_id < 0) break;
            const Item I = decode_item<W13>(p, it_id, U, G.slot_ci[slot]);
            const int sel = (I.ci.bits - 1) * 2 + (I.ci.nv > 8 ? 1 : 0);
            bool run_ok;
#define MC_RUN(NT_, B_) \
    run_item<W13, NT_, B_, GPT, kPPKPS>(p, Gc, R, I, nrb, tl, lane, slot, phase, hs2, items, cbar_uses)
            switch (sel) {
            case 0: run_ok = MC_RUN(1, 1); break;
            case 1: run_ok = MC_RUN(2, 1); break;
            case 2: run_ok = MC_RUN(1, 2); break;
            case 3: run_ok = MC_RUN(2, 2); break;
            case 4: run_ok = MC_RUN(1, 3); break;
            default: run_ok = MC_RUN(2, 3); break;
            }
#undef MC_RUN
            if (!run_ok) break;
        }
    }
    __syncthreads();
    // On an abort, let copies that were issued but never consumed land before the
    // CTA's shared memory is released (bounded).
    if (threadIdx.x == 0 && sh->abort) {
        for (int gg = 0; gg < 2; ++gg) {
            PPGroup &Q = sh->g[gg];
            for (int it = max(0, Q.issued - kPPSlots); it < Q.issued; ++it) {
                const uint64_t t0 = globaltimer_ns();
                while (!mbar_try_wait(&Q.full[it % kPPSlots], (it / kPPSlots) & 1))
                    if (globaltimer_ns() - t0 > p.timeout_ns) break;
            }
        }
    }
}

// ---------------------------------------------------------------- combine --
// y[t] = w0 * o[p(t,0)] + w1 * o[p(t,1)] (second term absent when pruned),
// summing the column splits of the W2 pass in a fixed order (Eq. 1 with Eq. 5);
// with a residual (the pre-norm stack), y[t] = resid[t] + that, rounded to bf16
// first (the layer's own output) and once more after the fp32 add.
//   Every load of a slot's column splits is issued before the first is used.
__global__ void __launch_bounds__(256) combine_kernel(CombineParams p)
{
    pdl_trigger();
    pdl_wait();
    const int H8 = p.H / 8;
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= p.T * H8) return;
    const int t = idx / H8, c = (idx % H8) * 8;
    float out[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    const int2 q2 = *reinterpret_cast<const int2 *>(p.inv + 2 * t);
    const float2 w2 = *reinterpret_cast<const float2 *>(p.w + 2 * t);
    for (int slot = 0; slot < 2; ++slot) {
        const int q = slot ? q2.y : q2.x;
        if (q < 0) continue;
        const float wt = slot ? w2.y : w2.x;
        float4 a[kMaxKS], b[kMaxKS];
#pragma unroll
        for (int ks = 0; ks < kMaxKS; ++ks)
            if (ks < p.KS) {
                const float4 *src = reinterpret_cast<const float4 *>(p.opart + ((size_t)ks * p.Pmax + q) * p.H + c);
                a[ks] = src[0];
                b[ks] = src[1];
            }
        float o[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
        for (int ks = 0; ks < kMaxKS; ++ks)
            if (ks < p.KS) {
                o[0] += a[ks].x; o[1] += a[ks].y; o[2] += a[ks].z; o[3] += a[ks].w;
                o[4] += b[ks].x; o[5] += b[ks].y; o[6] += b[ks].z; o[7] += b[ks].w;
            }
#pragma unroll
        for (int k = 0; k < 8; ++k) out[k] = fmaf(wt, o[k], out[k]);
    }
    __nv_bfloat16 r[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) r[k] = __float2bfloat16_rn(out[k]);
    if (p.resid) {
        const uint4 rv = *reinterpret_cast<const uint4 *>(p.resid + (size_t)t * p.H + c);
        const __nv_bfloat16 *rb = reinterpret_cast<const __nv_bfloat16 *>(&rv);
#pragma unroll
        for (int k = 0; k < 8; ++k) r[k] = __float2bfloat16_rn(__bfloat162float(rb[k]) + __bfloat162float(r[k]));
    }
    *reinterpret_cast<uint4 *>(p.y + (size_t)t * p.H + c) = *reinterpret_cast<uint4 *>(r);
}

// The same for decode-sized calls (T <= 64): one thread per 4 output columns in
// 128-thread CTAs, so that the grid spreads over the SMs, and every split of
// both slots loaded before the first is used (one round trip after the routing
// outputs).  Same summation order as combine_kernel.
constexpr int kCombine4MaxT = 64;

__global__ void __launch_bounds__(128) combine4_kernel(CombineParams p)
{
    pdl_trigger();
    pdl_wait();
    const int H4 = p.H / 4;
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= p.T * H4) return;
    const int t = idx / H4, c = (idx % H4) * 4;
    const int2 q2 = *reinterpret_cast<const int2 *>(p.inv + 2 * t);
    const float2 w2 = *reinterpret_cast<const float2 *>(p.w + 2 * t);
    const uint2 rv = p.resid ? *reinterpret_cast<const uint2 *>(p.resid + (size_t)t * p.H + c) : make_uint2(0, 0);
    float4 a[2][kMaxKS];
#pragma unroll
    for (int slot = 0; slot < 2; ++slot) {
        const int q = slot ? q2.y : q2.x;
#pragma unroll
        for (int ks = 0; ks < kMaxKS; ++ks)
            if (ks < p.KS && q >= 0)
                a[slot][ks] = *reinterpret_cast<const float4 *>(p.opart + ((size_t)ks * p.Pmax + q) * p.H + c);
    }
    float out[4] = {0, 0, 0, 0};
#pragma unroll
    for (int slot = 0; slot < 2; ++slot) {
        if ((slot ? q2.y : q2.x) < 0) continue;
        const float wt = slot ? w2.y : w2.x;
        float o[4] = {0, 0, 0, 0};
#pragma unroll
        for (int ks = 0; ks < kMaxKS; ++ks)
            if (ks < p.KS) {
                o[0] += a[slot][ks].x;
                o[1] += a[slot][ks].y;
                o[2] += a[slot][ks].z;
                o[3] += a[slot][ks].w;
            }
#pragma unroll
        for (int k = 0; k < 4; ++k) out[k] = fmaf(wt, o[k], out[k]);
    }
    __nv_bfloat16 r[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) r[k] = __float2bfloat16_rn(out[k]);
    if (p.resid) {
        const __nv_bfloat16 *rb = reinterpret_cast<const __nv_bfloat16 *>(&rv);
#pragma unroll
        for (int k = 0; k < 4; ++k) r[k] = __float2bfloat16_rn(__bfloat162float(rb[k]) + __bfloat162float(r[k]));
    }
    *reinterpret_cast<uint2 *>(p.y + (size_t)t * p.H + c) = *reinterpret_cast<uint2 *>(r);
}

// -------------------------------------------------------------- launchers --

int launch_gemv(ExpertParams ep, cudaStream_t st)
{
    int dev = 0, maxsm = 0, nsm = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&maxsm, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "device query: %s", cudaGetErrorString(err));
    // 16-bit experts are all or none of a layer (check_bits).  Quantised layers of
    // >= 16 tokens run the two-group kernel: measured on the Mixtral-8x7b layer at
    // 16 tokens 127.9 K against 120.8 K tokens/s; at 1 and 4 tokens it was slower
    // (15.3 / 33.2 K against 17.2 / 36.3 K: with about one item per SM one group
    // idles and the other's two-slot ring is too shallow to keep the stream busy)
    const bool dense = ep.bits[0] == 16;
    if (!dense && ep.Pmax >= kPPMinPairs) {
        const size_t smp = pp_smem(ep.group);
        if ((size_t)maxsm < smp) return set_error(MC_ERR_UNSUPPORTED, "not enough shared memory for the GEMV rings");
        auto p13 = ep.group == 64 ? gemv_pp_kernel<true, 2> : gemv_pp_kernel<true, 1>;
        auto p2 = ep.group == 64 ? gemv_pp_kernel<false, 2> : gemv_pp_kernel<false, 1>;
        err = cudaFuncSetAttribute(p13, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smp);
        if (err == cudaSuccess) err = cudaFuncSetAttribute(p2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smp);
        if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(err));
        ep.nslots = kPPSlots;
        profile_begin(kKFragX, st);
        err = launch_k(frag_x_kernel, dim3(ep.max_chunks, ep.H / kTileK), dim3(256), 0, st, ep);
        profile_end(kKFragX, st);
        if (err == cudaSuccess) {
            profile_begin(kKGemvW13, st);
            err = launch_k(p13, dim3(nsm), dim3(kPPThreads), smp, st, ep);
            profile_end(kKGemvW13, st);
        }
        if (err == cudaSuccess) {
            profile_begin(kKGemvW2, st);
            err = launch_k(p2, dim3(nsm), dim3(kPPThreads), smp, st, ep);
            profile_end(kKGemvW2, st);
        }
        if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "GEMV launch: %s", cudaGetErrorString(err));
        return MC_OK;
    }
    int nslots = (int)((maxsm - gemv_smem(0, ep.group, dense)) / slot_bytes(ep.group, dense));
    nslots = nslots > kMaxSlots ? kMaxSlots : nslots;
    if (nslots < 2) return set_error(MC_ERR_UNSUPPORTED, "not enough shared memory for the GEMV ring");
    ep.nslots = nslots;
    const size_t sm = gemv_smem(nslots, ep.group, dense);
    auto k13 = dense ? (ep.group == 64 ? gemv_kernel<true, 2, true> : gemv_kernel<true, 1, true>)
                     : (ep.group == 64 ? gemv_kernel<true, 2, false> : gemv_kernel<true, 1, false>);
    auto k2 = dense ? (ep.group == 64 ? gemv_kernel<false, 2, true> : gemv_kernel<false, 1, true>)
                    : (ep.group == 64 ? gemv_kernel<false, 2, false> : gemv_kernel<false, 1, false>);
    err = cudaFuncSetAttribute(k13, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (err == cudaSuccess) err = cudaFuncSetAttribute(k2, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(err));

    profile_begin(kKFragX, st);
    err = launch_k(frag_x_kernel, dim3(ep.max_chunks, ep.H / kTileK), dim3(256), 0, st, ep);
    profile_end(kKFragX, st);
    if (err == cudaSuccess) {
        profile_begin(kKGemvW13, st);
        err = launch_k(k13, dim3(nsm), dim3(kGemvThreads), sm, st, ep);
        profile_end(kKGemvW13, st);
    }
    if (err == cudaSuccess) {
        profile_begin(kKGemvW2, st);
        err = launch_k(k2, dim3(nsm), dim3(kGemvThreads), sm, st, ep);
        profile_end(kKGemvW2, st);
    }
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "GEMV launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

int launch_combine(const CombineParams &cp, cudaStream_t st)
{
    if (cp.KS < 1 || cp.KS > kMaxKS) return set_error(MC_ERR_INVALID_ARG, "combine: %d column splits", cp.KS);
    profile_begin(kKCombine, st);
    cudaError_t err;
    if (cp.T <= kCombine4MaxT) {
        const int n = cp.T * (cp.H / 4);
        err = launch_k(combine4_kernel, dim3((n + 127) / 128), dim3(128), 0, st, cp);
    } else {
        const int n = cp.T * (cp.H / 8);
        err = launch_k(combine_kernel, dim3((n + 255) / 256), dim3(256), 0, st, cp);
    }
    profile_end(kKCombine, st);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "combine launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

}  // namespace mc
