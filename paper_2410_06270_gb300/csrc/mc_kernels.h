// mc_kernels.h -- kernel parameter blocks and host launchers shared by the
// translation units of the library (host side: mc_api.cu).
#pragma once
#include <cuda_runtime.h>

#include "mc_device.cuh"

namespace mc {

// Activations of up to 16 pairs of one expert ("chunk") are processed together:
// two mma n-tiles of 8.  NT = 1 when the chunk has at most 8 pairs.
constexpr int kChunk = 16;

// One chunk of one expert, written by permute_kernel in the order the expert
// kernels schedule them (experts with more bits first).
struct ChunkInfo {
    int32_t e;          // expert
    int32_t pair_base;  // first pair (position in perm) of the chunk
    int32_t nv;         // valid pairs, 1..16
    int32_t bits;
};

// Fragment-ordered activations of one chunk and one 128-column tile:
//   frag [j (2)][s (8)][lane (32)] x 8 bytes = 4 fp16 (B operand of mma k-step s,
//   n-tile j); j-major so that an NT = 1 chunk copies only the first 2 KB.
constexpr int kFragBytes = 2 * 8 * 32 * 8;
// Offset tables of one chunk and one tile: [n (16)][group-in-tile][8 floats].
__host__ __device__ inline int tab_bytes(int group) { return kChunk * (kTileK / group) * kTabFloats * 4; }

// Vector block of the mma.sync path: one (chunk, n-tile j, 128-column step),
//   [fragments of pairs 8j..8j+7: 256 x 8 bytes][their offset tables [8][g][8]]
// stored [chunk][j (2)][column step] so that consecutive steps are contiguous.
constexpr int kVecFragBytes = 2048;
__host__ __device__ inline int vec_bytes(int group) { return kVecFragBytes + 8 * (kTileK / group) * kTabFloats * 4; }
__host__ __device__ inline size_t vec_off(int k, int j, int kt, int KT, int group)
{
    return (((size_t)k * 2 + j) * KT + kt) * (size_t)vec_bytes(group);
}

struct RouteParams {
    const __nv_bfloat16 *x;     // [T, H]
    const __nv_bfloat16 *gate;  // [E, H]
    int T, H, E;
    float neg_log_mu;           // prune iff (l0 - l1) > neg_log_mu  (+inf: never)
    const uint8_t *protect;     // [T] or null
    int32_t *idx;               // [T, 2]
    float *w;                   // [T, 2]
    uint8_t *pruned;            // [T]
    int32_t *idx_out;           // optional copies
    float *w_out;
    uint8_t *pruned_out;
    // optional pre-norm (the stack): x = RMSNorm(h_in) with gamma and eps, computed
    // here, written to x (which the expert kernels then read) and routed on
    const __nv_bfloat16 *h_in;  // [T, H] or null
    const __nv_bfloat16 *gamma; // [H]
    float eps;
};

struct PermuteParams {
    const int32_t *idx;
    const uint8_t *pruned;
    int T, E;
    int8_t bits[kMaxE];
    int32_t *offsets;     // [E+1]
    int32_t *perm;        // [2T]
    int32_t *inv;         // [2T] or null
    ChunkInfo *chunks;    // [max_chunks] or null
    int32_t *nchunks;     // [1]
    int32_t *counters;    // [4] work counters of the expert kernels, reset here
    int chunk;            // pairs per work chunk: 16 (GEMV paths) or 128 (prefill GEMM)
};

// Decode-path expert kernels (persistent, mma.sync).
struct ExpertParams {
    const uint8_t *packed;
    uint64_t mat_off[kMaxE][3];
    int8_t bits[kMaxE];
    int E, H, F, group;
    const ChunkInfo *chunks;
    const int32_t *nchunks;
    int32_t *counters;
    const __nv_bfloat16 *x;  // [T, H]
    const int32_t *perm;     // [P]
    uint8_t *xvec;           // [max_chunks][2][H/128] vector blocks of x (mma.sync path)
    uint8_t *hvec;           // [max_chunks][2][F/128] vector blocks of h (mma.sync path)
    uint8_t *ximg;           // [max_blocks][H/128] 32 KB activation images (prefill path)
    uint8_t *himg;           // [max_blocks][F/128] 32 KB h images (prefill path)
    int max_blocks;          // token blocks of <= 128 pairs (prefill path)
    float *opart;            // [KS, Pmax, H]  expert outputs (fp32), pair order
    int KS;                  // column splits of the W2 pass
    int Pmax;                // 2 * T
    int max_chunks;
    int nslots;              // stages of the shared-memory ring
    int32_t *status;
    int32_t *hdr_ok;         // the packed header's verdict for this call (1: matches), written by frag_x_kernel
    uint64_t timeout_ns;
    int debug;               // test hooks (kDebugNoProducer)
};

// Word of the 256-byte status area at the start of a workspace that holds the
// packed header's verdict (the status word itself is word 0).
constexpr int kHdrOkWord = 16;

constexpr int kDebugNoProducer = 1;  // the copy producer never issues: waits expire
constexpr int kDebugNoPdl = 2;       // launch without programmatic dependent launch
constexpr int kDebugRouteFused = 4;  // mc_route takes the single-launch routing for T <= 64

constexpr int kMaxKS = 8;  // column splits of the W2 GEMV pass, at most

struct CombineParams {
    const float *opart;   // [KS, Pmax, H]
    const float *w;       // [T, 2]
    const int32_t *inv;   // [2T]
    int T, H, KS, Pmax;
    __nv_bfloat16 *y;     // [T, H]
    // optional residual: y = resid + (the layer output rounded to bf16), added in
    // fp32 and rounded once more (resid may alias y); null: y = the layer output
    const __nv_bfloat16 *resid;
};

// Launch with programmatic stream serialisation (unless switched off by
// mc_set_debug bit 2): the kernel's launch and prologue overlap the end of the
// kernel before it on the stream; the kernel itself calls pdl_wait before it
// reads or writes global memory.
bool pdl_enabled();
template <typename... P, typename... A>
inline cudaError_t launch_k(void (*kernel)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, A &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<A &&>(args)...);
}

// Host launchers: MC_OK or an MC_ERR_* code with the message set.
// done: a zeroed device counter enabling the single-launch routing + placement for
// T <= 64 (left at zero), or NULL for two launches.
int launch_route(const RouteParams &rp, const PermuteParams &pp, cudaStream_t st, int32_t *done = nullptr);
int launch_gemv(ExpertParams ep, cudaStream_t st);   // mma.sync path
int launch_gemm(ExpertParams ep, cudaStream_t st);   // prefill path (tcgen05 grouped GEMM)
size_t img_buffer_bytes(int max_blocks, int cols);
int max_blocks_for(int T, int E);
int launch_combine(const CombineParams &cp, cudaStream_t st);
int max_chunks_for(int T, int E);
int32_t *route_done_word();  // mc_route's arrival word for the single-launch routing
// Column splits of the W2 GEMV pass: the most a workspace for T tokens holds, and
// the count a forward picks (the one whose work items fill the SMs' last wave
// best, among the divisors of F/128 that leave every item >= 8 column steps).
int max_ks(const mc_shape *s, int T);
int choose_ks(const mc_shape *s, int T, int nsm);
// The pre-norm residual form of one layer, for mc_stack_forward: with norm_in,
// the routing launch computes x = RMSNorm(norm_in) (gamma, eps; bit for bit
// mc_rmsnorm) into the buffer x and routes on it; with resid, the last kernel
// writes y = resid + the layer output (resid may alias y).  Both null:
// mc_moe_forward itself.
struct LayerPrePost {
    const void *norm_in;  // bf16 [T, H] or null (16-byte aligned)
    const void *gamma;    // bf16 [H] (16-byte aligned)
    float eps;
    const void *resid;    // bf16 [T, H] or null
};
int moe_forward_ex(const void *x, const void *gate_w, int T, const mc_shape *shape, const int8_t *bits_host,
                   const void *packed_dev, float mu, const uint8_t *protect, void *y, const LayerPrePost *pp,
                   void *workspace, size_t ws_bytes, int32_t *topk_idx_out, float *topk_w_out, uint8_t *pruned_out,
                   void *stream);
// The test hooks of mc_set_debug: its flags and the bound on device waits.
int debug_flags();
uint64_t wait_bound_ns();

}  // namespace mc
