// mc_kernels.h -- kernel parameter blocks and launch declarations shared by the
// translation units of the library (host side: mc_api.cu).
#pragma once
#include <cuda_runtime.h>

#include "mc_device.cuh"

namespace mc {

struct RouteParams {
    const __nv_bfloat16 *x;     // [T, H]
    const __nv_bfloat16 *gate;  // [E, H]
    int T, H, E, group;
    float neg_log_mu;           // prune iff (l0 - l1) > neg_log_mu  (+inf: never)
    const uint8_t *protect;     // [T] or null
    int32_t *idx;               // [T, 2]
    float *w;                   // [T, 2]
    uint8_t *pruned;            // [T]
    int32_t *idx_out;           // optional copies
    float *w_out;
    uint8_t *pruned_out;
    __half *xh;                 // [T, H] fp16 copy, or null (routing only)
    float *xtab;                // [T, H/group, 8]
    int32_t *status;
};

struct PermuteParams {
    const int32_t *idx;
    const uint8_t *pruned;
    int T, E;
    int32_t *offsets;  // [E+1]
    int32_t *perm;     // [2T]
    int32_t *inv;      // [2T]
};

// Expert GEMV/GEMM work description shared by the decode and prefill kernels.
struct ExpertParams {
    const uint8_t *packed;
    uint64_t mat_off[kMaxE][3];
    int8_t bits[kMaxE];
    int E, H, F, group;
    const int32_t *offsets;  // [E+1]
    const int32_t *perm;     // [P]
    const __half *xh;        // [T, H]
    const float *xtab;       // [T, H/g, 8]
    __half *h;               // [Pmax, F]   SwiGLU output, pair order
    float *htab;             // [Pmax, F/g, 8]
    float *opart;            // [KS, Pmax, H]  expert outputs (fp32), pair order
    int KS;                  // column splits of the W2 pass
    int Pmax;                // 2 * T
    int32_t *status;
    uint64_t timeout_ns;
    int debug;               // test hooks (kDebugNoProducer)
};

constexpr int kDebugNoProducer = 1;  // the copy producer never issues: waits expire

struct CombineParams {
    const float *opart;   // [KS, Pmax, H]
    const float *w;       // [T, 2]
    const int32_t *inv;   // [2T]
    int T, H, KS, Pmax;
    __nv_bfloat16 *y;     // [T, H]
};

__global__ void route_kernel(RouteParams p);
__global__ void permute_kernel(PermuteParams p);
__global__ void combine_kernel(CombineParams p);

// decode (mma.sync) expert kernels; NT = n-tiles of 8 pairs per expert.
// Host launchers return MC_OK or an MC_ERR_* code with the message set.
int launch_gemv(const ExpertParams &ep, int NT, cudaStream_t st);
int launch_combine(const CombineParams &cp, cudaStream_t st);
size_t gemv_smem_bytes(int NT, bool w13, const ExpertParams &p);

}  // namespace mc
