// mc_importance.cu -- the token importance of Sec. 2.3.2 (Eq. 6), the mask of the
// most important tokens that ODP never prunes, and the Eq. 5 threshold taken from
// calibration routing weights (Sec. 2.3.1).
//
//   I_j = ||t_j||_1 * (1 / (L - j)) * sum_{i=j}^{L-1} Abar[i][j]      (0-based j)
//   Abar = the mean over the nh heads of the attention probabilities attn[h][i][j]
//          (query i, key j; a causal map, so key j is seen by queries i >= j)
//
// colsum_kernel: one CTA per (32 key columns, head, 256-row chunk), 32 columns
//   x 8 row lanes, reading 128 contiguous bytes of a row per warp; each CTA adds
//   its partial column sums to a fixed-point (2^-40) int64 accumulator with
//   integer atomics, which commute, so the result does not depend on the order
//   the CTAs run in (the partial of a CTA is a fixed sequence of fp32 adds).
// importance_kernel: one warp per token: the l1 norm of t_j, times the column mean.
// select_kernel: one CTA: radix select of the n-th largest importance (8 bits per
//   pass over the float bit patterns, which order like the values for
//   non-negative floats), then the mask: every token above that value and, among
//   the tokens equal to it, the lowest indices until n are chosen.
// rank_select_kernel (L <= 1024): the same mask from each token's rank, the number
//   of tokens with a larger bit pattern or an equal one at a lower index, counted
//   over the importances held in shared memory (one pass, no histogram rounds).
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "mc_host.h"
#include "mc_kernels.h"
#include "mc_profile.h"

namespace mc {

constexpr int kColTile = 32, kRowChunk = 256, kRowLanes = 8;
constexpr double kFix = 1099511627776.0;  // 2^40: fixed-point scale of the column sums

__global__ void zero_kernel(unsigned long long *acc, int L)
{
    pdl_trigger();
    pdl_wait();
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j < L) acc[j] = 0ull;
}

__global__ void __launch_bounds__(kColTile * kRowLanes) colsum_kernel(const float *attn, int L, unsigned long long *acc)
{
    __shared__ float part[kRowLanes][kColTile + 1];
    pdl_trigger();
    pdl_wait();
    const int c = threadIdx.x & 31, r = threadIdx.x >> 5;
    const int j0 = blockIdx.x * kColTile, j = j0 + c, h = blockIdx.y;
    const int i0 = max(j0, blockIdx.z * kRowChunk), i1 = min(L, (blockIdx.z + 1) * kRowChunk);
    if (i0 >= i1) return;  // the chunk lies above the tile's diagonal (whole CTA)
    const float *a = attn + (size_t)h * L * L;
    float s = 0.f;
    if (j < L)
#pragma unroll 4
        for (int i = i0 + r; i < i1; i += kRowLanes)
            if (i >= j) s += a[(size_t)i * L + j];
    part[r][c] = s;
    __syncthreads();
    if (r == 0 && j < L) {
        float t = 0.f;
#pragma unroll
        for (int q = 0; q < kRowLanes; ++q) t += part[q][c];
        atomicAdd(acc + j, (unsigned long long)llrint((double)t * kFix));
    }
}

__global__ void __launch_bounds__(256) importance_kernel(const __nv_bfloat16 *t, int L, int H, int nh,
                                                         const unsigned long long *acc, float *imp)
{
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31, j = blockIdx.x * 8 + (threadIdx.x >> 5);
    if (j >= L) return;
    const __nv_bfloat16 *row = t + (size_t)j * H;
    float l1 = 0.f;
    for (int h = lane; h < H; h += 32) l1 += fabsf(__bfloat162float(row[h]));
    for (int m = 16; m >= 1; m >>= 1) l1 += __shfl_xor_sync(0xffffffffu, l1, m);
    if (lane == 0) imp[j] = (float)((double)l1 * ((double)acc[j] / kFix) / ((double)nh * (double)(L - j)));
}

__global__ void __launch_bounds__(1024) select_kernel(const float *imp, int L, int n, uint8_t *mask)
{
    __shared__ int hist[256];
    __shared__ unsigned s_prefix, s_bits;
    __shared__ int s_k, s_base;
    __shared__ int wsum[32];
    pdl_trigger();
    pdl_wait();
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
        s_prefix = 0;
        s_bits = 0;
        s_k = n;
    }
    __syncthreads();
    // the n-th largest key (n >= 1): 4 passes of 8 bits, most significant first
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int b = tid; b < 256; b += blockDim.x) hist[b] = 0;
        __syncthreads();
        const unsigned prefix = s_prefix, bits = s_bits;
        for (int j = tid; j < L; j += blockDim.x) {
            const unsigned u = __float_as_uint(imp[j]);
            if ((u & bits) == prefix) atomicAdd(&hist[(u >> shift) & 255], 1);
        }
        __syncthreads();
        if (tid == 0) {
            int k = s_k, cum = 0, b = 255;
            for (; b > 0; --b) {
                if (cum + hist[b] >= k) break;
                cum += hist[b];
            }
            s_k = k - cum;  // still to take among the keys of bin b
            s_prefix = prefix | ((unsigned)b << shift);
            s_bits = bits | (255u << shift);
        }
        __syncthreads();
    }
    const unsigned key = s_prefix;
    const int k = s_k;  // tokens equal to key to select, lowest indices first
    if (tid == 0) s_base = 0;
    __syncthreads();
    for (int j0 = 0; j0 < L; j0 += blockDim.x) {
        const int j = j0 + tid;
        const unsigned u = j < L ? __float_as_uint(imp[j]) : 0u;
        const int eq = j < L && u == key;
        // exclusive prefix count of eq over the chunk, in index order
        const unsigned bal = __ballot_sync(0xffffffffu, eq);
        if (lane == 0) wsum[warp] = __popc(bal);
        __syncthreads();
        int before = s_base + __popc(bal & ((1u << lane) - 1));
        for (int w = 0; w < warp; ++w) before += wsum[w];
        if (j < L) mask[j] = (u > key || (eq && before < k)) ? 1 : 0;
        __syncthreads();
        if (tid == 0) {
            int s = 0;
            for (int w = 0; w < (int)(blockDim.x >> 5); ++w) s += wsum[w];
            s_base += s;
        }
        __syncthreads();
    }
}

constexpr int kRankMaxL = 1024;

__global__ void __launch_bounds__(1024) rank_select_kernel(const float *imp, int L, int n, uint8_t *mask)
{
    __shared__ unsigned key[kRankMaxL];
    pdl_trigger();
    pdl_wait();
    for (int j = threadIdx.x; j < L; j += blockDim.x) key[j] = __float_as_uint(imp[j]);
    __syncthreads();
    for (int j = threadIdx.x; j < L; j += blockDim.x) {
        const unsigned kj = key[j];
        int r = 0;
        for (int i = 0; i < L; ++i) {
            const unsigned ki = key[i];  // the same word for every lane: a broadcast
            r += ki > kj || (ki == kj && i < j);
        }
        mask[j] = r < n ? 1 : 0;
    }
}

__global__ void fill_kernel(uint8_t *mask, int L, uint8_t v)
{
    pdl_trigger();
    pdl_wait();
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j < L) mask[j] = v;
}

}  // namespace mc

using namespace mc;

extern "C" {

size_t mc_token_importance_workspace_size(int L) { return L <= 0 ? 0 : (((size_t)L * 8 + 255) & ~(size_t)255); }

int mc_token_importance(const void *t, const float *attn, int L, int H, int nh, float protect_frac,
                        float *importance, uint8_t *mask, void *workspace, size_t ws_bytes, void *stream)
{
    clear_error();
    if (L < 0 || H <= 0 || nh <= 0 || nh > 65535 || !(protect_frac >= 0.f && protect_frac <= 1.f))
        return set_error(MC_ERR_INVALID_ARG, "L=%d H=%d nh=%d protect_frac=%g", L, H, nh, (double)protect_frac);
    if (L == 0) return MC_OK;
    if (!t || !attn || !importance || !workspace) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    if (ws_bytes < mc_token_importance_workspace_size(L))
        return set_error(MC_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu", ws_bytes,
                         mc_token_importance_workspace_size(L));
    if ((double)nh * L * L > 9.0e18 / 4 || (double)nh * L > 2.0e9 * kRowChunk)
        return set_error(MC_ERR_INVALID_ARG, "attention map too large");
    cudaStream_t st = (cudaStream_t)stream;
    unsigned long long *acc = (unsigned long long *)workspace;
    const dim3 grid((L + kColTile - 1) / kColTile, nh, (L + kRowChunk - 1) / kRowChunk);
    profile_begin(kKImportance, st);
    cudaError_t err = launch_k(zero_kernel, dim3((L + 255) / 256), dim3(256), 0, st, acc, L);
    profile_end(kKImportance, st);
    if (err == cudaSuccess) {
        profile_begin(kKImportance, st);
        err = launch_k(colsum_kernel, grid, dim3(kColTile * kRowLanes), 0, st, attn, L, acc);
        profile_end(kKImportance, st);
    }
    if (err == cudaSuccess) {
        profile_begin(kKImportance, st);
        err = launch_k(importance_kernel, dim3((L + 7) / 8), dim3(256), 0, st, (const __nv_bfloat16 *)t, L, H, nh,
                       (const unsigned long long *)acc, importance);
        profile_end(kKImportance, st);
    }
    if (err == cudaSuccess && mask) {
        // ceil(frac * L); a product within 1e-6 of an integer counts as that integer
        const int n = (int)ceil((double)protect_frac * L - 1e-6);
        profile_begin(kKImportance, st);
        if (n <= 0 || n >= L)
            err = launch_k(fill_kernel, dim3((L + 255) / 256), dim3(256), 0, st, mask, L, (uint8_t)(n > 0));
        else if (L <= kRankMaxL)
            err = launch_k(rank_select_kernel, dim3(1), dim3(1024), 0, st, (const float *)importance, L, n, mask);
        else
            err = launch_k(select_kernel, dim3(1), dim3(1024), 0, st, (const float *)importance, L, n, mask);
        profile_end(kKImportance, st);
    }
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "importance launch: %s", cudaGetErrorString(err));
    return MC_OK;
}

int mc_odp_threshold_host(const float *w_host, const uint8_t *mask_host, int T, double q, float *mu_out)
{
    clear_error();
    if (T < 0 || !(q >= 0.0 && q <= 1.0)) return set_error(MC_ERR_INVALID_ARG, "T=%d q=%g", T, q);
    if (!w_host || !mu_out) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    std::vector<double> r;
    r.reserve((size_t)T);
    for (int t = 0; t < T; ++t) {
        if (mask_host && mask_host[t] != 0) continue;  // protected or dropped: never pruned
        const double w0 = w_host[2 * t], w1 = w_host[2 * t + 1];
        if (w0 > 0.0) r.push_back(w1 / w0);
    }
    if (r.empty()) return set_error(MC_ERR_INVALID_ARG, "no prunable token with a positive primary weight");
    std::sort(r.begin(), r.end());
    // linear interpolation between the order statistics around q * (n - 1)
    const double pos = q * (double)(r.size() - 1);
    const size_t lo = (size_t)floor(pos), hi = std::min(lo + 1, r.size() - 1);
    *mu_out = (float)(r[lo] + (pos - (double)lo) * (r[hi] - r[lo]));
    return MC_OK;
}

}  // extern "C"
