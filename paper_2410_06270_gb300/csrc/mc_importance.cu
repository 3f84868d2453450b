// mc_importance.cu -- the token importance of Sec. 2.3.2 (Eq. 6), the mask of the
// most important tokens that ODP never prunes, and the Eq. 5 threshold taken from
// calibration routing weights (Sec. 2.3.1).
//
//   I_j = ||t_j||_1 * (1 / (L - j)) * sum_{i=j}^{L-1} Abar[i][j]      (0-based j)
//   Abar = the mean over the nh heads of the attention probabilities attn[h][i][j]
//          (query i, key j; a causal map, so key j is seen by queries i >= j)
//
// colsum_kernel: one CTA per 32 key columns, 32 row lanes x 32 columns: lane r
//   adds rows i = j0 + r, j0 + r + 32, ... (i >= j) of every head in order, reading
//   128 contiguous bytes of a row per warp; the CTA adds its 32 row lanes in order,
//   so the result does not depend on scheduling.
// importance_kernel: one warp per token: the l1 norm of t_j, times the column mean
//   (the column sums are staged in the importance buffer itself).
// select_kernel: one CTA: radix select of the n-th largest importance (8 bits per
//   pass over the float bit patterns, which order like the values for
//   non-negative floats), then the mask: every token above that value and, among
//   the tokens equal to it, the lowest indices until n are chosen.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <algorithm>
#include <vector>

#include "mc_host.h"
#include "mc_kernels.h"

namespace mc {

constexpr int kColTile = 32;

__global__ void __launch_bounds__(1024) colsum_kernel(const float *attn, int L, int nh, float *colsum)
{
    __shared__ float part[32][kColTile + 1];
    pdl_trigger();
    pdl_wait();
    const int c = threadIdx.x & 31, r = threadIdx.x >> 5;
    const int j0 = blockIdx.x * kColTile, j = j0 + c;
    float acc = 0.f;
    if (j < L)
        for (int h = 0; h < nh; ++h) {
            const float *a = attn + (size_t)h * L * L;
            for (int i = j0 + r; i < L; i += 32)
                if (i >= j) acc += a[(size_t)i * L + j];
        }
    part[r][c] = acc;
    __syncthreads();
    if (r == 0 && j < L) {
        float s = 0.f;
        for (int q = 0; q < 32; ++q) s += part[q][c];
        colsum[j] = s;
    }
}

__global__ void __launch_bounds__(256) importance_kernel(const __nv_bfloat16 *t, int L, int H, int nh, float *imp)
{
    pdl_trigger();
    pdl_wait();
    const int lane = threadIdx.x & 31, j = blockIdx.x * 8 + (threadIdx.x >> 5);
    if (j >= L) return;
    const __nv_bfloat16 *row = t + (size_t)j * H;
    float l1 = 0.f;
    for (int h = lane; h < H; h += 32) l1 += fabsf(__bfloat162float(row[h]));
    for (int m = 16; m >= 1; m >>= 1) l1 += __shfl_xor_sync(0xffffffffu, l1, m);
    if (lane == 0) imp[j] = l1 * (imp[j] / ((float)nh * (float)(L - j)));
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

int mc_token_importance(const void *t, const float *attn, int L, int H, int nh, float protect_frac,
                        float *importance, uint8_t *mask, void *stream)
{
    clear_error();
    if (L < 0 || H <= 0 || nh <= 0 || !(protect_frac >= 0.f && protect_frac <= 1.f))
        return set_error(MC_ERR_INVALID_ARG, "L=%d H=%d nh=%d protect_frac=%g", L, H, nh, (double)protect_frac);
    if (L == 0) return MC_OK;
    if (!t || !attn || !importance) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    if ((double)nh * L * L > 9.0e18 / 4) return set_error(MC_ERR_INVALID_ARG, "attention map too large");
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t err = launch_k(colsum_kernel, dim3((L + kColTile - 1) / kColTile), dim3(1024), 0, st, attn, L, nh,
                               importance);
    if (err == cudaSuccess)
        err = launch_k(importance_kernel, dim3((L + 7) / 8), dim3(256), 0, st, (const __nv_bfloat16 *)t, L, H, nh,
                       importance);
    if (err == cudaSuccess && mask) {
        // ceil(frac * L); a product within 1e-6 of an integer counts as that integer
        const int n = (int)ceil((double)protect_frac * L - 1e-6);
        if (n <= 0 || n >= L)
            err = launch_k(fill_kernel, dim3((L + 255) / 256), dim3(256), 0, st, mask, L, (uint8_t)(n > 0));
        else
            err = launch_k(select_kernel, dim3(1), dim3(1024), 0, st, (const float *)importance, L, n, mask);
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
