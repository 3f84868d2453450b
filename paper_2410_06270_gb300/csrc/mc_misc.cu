// mc_misc.cu -- device unpacking of the packed expert layout (the codes the
// expert kernels decode, for bit-exact checks), RMSNorm and the residual add
// used between stacked layers.
#include "mc_host.h"
#include "mc_kernels.h"

namespace mc {

// One thread per (tile, lane): the exact inverse of mc_pack.cpp's packing.
__global__ void unpack_kernel(const uint8_t *packed, uint64_t mat_off, int mat, int rows, int cols, int bits,
                              int group, int E, int H, int F, int expert, uint8_t *codes, uint16_t *scale,
                              uint16_t *zero, int32_t *status)
{
    const PackHeader *hd = reinterpret_cast<const PackHeader *>(packed);
    if (hd->magic != kMagic || hd->version != kFormatVersion || hd->E != E || hd->H != H || hd->F != F ||
        hd->group != group || hd->bits[expert] != bits || hd->mat_off[expert][mat] != mat_off) {
        if (blockIdx.x == 0 && threadIdx.x == 0) set_status(status, MC_ERR_BAD_PACK);
        return;
    }
    const int KT = cols / kTileK, ng = cols / group, gpt = kTileK / group;
    const int ntiles = (rows / kTileRows) * KT;
    const int gid = blockIdx.x * blockDim.x + threadIdx.x;
    const int tile_id = gid >> 5, lane = gid & 31;
    if (tile_id >= ntiles) return;
    const int rb = tile_id / KT, kt = tile_id % KT;
    const uint8_t *tile = packed + mat_off + tile_off(mat, rb, kt, KT, rows / kBlockRows, bits, group);
    const int R0 = rb * kTileRows, K0 = kt * kTileK;
    uint32_t w[6] = {0, 0, 0, 0, 0, 0};
    for (int wi = 0; wi < 2 * bits; ++wi) w[wi] = *reinterpret_cast<const uint32_t *>(tile + code_word_off(bits, lane, wi));
    for (int j = 0; j < 32; ++j) {
        int row, col;
        pair_pos(lane, j, row, col);
        uint8_t *d = codes + (size_t)(R0 + row) * cols + K0 + col;
        for (int h = 0; h < 2; ++h) {
            uint32_t q = 0;
            for (int c = 0; c < bits; ++c) {
                int wi, bi;
                code_bit(bits, j, h, c, wi, bi);
                q |= ((w[wi] >> bi) & 1u) << c;
            }
            d[h] = (uint8_t)q;
        }
    }
    if (lane < 8 * gpt) {
        const int gi = lane >> 3, g8 = lane & 7;
        const uint16_t *m4 = reinterpret_cast<const uint16_t *>(tile + tile_code_bytes(bits)) + (gi * 8 + g8) * 4;
        const int gcol = (K0 + gi * group) / group;
        const size_t i0 = (size_t)(R0 + g8) * ng + gcol, i1 = (size_t)(R0 + g8 + 8) * ng + gcol;
        if (scale) { scale[i0] = m4[0]; scale[i1] = m4[2]; }
        if (zero) { zero[i0] = m4[1]; zero[i1] = m4[3]; }
    }
}

// One CTA of 256 threads per row; fp32 statistics.  For H % 8 == 0 the sum of
// squares takes the order of rmsnorm_vec_kernel (thread i over the 8-element
// chunks i, i + 256, ..., each chunk's elements in turn), so that the result does
// not depend on which of the two kernels the alignment of the arguments picks.
__global__ void __launch_bounds__(256) rmsnorm_kernel(const __nv_bfloat16 *x, const __nv_bfloat16 *gamma, int H,
                                                      float eps, __nv_bfloat16 *out)
{
    pdl_trigger();
    pdl_wait();
    const __nv_bfloat16 *xr = x + (size_t)blockIdx.x * H;
    __shared__ float red[8];
    float ss = 0.f;
    if (H % 8 == 0) {
        for (int c = threadIdx.x; c < H / 8; c += blockDim.x)
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float v = __bfloat162float(xr[8 * c + e]);
                ss = fmaf(v, v, ss);
            }
    } else {
        for (int c = threadIdx.x; c < H; c += blockDim.x) {
            const float v = __bfloat162float(xr[c]);
            ss = fmaf(v, v, ss);
        }
    }
    for (int m = 16; m >= 1; m >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, m);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) tot += red[w];
    const float inv = rsqrtf(tot / H + eps);
    __syncthreads();  // every thread has read x before any in-place write
    for (int c = threadIdx.x; c < H; c += blockDim.x)
        out[(size_t)blockIdx.x * H + c] =
            __float2bfloat16_rn(__bfloat162float(xr[c]) * inv * __bfloat162float(gamma[c]));
}

// The same with 16-byte accesses (H % 8 == 0, 16-byte aligned rows, H <= 16384):
// the row is loaded once into registers, every load issued before the first use,
// and normalised from there (an in-place call is safe: all loads precede the
// block barrier).
constexpr int kRmsPer = 8;  // 16-byte chunks per thread: 256 x 8 x 8 = 16384 columns
__global__ void __launch_bounds__(256) rmsnorm_vec_kernel(const __nv_bfloat16 *x, const __nv_bfloat16 *gamma,
                                                          int H, float eps, __nv_bfloat16 *out)
{
    pdl_trigger();
    pdl_wait();
    const int n8 = H >> 3;
    const uint4 *xr = reinterpret_cast<const uint4 *>(x + (size_t)blockIdx.x * H);
    const uint4 *g4 = reinterpret_cast<const uint4 *>(gamma);
    uint4 *orow = reinterpret_cast<uint4 *>(out + (size_t)blockIdx.x * H);
    __shared__ float red[8];
    uint4 v[kRmsPer];
#pragma unroll
    for (int i = 0; i < kRmsPer; ++i) {
        const int c = threadIdx.x + 256 * i;
        v[i] = c < n8 ? xr[c] : make_uint4(0, 0, 0, 0);
    }
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < kRmsPer; ++i) {
        const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&v[i]);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 f = __bfloat1622float2(b2[k]);
            ss = fmaf(f.x, f.x, ss);
            ss = fmaf(f.y, f.y, ss);
        }
    }
    for (int m = 16; m >= 1; m >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, m);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) tot += red[w];
    const float inv = rsqrtf(tot / H + eps);
#pragma unroll
    for (int i = 0; i < kRmsPer; ++i) {
        const int c = threadIdx.x + 256 * i;
        if (c >= n8) continue;
        const uint4 gv = g4[c];
        const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&v[i]);
        const __nv_bfloat162 *gg = reinterpret_cast<const __nv_bfloat162 *>(&gv);
        uint4 o;
        __nv_bfloat162 *o2 = reinterpret_cast<__nv_bfloat162 *>(&o);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 f = __bfloat1622float2(b2[k]), g = __bfloat1622float2(gg[k]);
            o2[k] = __floats2bfloat162_rn(f.x * inv * g.x, f.y * inv * g.y);
        }
        orow[c] = o;
    }
}

// out = a + b, eight bf16 per thread (n % 8 == 0, 16-byte aligned).
__global__ void add_vec_kernel(const uint4 *a, const uint4 *b, size_t n8, uint4 *out)
{
    pdl_trigger();
    pdl_wait();
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n8) return;
    const uint4 x = a[i], y = b[i];
    const __nv_bfloat162 *x2 = reinterpret_cast<const __nv_bfloat162 *>(&x);
    const __nv_bfloat162 *y2 = reinterpret_cast<const __nv_bfloat162 *>(&y);
    uint4 o;
    __nv_bfloat162 *o2 = reinterpret_cast<__nv_bfloat162 *>(&o);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 f = __bfloat1622float2(x2[k]), g = __bfloat1622float2(y2[k]);
        o2[k] = __floats2bfloat162_rn(f.x + g.x, f.y + g.y);
    }
    out[i] = o;
}

__global__ void add_kernel(const __nv_bfloat16 *a, const __nv_bfloat16 *b, size_t n, __nv_bfloat16 *out)
{
    pdl_trigger();
    pdl_wait();
    size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) out[i] = __float2bfloat16_rn(__bfloat162float(a[i]) + __bfloat162float(b[i]));
}

}  // namespace mc

using namespace mc;

extern "C" {

int mc_unpack_experts(const mc_shape *shape, const int8_t *bits_host, const void *packed_dev, int expert, int mat,
                      uint8_t *codes_dev, uint16_t *scale_dev, uint16_t *zero_dev, int32_t *status_dev, void *stream)
{
    clear_error();
    int rc = check_bits(shape, bits_host);
    if (rc) return rc;
    if (!packed_dev || !codes_dev) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    if (expert < 0 || expert >= shape->E || mat < 0 || mat > 2)
        return set_error(MC_ERR_INVALID_ARG, "expert %d / matrix %d out of range", expert, mat);
    if (bits_host[expert] == 16)
        return set_error(MC_ERR_UNSUPPORTED, "16-bit experts hold no codes (mc_unpack_experts_host reads them)");
    uint64_t off[kMaxE][3], total;
    layout_offsets(shape, bits_host, off, &total);
    const int rows = mat < 2 ? shape->F : shape->H, cols = mat < 2 ? shape->H : shape->F;
    const int ntiles = (rows / kTileRows) * (cols / kTileK);
    const long threads = (long)ntiles * 32;
    unpack_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, (cudaStream_t)stream>>>(
        (const uint8_t *)packed_dev, off[expert][mat], mat, rows, cols, bits_host[expert], shape->group, shape->E,
        shape->H, shape->F, expert, codes_dev, scale_dev, zero_dev, status_dev);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return set_error(MC_ERR_CUDA, "unpack launch: %s", cudaGetErrorString(e));
    return MC_OK;
}

int mc_rmsnorm(const void *x, const void *gamma, int T, int H, float eps, void *out, void *stream)
{
    clear_error();
    if (T < 0 || H <= 0 || !(eps >= 0.f)) return set_error(MC_ERR_INVALID_ARG, "bad T/H/eps");
    if (T == 0) return MC_OK;
    if (!x || !gamma || !out) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    const bool vec = H % 8 == 0 && H <= 256 * 8 * kRmsPer && aligned(x, 16) && aligned(gamma, 16) && aligned(out, 16);
    cudaError_t e = launch_k(vec ? rmsnorm_vec_kernel : rmsnorm_kernel, dim3(T), dim3(256), 0, (cudaStream_t)stream,
                             (const __nv_bfloat16 *)x, (const __nv_bfloat16 *)gamma, H, eps, (__nv_bfloat16 *)out);
    if (e != cudaSuccess) return set_error(MC_ERR_CUDA, "rmsnorm launch: %s", cudaGetErrorString(e));
    return MC_OK;
}

int mc_add(const void *a, const void *b, size_t n, void *out, void *stream)
{
    clear_error();
    if (n == 0) return MC_OK;
    if (!a || !b || !out) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    cudaError_t e;
    if (n % 8 == 0 && aligned(a, 16) && aligned(b, 16) && aligned(out, 16))
        e = launch_k(add_vec_kernel, dim3((unsigned)((n / 8 + 255) / 256)), dim3(256), 0, (cudaStream_t)stream,
                     (const uint4 *)a, (const uint4 *)b, n / 8, (uint4 *)out);
    else
        e = launch_k(add_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, (cudaStream_t)stream,
                     (const __nv_bfloat16 *)a, (const __nv_bfloat16 *)b, n, (__nv_bfloat16 *)out);
    if (e != cudaSuccess) return set_error(MC_ERR_CUDA, "add launch: %s", cudaGetErrorString(e));
    return MC_OK;
}

}  // extern "C"
