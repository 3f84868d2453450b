// mc_selftest.cu -- a one-CTA fp16 GEMM through the tcgen05 path (SW128 operands
// written by threads, one-thread MMA issue, commit to an mbarrier, TMEM loads).
// It checks the tensor-core building blocks of mc_umma.cuh against a plain
// matrix product and is exported for the test suite only.
#include "mc_host.h"
#include "mc_umma.cuh"

namespace mc {

__global__ void __launch_bounds__(128) selftest_umma_kernel(const __half *A, const __half *B, float *D, int N, int K,
                                                             int32_t *status, uint64_t timeout_ns)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int natoms = K / 64;
    uint8_t *sA = smem;                                   // natoms x 16 KB
    uint8_t *sB = smem + natoms * 16384;                  // natoms x N*128 B
    uint64_t *bar = reinterpret_cast<uint64_t *>(sB + natoms * N * 128);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + 1);
    const uint32_t ncols = N <= 32 ? 32 : (N <= 64 ? 64 : (N <= 128 ? 128 : 256));

    for (int idx = tid; idx < 128 * (K / 8); idx += blockDim.x) {
        const int r = idx / (K / 8), c8 = idx % (K / 8);
        const uint4 v = *reinterpret_cast<const uint4 *>(A + (size_t)r * K + c8 * 8);
        *reinterpret_cast<uint4 *>(sA + (c8 / 8) * 16384 + sw128_offset(r, (c8 % 8) * 8)) = v;
    }
    for (int idx = tid; idx < N * (K / 8); idx += blockDim.x) {
        const int r = idx / (K / 8), c8 = idx % (K / 8);
        const uint4 v = *reinterpret_cast<const uint4 *>(B + (size_t)r * K + c8 * 8);
        *reinterpret_cast<uint4 *>(sB + (c8 / 8) * (N * 128) + sw128_offset(r, (c8 % 8) * 8)) = v;
    }
    fence_proxy_async_smem();
    if (warp == 0) tmem_alloc(tslot, ncols);
    if (tid == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    if (tid == 0) {
        const uint32_t idesc = umma_idesc_f16(128, N);
        for (int s = 0; s < K / 16; ++s) {
            const int atom = s >> 2, sub = s & 3;
            const uint64_t ad = umma_desc_sw128(sA + atom * 16384 + sub * 32);
            const uint64_t bd = umma_desc_sw128(sB + atom * (N * 128) + sub * 32);
            umma_f16(tbase, ad, bd, idesc, s > 0);
        }
        umma_commit(bar);
    }
    const bool ok = mbar_wait(bar, 0, timeout_ns, status);
    tc_fence_after();
    if (ok) {
        for (int c0 = 0; c0 < N; c0 += 16) {
            float v[16];
            tmem_ld16(tbase + ((uint32_t)(32 * warp) << 16) + (uint32_t)c0, v);
            for (int i = 0; i < 16; ++i) D[(size_t)(32 * warp + lane) * N + c0 + i] = v[i];
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, ncols);
}

// Same product with A held in tensor memory: thread r of warps 0..3 writes row r
// (fp16 pairs, one 32-bit column per pair) with tcgen05.st, the MMA reads it.
__global__ void __launch_bounds__(128) selftest_umma_ts_kernel(const __half *A, const __half *B, float *D, int N,
                                                                int K, int32_t *status, uint64_t timeout_ns)
{
    extern __shared__ __align__(1024) uint8_t smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int natoms = K / 64;
    uint8_t *sB = smem;
    uint64_t *bar = reinterpret_cast<uint64_t *>(sB + natoms * N * 128);
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bar + 1);
    for (int idx = tid; idx < N * (K / 8); idx += blockDim.x) {
        const int r = idx / (K / 8), c8 = idx % (K / 8);
        const uint4 v = *reinterpret_cast<const uint4 *>(B + (size_t)r * K + c8 * 8);
        *reinterpret_cast<uint4 *>(sB + (c8 / 8) * (N * 128) + sw128_offset(r, (c8 % 8) * 8)) = v;
    }
    fence_proxy_async_smem();
    if (warp == 0) tmem_alloc(tslot, 512);
    if (tid == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const uint32_t acol = 256;  // A occupies columns [256, 256 + K/2)
    for (int a = 0; a < natoms; ++a) {
        uint32_t v[32];
        const uint32_t *src = reinterpret_cast<const uint32_t *>(A + (size_t)tid * K + a * 64);
        for (int i = 0; i < 32; ++i) v[i] = src[i];
        tmem_st32(tbase + ((uint32_t)(32 * warp) << 16) + acol + a * 32, v);
    }
    tmem_st_wait();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (tid == 0) {
        const uint32_t idesc = umma_idesc_f16(128, N);
        for (int s = 0; s < K / 16; ++s) {
            const uint64_t bd = umma_desc_sw128(sB + (s >> 2) * (N * 128) + (s & 3) * 32);
            umma_f16_ts(tbase, tbase + acol + s * 8, bd, idesc, s > 0);
        }
        umma_commit(bar);
    }
    const bool ok = mbar_wait(bar, 0, timeout_ns, status);
    tc_fence_after();
    if (ok) {
        for (int c0 = 0; c0 < N; c0 += 16) {
            float v[16];
            tmem_ld16(tbase + ((uint32_t)(32 * warp) << 16) + (uint32_t)c0, v);
            for (int i = 0; i < 16; ++i) D[(size_t)(32 * warp + lane) * N + c0 + i] = v[i];
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

}  // namespace mc

using namespace mc;

extern "C" int mc_selftest_umma(const void *A, const void *B, float *D, int N, int K, int32_t *status, void *stream)
{
    const bool a_in_tmem = N < 0;  // negative N: the A-in-tensor-memory variant
    if (a_in_tmem) N = -N;
    clear_error();
    if (!A || !B || !D) return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    if (N < 16 || N > 256 || N % 16 || K < 64 || K > 256 || K % 64)
        return set_error(MC_ERR_INVALID_ARG, "need 16 <= N <= 256 (multiple of 16), 64 <= K <= 256 (multiple of 64)");
    if (a_in_tmem && N > 128) return set_error(MC_ERR_INVALID_ARG, "A-in-TMEM variant: N <= 128");
    const size_t sm = (size_t)(K / 64) * ((a_in_tmem ? 0 : 16384) + N * 128) + 64;
    if (sm > 200 * 1024) return set_error(MC_ERR_INVALID_ARG, "tile too large");
    cudaError_t err = cudaFuncSetAttribute(a_in_tmem ? selftest_umma_ts_kernel : selftest_umma_kernel,
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(err));
    if (a_in_tmem)
        selftest_umma_ts_kernel<<<1, 128, sm, (cudaStream_t)stream>>>((const __half *)A, (const __half *)B, D, N, K,
                                                                      status, 1000000000ull);
    else
        selftest_umma_kernel<<<1, 128, sm, (cudaStream_t)stream>>>((const __half *)A, (const __half *)B, D, N, K,
                                                                   status, 1000000000ull);
    err = cudaGetLastError();
    if (err != cudaSuccess) return set_error(MC_ERR_CUDA, "launch: %s", cudaGetErrorString(err));
    return MC_OK;
}
