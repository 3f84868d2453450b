// mc_device.cuh -- device helpers shared by the kernels: the status word,
// mbarrier / bulk-copy wrappers with bounded waits, mma.sync, small conversions.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include "../../include/mc.h"
#include "mc_layout.h"

namespace mc {

// Record the first error code in the status word (device int32, 0 = OK).
__device__ __forceinline__ void set_status(int32_t *status, int code)
{
    if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ uint64_t globaltimer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Programmatic dependent launch.  pdl_trigger: the next kernel on the stream may
// be launched now (it is, once every CTA of this grid has triggered or exited).
// pdl_wait: returns once the kernel before this one on the stream has completed
// and its memory operations are visible; a no-op for a kernel launched without
// programmatic serialisation.  Every kernel of the library calls pdl_wait before
// its first global memory access.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

// ---------------------------------------------------------------- mbarrier --

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar)
{
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(smem_u32(bar))
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.expect_tx.shared::cta.b64 st, [%0], %1;\n\t}" ::"r"(
                     smem_u32(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// Same test, but a thread whose phase is not yet complete may be suspended for
// up to `hint_ns` (it resumes as soon as the phase completes), so that waiting
// warps do not take issue slots from working ones.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t *bar, uint32_t parity, uint32_t hint_ns)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\tselp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
        : "memory");
    return ok != 0;
}

constexpr uint32_t kWaitHintNs = 20000;  // re-check timeouts / abort flags every 20 us at most

// Wait for phase `parity` of `bar` to complete, for at most timeout_ns
// nanoseconds.  Returns false (and records MC_ERR_TIMEOUT) if it expired.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, uint64_t timeout_ns, int32_t *status)
{
    if (mbar_try_wait(bar, parity)) return true;
    uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait_sleep(bar, parity, kWaitHintNs)) return true;
        if (globaltimer_ns() - t0 > timeout_ns) {
            set_status(status, MC_ERR_TIMEOUT);
            return false;
        }
    }
}

// 1-D bulk copy global -> shared, completion counted on `bar` (tx bytes).
// Both addresses 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void *dst_smem, const void *src_gmem, uint32_t bytes, uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst_smem)),
        "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

// Same, with an L2 evict-first policy for data read exactly once (weights).
__device__ __forceinline__ void bulk_g2s_stream(void *dst_smem, const void *src_gmem, uint32_t bytes,
                                                uint64_t *bar, uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
        "%4;" ::"r"(smem_u32(dst_smem)),
        "l"(src_gmem), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
        : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_first()
{
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

// --------------------------------------------------------------------- mma --

// D += A * B, m16n8k16, fp16 inputs, fp32 accumulate.
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// ------------------------------------------------------- code -> fp16 pairs --
// (w & field_mask) | exponent constant: an fp16 pair reading (2^E + q) with
// E = 10 - (mantissa bit of the field) (see mc_layout.h).

__device__ __forceinline__ uint32_t lop_and_or(uint32_t w, uint32_t mask, uint32_t c)
{
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(w), "r"(mask), "r"(c));
    return r;
}

// fp16 exponent constants, both halves.
#define MC_C(e) (((uint32_t)(e) << 10) * 0x00010001u)

// 2-bit code word -> 8 registers (positions 0..7)
__device__ __forceinline__ void cvt2(uint32_t w, uint32_t (&r)[8])
{
    r[0] = lop_and_or(w, 0x00030003u, MC_C(25));
    r[1] = lop_and_or(w, 0x000C000Cu, MC_C(23));
    r[2] = lop_and_or(w, 0x00300030u, MC_C(21));
    r[3] = lop_and_or(w, 0x00C000C0u, MC_C(19));
    r[4] = lop_and_or(w, 0x03000300u, MC_C(17));
    uint32_t v = w >> 10;
    r[5] = lop_and_or(v, 0x00030003u, MC_C(25));
    r[6] = lop_and_or(v, 0x000C000Cu, MC_C(23));
    r[7] = lop_and_or(v, 0x00300030u, MC_C(21));
}

// 1-bit code word, positions [p0, p0+8) -> 8 registers (p0 = 0 or 8).
__device__ __forceinline__ void cvt1_half(uint32_t w, int p0, uint32_t (&r)[8])
{
    const uint32_t v = w >> 10;
    if (p0 == 0) {
#pragma unroll
        for (int p = 0; p < 8; ++p) r[p] = lop_and_or(w, 0x00010001u << p, MC_C(25 - p));
    } else {
        r[0] = lop_and_or(w, 0x00010001u << 8, MC_C(17));
        r[1] = lop_and_or(w, 0x00010001u << 9, MC_C(16));
#pragma unroll
        for (int p = 0; p < 6; ++p) r[2 + p] = lop_and_or(v, 0x00010001u << p, MC_C(25 - p));
    }
}

// (x & m) | (y & ~m)
__device__ __forceinline__ uint32_t lop_sel(uint32_t x, uint32_t y, uint32_t m)
{
    uint32_t r;
    asm("lop3.b32 %0, %1, %2, %3, 0xE4;" : "=r"(r) : "r"(x), "r"(y), "r"(m));
    return r;
}

// 3-bit code words (6 per lane) -> the 8 registers of pairs 8qd .. 8qd+7.
// Pairs j < 30 take one LOP3 each (fields at mantissa bits 1, 4, 7 directly,
// fields at bits 10, 13 after a shift by 10); pairs 30 and 31 gather their
// three bits from bit 0 / 16 of three words.
__device__ __forceinline__ uint32_t cvt3_pair(const uint32_t (&w)[6], int j)
{
    if (j < 30) {
        const int i = j / 5, p = j % 5;
        if (p < 3) return lop_and_or(w[i], 0x00070007u << (1 + 3 * p), MC_C(24 - 3 * p));
        return lop_and_or(w[i] >> 10, 0x00070007u << (3 * (p - 3)), MC_C(25 - 3 * (p - 3)));
    }
    const int b = 3 * (j - 30);
    const uint32_t t = lop_sel(w[b], w[b + 1] << 1, 0x00010001u);
    return lop_and_or(lop_sel(t, w[b + 2] << 2, 0x00030003u), 0x00070007u, MC_C(25));
}

__device__ __forceinline__ void cvt3(const uint32_t (&w)[6], int qd, uint32_t (&r)[8])
{
#pragma unroll
    for (int i = 0; i < 8; ++i) r[i] = cvt3_pair(w, 8 * qd + i);
}

// silu(g) = g / (1 + e^-g); the fast reciprocal-based division returns 0 once
// e^-g overflows, which is the function's limit there.
__device__ __forceinline__ float silu(float g) { return __fdividef(g, 1.0f + __expf(-g)); }

}  // namespace mc
