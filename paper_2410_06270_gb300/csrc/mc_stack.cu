// mc_stack.cu -- mc_stack_forward: a stack of pre-norm residual MoE layers,
// h <- h + MoE_l(RMSNorm_l(h)) for l = 0 .. layers-1, each layer the compressed
// block of mc_moe_forward with its own gate, packed experts, bit table and ODP
// threshold.  Every step is a launch of this library on one stream, so the whole
// stack can be captured into one CUDA graph by the caller.
#include <string.h>

#include "mc_host.h"
#include "mc_kernels.h"

using namespace mc;

static inline size_t align256(size_t x) { return (x + 255) & ~(size_t)255; }

extern "C" size_t mc_stack_workspace_size(const mc_shape *shape, int T_max)
{
    const size_t ws = mc_moe_workspace_size(shape, T_max);
    if (!ws) return 0;
    return align256(ws) + 2 * align256((size_t)T_max * shape->H * 2);
}

extern "C" int mc_stack_forward(void *h, int T, const mc_shape *shape, int layers, const void *const *gate_w,
                                const int8_t *bits_host, const void *const *packed_dev, const float *mu_host,
                                const uint8_t *protect, const void *gamma, float eps, void *workspace,
                                size_t ws_bytes, void *stream)
{
    clear_error();
    if (layers < 0 || T < 0) return set_error(MC_ERR_INVALID_ARG, "layers=%d, T=%d", layers, T);
    if (layers == 0 || T == 0) return MC_OK;
    if (!h || !gate_w || !bits_host || !packed_dev || !mu_host || !gamma || !workspace)
        return set_error(MC_ERR_INVALID_ARG, "NULL pointer argument");
    int rc = check_shape(shape);
    if (rc) return rc;
    const size_t need = mc_stack_workspace_size(shape, T);
    if (ws_bytes < need) return set_error(MC_ERR_INVALID_ARG, "workspace has %zu bytes, needs %zu", ws_bytes, need);
    const size_t fw = align256(mc_moe_workspace_size(shape, T));
    const size_t act = align256((size_t)T * shape->H * 2);
    void *xn = (uint8_t *)workspace + fw, *y = (uint8_t *)workspace + fw + act;
    // With 16-byte aligned rows the layer's routing launch computes its RMSNorm (bit
    // for bit mc_rmsnorm) into xn and routes on it, and its combine adds the layer
    // output to h in place (rounded like mc_add of the layer's bf16 output).  An
    // unaligned h takes mc_rmsnorm, the layer into y and mc_add: the same result.
    const bool h_aligned = (uintptr_t)h % 16 == 0;
    const bool fused_norm = h_aligned && ((uintptr_t)gamma % 16 == 0) && shape->H % 8 == 0;
    for (int l = 0; l < layers; ++l) {
        const void *g = (const uint8_t *)gamma + (size_t)l * shape->H * 2;
        const int8_t *bl = bits_host + (size_t)l * shape->E;
        if (!fused_norm && (rc = mc_rmsnorm(h, g, T, shape->H, eps, xn, stream))) return rc;
        if (h_aligned) {
            LayerPrePost lpp{fused_norm ? h : nullptr, g, eps, h};
            rc = moe_forward_ex(xn, gate_w[l], T, shape, bl, packed_dev[l], mu_host[l], protect, h, &lpp, workspace,
                                fw, nullptr, nullptr, nullptr, stream);
        } else {
            rc = mc_moe_forward(xn, gate_w[l], T, shape, bl, packed_dev[l], mu_host[l], protect, y, workspace, fw,
                                nullptr, nullptr, nullptr, stream);
            if (!rc) rc = mc_add(h, y, (size_t)T * shape->H, h, stream);
        }
        if (rc) return rc;
    }
    return MC_OK;
}
