/*
 * mc.h -- C ABI of the GB300 (sm_103a) library for the compressed MoE layer of
 * "MC: Mixture Compressor for MoE LLMs" (Huang et al., ICLR 2025).
 *
 * The layer (Sec. 2.1 Eq. 1, Sec. 2.3 Eq. 5/6):
 *   logits  = x Wg^T                                  (gate G of Eq. 1)
 *   (e0,e1) = top-2 experts, w = renormalised softmax  (Eq. 1)
 *   pruned  = !protect && w1/w0 < mu  -> w = (1, 0)    (Eq. 5, Sec. 2.3.2)
 *   dropped = mask byte 2              -> w = (0, 0)    (Sec. 3.2, Fig. 9)
 *   y       = sum over kept slots of w * E_e(x)        (Eq. 1)
 *   E(x)    = W2 (silu(W1 x) * W3 x)                   (Mixtral SwiGLU expert)
 * with every expert's W1, W3, W2 quantised weight-only to that expert's bit width
 * b in {1,2,3} (PMQ, Sec. 2.2), group-wise along the input dimension, asymmetric:
 *   w = (q - z) * s,  q in [0, 2^b - 1], one fp16 s and one fp16 z per group
 * (Sec. 2.1, Eq. 2's integer grid; 1-bit codes are App. A.2's (sign(W)+1)/2 with
 * z = 1/2, s = 2*alpha).
 *
 * Conventions for every entry point:
 *   - Pointers are DEVICE pointers unless the parameter name ends in _host.
 *   - The caller allocates every buffer; no entry point allocates device memory
 *     except mc_pack_experts, which uses a temporary pinned host staging buffer.
 *   - Device work is enqueued on `stream` (a cudaStream_t passed as void*; NULL is
 *     the legacy default stream) and is asynchronous unless stated otherwise.
 *   - Return value: MC_OK (0) or a negative MC_ERR_* code; mc_last_error() gives a
 *     thread-local message for the last failing call on the calling thread.
 *   - Bad arguments are rejected on the host before anything is enqueued.
 *   - Device-detected faults (a packed buffer whose header does not match the
 *     shape, activations outside the fp16 range, a bounded wait that expired) do
 *     not abort: the kernels record a code in the status word at the start of the
 *     workspace and skip their work; mc_check_status() reads it.
 * Shapes supported by this version: E <= 16, top_k == 2, group in {64, 128},
 * H and F multiples of 128, H <= 16384, F <= 65536.
 */
#ifndef MC_H_
#define MC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    MC_OK = 0,
    MC_ERR_INVALID_ARG = -1, /* null/misaligned pointer, bad shape, bad mu, ... */
    MC_ERR_UNSUPPORTED = -2, /* a bit width outside {1,2,3,16}, E > 16, ... */
    MC_ERR_CUDA = -3,        /* a CUDA runtime call failed (message has the text) */
    MC_ERR_TIMEOUT = -4,     /* a bounded device wait expired (status word) */
    MC_ERR_BAD_PACK = -5,    /* packed buffer header does not match (magic/shape/bits) */
    MC_ERR_RANGE = -6        /* an activation (x, or the SwiGLU product h that feeds W2) was
                                non-finite or outside the fp16 range */
};

/* Layer shape.  E experts, hidden size H, SwiGLU width F, quantisation group
 * size `group` (weights per scale/zero along the input dimension), top_k = 2. */
typedef struct {
    int32_t E, H, F, group, top_k;
} mc_shape;

/* Thread-local text of the last error on this thread ("" if none). */
const char *mc_last_error(void);

/* Library version (major*10000 + minor*100 + patch) and packed-format version. */
int mc_version(void);
int mc_pack_format_version(void);

/* ------------------------------------------------------------------------ *
 * Packed expert weights (PMQ storage, Sec. 2.2 / App. A.2).
 *
 * Canonical input, per expert e and matrix m (0 = W1 [F,H], 1 = W3 [F,H],
 * 2 = W2 [H,F], row-major, groups of `group` consecutive columns):
 *   codes  uint8 [rows*cols], one code per byte, value < 2^bits[e]
 *   scale  fp16 bit patterns [rows, cols/group]
 *   zero   fp16 bit patterns [rows, cols/group]
 * bits[e] = 16 (the unquantised fp16 baseline; all experts of a layer or none):
 * codes is the matrix itself as fp16 bit patterns (uint16 [rows*cols], passed
 * through the uint8 pointer) and scale / zero are unused (may be NULL).
 * The packed layout is private to this library and versioned by a header at the
 * start of the buffer; only its total size is part of the ABI.
 * ------------------------------------------------------------------------ */

/* Bytes needed for the packed buffer of this shape and bit table (host int8[E]),
 * or 0 if the shape or a bit width is invalid (mc_last_error says which). */
size_t mc_packed_size(const mc_shape *shape, const int8_t *bits_host);

/* Pack canonical host arrays into a HOST buffer of mc_packed_size() bytes.  The
 * arrays are indexed [3*e + m].  Pure host code (no GPU needed).  Returns
 * MC_ERR_INVALID_ARG for a code >= 2^bits, a null array or a short buffer;
 * MC_ERR_UNSUPPORTED for a bit width outside {1,2,3,16} or 16-bit experts mixed
 * with quantised ones. */
int mc_pack_experts_host(const mc_shape *shape, const int8_t *bits_host,
                         const uint8_t *const *codes_host,
                         const uint16_t *const *scale_host,
                         const uint16_t *const *zero_host,
                         void *packed_host, size_t packed_bytes);

/* mc_pack_experts_host into a pinned staging buffer, then a copy to packed_dev
 * on `stream`.  SYNCHRONOUS: returns after the copy has completed. */
int mc_pack_experts(const mc_shape *shape, const int8_t *bits_host,
                    const uint8_t *const *codes_host,
                    const uint16_t *const *scale_host,
                    const uint16_t *const *zero_host,
                    void *packed_dev, size_t packed_bytes, void *stream);

/* Inverse of the packing for one (expert, matrix), from a HOST packed buffer:
 * writes canonical codes [rows*cols] and fp16 scale/zero [rows, cols/group]
 * (scale_host / zero_host may be NULL); a 16-bit expert's fp16 weights go to
 * codes_host as uint16 [rows*cols].  Pure host code.  MC_ERR_BAD_PACK if the
 * header is not a valid packed buffer. */
int mc_unpack_experts_host(const void *packed_host, size_t packed_bytes, int expert, int mat,
                           uint8_t *codes_host, uint16_t *scale_host, uint16_t *zero_host);

/* The same inverse run by a device kernel on a DEVICE packed buffer (the codes
 * the GPU kernels actually decode), writing device arrays.  Asynchronous.
 * `shape` and `bits_host` describe the buffer; the kernel also checks the header
 * and records MC_ERR_BAD_PACK in *status_dev (a device int32, may be NULL). */
int mc_unpack_experts(const mc_shape *shape, const int8_t *bits_host,
                      const void *packed_dev, int expert, int mat,
                      uint8_t *codes_dev, uint16_t *scale_dev, uint16_t *zero_dev,
                      int32_t *status_dev, void *stream);

/* Read and check the header of a DEVICE packed buffer against shape/bits.
 * SYNCHRONOUS.  MC_OK or MC_ERR_BAD_PACK. */
int mc_pack_verify(const mc_shape *shape, const int8_t *bits_host, const void *packed_dev,
                   size_t packed_bytes);

/* ------------------------------------------------------------------------ *
 * Routing: Eq. 1 gate + top-2 + renormalised softmax, Eq. 5 ODP, Sec. 2.3.2
 * protection, the Sec. 3.2 (Fig. 9) token drop, then the permutation of kept
 * (token, slot) pairs by expert.
 *   x       bf16 [T, H]        gate_w  bf16 [E, H]
 *   mu      Eq. 5 threshold (finite, >= 0; 0 disables pruning; > 1 prunes every
 *           unprotected token)
 *   protect uint8 [T] token mask, may be NULL (all 0): 0 = prunable by Eq. 5,
 *           2 = dropped (all of the token's experts masked: no pair, output 0),
 *           any other value = protected (never pruned)
 * Outputs (device):
 *   topk_idx int32 [T, 2]  slot 0 = primary (larger weight), ties -> lower index
 *   topk_w   fp32  [T, 2]  renormalised weights; (1, 0) for a pruned token,
 *                          (0, 0) for a dropped one
 *   pruned   uint8 [T]     0 kept, 1 secondary pruned, 2 token dropped
 *   expert_offsets int32 [E+1]  exclusive prefix counts of kept pairs
 *   perm     int32 [2T]   first expert_offsets[E] entries valid: 2*token + slot,
 *                          grouped by expert, ascending token within an expert
 * The decision is taken on fp32 logits; the ODP test is evaluated as
 * (l0 - l1) > -ln(mu), which equals w1/w0 < mu.
 * ------------------------------------------------------------------------ */
int mc_route(const void *x, const void *gate_w, int T, const mc_shape *shape, float mu,
             const uint8_t *protect, int32_t *topk_idx, float *topk_w, uint8_t *pruned,
             int32_t *expert_offsets, int32_t *perm, void *stream);

/* ------------------------------------------------------------------------ *
 * The whole layer (Eq. 1 with Eq. 5 on PMQ experts).
 *   x bf16 [T, H] (values must be finite and |x| <= 65504; the SwiGLU product
 *   h = silu(W1 x) * (W3 x) that feeds W2 must be too, else the status word
 *   reports MC_ERR_RANGE), gate_w bf16 [E, H],
 *   packed_dev: the buffer written by mc_pack_experts for (shape, bits_host),
 *   mu, protect as in mc_route, y bf16 [T, H] output.
 *   workspace: device scratch of mc_moe_workspace_size(shape, T_max) bytes for
 *   some T_max >= T (one workspace serves every T up to the one it was sized
 *   for), 256-byte aligned, ZEROED before its first use (every call leaves the
 *   parts that need it at zero again; they sit at offsets that do not depend on
 *   T); its first 4 bytes are the status word (see mc_check_status).
 *   topk_idx_out int32 [T,2], topk_w_out fp32 [T,2], pruned_out uint8 [T]: optional
 *   copies of the routing decisions (NULL to skip).
 * Never synchronises and never allocates; capturable in a CUDA graph.
 * T == 0 is a no-op returning MC_OK.
 * ------------------------------------------------------------------------ */
size_t mc_moe_workspace_size(const mc_shape *shape, int T_max);

int mc_moe_forward(const void *x, const void *gate_w, int T, const mc_shape *shape,
                   const int8_t *bits_host, const void *packed_dev, float mu,
                   const uint8_t *protect, void *y, void *workspace, size_t ws_bytes,
                   int32_t *topk_idx_out, float *topk_w_out, uint8_t *pruned_out,
                   void *stream);

/* mc_moe_forward without a workspace: the same layer (routing, ODP, experts on
 * the mma.sync path, combine), with its scratch in a fixed 16 MiB device array
 * that belongs to the library (one per device).  The paper has no counterpart;
 * this entry point exists for callers that must not allocate device memory once
 * they are running: a serving loop that freezes its memory plan at start-up, a
 * plug-in whose device memory belongs to a host framework, a plain C caller
 * with no device allocator of its own.  It allocates nothing.
 *   Arguments as mc_moe_forward; no workspace and no routing outputs.
 *   status_dev: optional device int32; when given, device-side errors
 *     (MC_ERR_TIMEOUT, MC_ERR_BAD_PACK, MC_ERR_RANGE) are recorded there and it
 *     must hold 0 when the call starts.  When NULL, they go to a status word in
 *     the scratch, which each call clears (cudaMemsetAsync on `stream`) before
 *     its kernels and which the caller cannot read.  No other byte of the
 *     scratch needs an initial value.
 *   Limit: the scratch must hold the call's buffers; a (shape, T) that needs
 *     more than 16 MiB returns MC_ERR_INVALID_ARG with the size in the message
 *     (at the Mixtral-8x7b shape, H 4096, F 14336, group 128, that is T > 96).
 *     The W2 pass takes mc_moe_forward's column splits when their partial
 *     outputs fit in the scratch, else a single split (same results).
 *   Set-up: the first call on a device, made with that device current, looks up
 *     the scratch's address once (cudaGetSymbolAddress) and keeps it for the
 *     life of the process; make that first call before any stream capture, and
 *     do not call it on a device after cudaDeviceReset (a reset reloads the
 *     library's device code, and the scratch may then sit elsewhere).
 *   The mc_set_debug hooks (flags, wait bound) apply as for mc_moe_forward.
 *   Concurrency: every call on a device uses the same scratch, so calls whose
 *     kernels may overlap (other streams, other host threads) race and corrupt
 *     each other's results; order them (one stream, or events). */
int mc_moe_forward_static(const void *x, const void *gate_w, int T, const mc_shape *shape,
                          const int8_t *bits_host, const void *packed_dev, float mu,
                          const uint8_t *protect, void *y, int32_t *status_dev, void *stream);

/* Workspace bytes of mc_stack_forward for up to T_max tokens: the layer
 * workspace (status word first) followed by two [T_max, H] bf16 activations (the
 * normalised layer input; the layer output when h is not 16-byte aligned). */
size_t mc_stack_workspace_size(const mc_shape *shape, int T_max);

/* A stack of `layers` pre-norm residual MoE blocks, the structure of the
 * Mixtral models the paper compresses (Sec. 3.1 model table: 32 MoE layers):
 *   for l in 0 .. layers-1:  h <- h + MoE_l(RMSNorm_l(h))
 * MoE_l is mc_moe_forward with gate_w[l] (device bf16 [E, H]), packed_dev[l],
 * the bit table bits_host[l*E .. l*E+E-1] and threshold mu_host[l]; RMSNorm_l
 * uses gamma + l*H (device bf16 [layers, H]) and eps.  h (device bf16 [T, H]) is
 * updated in place; every intermediate is bf16.  With 16-byte aligned h and
 * gamma each layer's RMSNorm runs inside its routing launch and its residual add
 * inside its combine, with the arithmetic and rounding of mc_rmsnorm and mc_add
 * (the result is bit for bit that of mc_rmsnorm, mc_moe_forward and mc_add in
 * turn, which is what runs for an h of any other alignment).  protect (device
 * [T] or NULL)
 * applies to every layer.  Device-detected faults of any layer go to the status
 * word at the start of `workspace` (mc_check_status).  All launches go to
 * `stream` and none synchronises, so a caller may capture one call into a CUDA
 * graph (after a first call has set the kernels' shared-memory attributes). */
int mc_stack_forward(void *h, int T, const mc_shape *shape, int layers, const void *const *gate_w,
                     const int8_t *bits_host, const void *const *packed_dev, const float *mu_host,
                     const uint8_t *protect, const void *gamma, float eps, void *workspace,
                     size_t ws_bytes, void *stream);

/* ------------------------------------------------------------------------ *
 * Token importance (Sec. 2.3.2, Eq. 6) and the protect mask of ODP.
 *   t      bf16 [L, H]      the tokens entering the MoE block (the l1 norm of Eq. 6)
 *   attn   fp32 [nh, L, L]  the block's attention probabilities, attn[h][i][j] =
 *                           weight of query i on key j (causal: used for i >= j;
 *                           entries must be finite and >= 0)
 *   importance fp32 [L] out: I_j = ||t_j||_1 * (1/(L - j)) * sum_{i=j}^{L-1} Abar[i][j]
 *                           (0-based j), Abar the mean over the heads: the mean
 *                           attention key j receives from the queries that see it
 *   protect_frac in [0, 1]: mask (uint8 [L] out, may be NULL) gets 1 for the
 *                           ceil(protect_frac * L) tokens of largest importance
 *                           (a product within 1e-6 of an integer counts as it)
 *                           (ties to the lower index), 0 for the others -- the
 *                           protect input of mc_route / mc_moe_forward.
 *   workspace: device scratch of at least mc_token_importance_workspace_size(L)
 *           bytes, 8-byte aligned (no initial contents needed).
 * Deterministic: the column sums are accumulated in 2^-40 fixed point with
 * integer atomics; asynchronous on `stream`.
 * ------------------------------------------------------------------------ */
size_t mc_token_importance_workspace_size(int L);
int mc_token_importance(const void *t, const float *attn, int L, int H, int nh, float protect_frac,
                        float *importance, uint8_t *mask, void *workspace, size_t ws_bytes, void *stream);

/* The Eq. 5 threshold from calibration routing weights (Sec. 2.3.1: the median
 * of w1/w0 over calibration data is q = 0.5): the q-quantile, linear between
 * order statistics, of w1/w0 over the tokens whose mask byte is 0 (mask_host
 * may be NULL) and whose primary weight is positive.  Host arrays: w_host
 * fp32 [T, 2] as written by mc_route.  MC_ERR_INVALID_ARG when no token qualifies. */
int mc_odp_threshold_host(const float *w_host, const uint8_t *mask_host, int T, double q, float *mu_out);

/* ------------------------------------------------------------------------ *
 * PMQ bit allocation (Sec. 2.2), host code run once per layer before
 * quantisation.
 * Expert significance from a calibration run's routing (Sec. 2.2.1): host arrays
 * idx int32 [T, 2], w fp32 [T, 2], pruned uint8 [T] (may be NULL) as written by
 * mc_route; phi[e] = n_e / N (activations of expert e per calibration token) and
 * wact[e] = (sum of its routing weights) / N, N = T; a pruned secondary or a
 * dropped token is not an activation.
 * ------------------------------------------------------------------------ */
int mc_expert_significance_host(const int32_t *idx, const float *w, const uint8_t *pruned, int T, int E,
                                double *phi, double *wact);

/* Eq. 4, solved exactly over all 3^E assignments: bits_out[i] in {1, 2, 3}
 * minimising sum_i phi_i^alpha * wact_i^beta * eps[i][bits_i - 1]^gamma subject
 * to sum_i bits_i = bits_total (n * k of Eq. 4), at least one 3-bit and one 2-bit
 * expert.  eps [E][3]: the F-norm of the layer output error with only expert i
 * quantised to 1, 2, 3 bits (Sec. 2.2.2), measured by the caller.  Ties go to
 * the assignment met first when expert 0's width varies fastest.  E <= 16;
 * MC_ERR_INVALID_ARG for an infeasible budget or a negative / non-finite input.
 * objective_out (may be NULL) receives the minimum. */
int mc_pmq_allocate(const double *phi, const double *wact, const double *eps, int E, int bits_total, double alpha,
                    double beta, double gamma, int8_t *bits_out, double *objective_out);

/* Test hook: choose the expert path of mc_moe_forward: 0 = automatic (the GEMV
 * below 240 kept-or-not pairs, 2T < 240, else the GEMM), 1 = the mma.sync
 * grouped GEMV with work chunks of 16 pairs (decode), 2 = the tcgen05 grouped
 * GEMM with token blocks of 128 pairs (prefill).  Both paths compute the same
 * layer; forcing one lets tests run both kernels at the same sizes.
 * Process-wide (an atomic word read once per mc_moe_forward call); returns the
 * previous value, or MC_ERR_INVALID_ARG (and no change) for another value. */
int mc_set_path(int path);

/* Test hook: `flags` bit 0 makes the expert kernels' weight producer issue no
 * copies, so every consumer wait reaches its bound and the status word reports
 * MC_ERR_TIMEOUT (no fault, no hang); bit 1 launches every kernel without
 * programmatic dependent launch (by default each kernel's launch overlaps the
 * end of the one before it on the stream; results are the same either way); bit
 * 2 makes mc_route take the single-launch routing mc_moe_forward uses for
 * T <= 64 (the last routing CTA places the pairs), with its arrival count in a
 * word owned by the library, so that tests can compare that placement with the
 * two-launch one (calls with the bit set must not overlap in time on a device).
 * `timeout_ns` (0 = keep) bounds every device wait (default 1 s).
 * Process-wide. */
int mc_set_debug(int flags, unsigned long long timeout_ns);

/* Self-test of the tensor-core (tcgen05) building blocks used by the expert
 * kernels: D = A * B^T for one 128-row tile, A fp16 [128, K], B fp16 [N, K]
 * (row-major, 16-byte aligned), D fp32 [128, N]; 16 <= N <= 256 (multiple of 16),
 * 64 <= K <= 256 (multiple of 64).  A negative N selects the variant with A held
 * in tensor memory (|N| <= 128).  A bounded wait records MC_ERR_TIMEOUT in
 * *status (device int32, may be NULL).  For the test suite; not on the layer path. */
int mc_selftest_umma(const void *A, const void *B, float *D, int N, int K, int32_t *status, void *stream);

/* Synchronise `stream`, read the status word at the start of `workspace`, clear
 * it, and return MC_OK or the recorded MC_ERR_* code. */
int mc_check_status(void *workspace, void *stream);

/* Per-kernel timing of this library's own launches with CUDA events recorded on
 * the launching stream (for benchmarks; off by default).  mc_profile_read
 * synchronises on the recorded events, writes the summed milliseconds and launch
 * counts of kernel ids 0 .. n-1 (names from mc_profile_name: route, permute,
 * gemv_w13, gemv_w2, combine, frag_x, gemm_w13, gemm_w2, rmsnorm, importance,
 * x_img) and
 * clears the records.  Inside stream capture the events become event nodes of
 * the graph: every replay records them again, and each mc_profile_read reports
 * the latest replay and keeps those records until mc_profile_clear. */
int mc_profile_enable(int on);
/* Bit mask of the kernel ids recorded while profiling is on (default: all), so
 * that a benchmark can time one kernel with two events per launch and leave the
 * others unperturbed.  Returns the previous mask. */
unsigned mc_profile_select(unsigned mask);
int mc_profile_read(double *ms_out, int *count_out, int n);
/* Drops every record, including those kept for captured graphs. */
int mc_profile_clear(void);
const char *mc_profile_name(int id);

/* RMSNorm used between stacked layers: out = x / sqrt(mean(x^2) + eps) * gamma,
 * x and out bf16 [T, H] (may alias), gamma bf16 [H]. */
int mc_rmsnorm(const void *x, const void *gamma, int T, int H, float eps, void *out,
               void *stream);

/* out = a + b elementwise over n bf16 values (residual add; may alias a). */
int mc_add(const void *a, const void *b, size_t n, void *out, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* MC_H_ */
