/*
 * mc_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously-correct CPU statement of the compressed MoE layer of
 * "MC: Mixture Compressor for MoE LLMs" (ICLR 2025):
 *   - the top-2 gate of Sec. 2.1, Eq. 1,
 *   - the group-wise asymmetric weight dequantisation of Sec. 2.1 (Eq. 2's
 *     integer grid) and the 1-bit storage transform of Appendix A.2,
 *   - Online Dynamic Pruning, Sec. 2.3.1, Eq. 5, with the significant-token
 *     protection of Sec. 2.3.2 and the less-significant-token drop of Sec. 3.2
 *     (Fig. 9),
 *   - the SwiGLU expert feed-forward of Mixtral (the E_i of Eq. 1),
 *   - the weighted combine of Eq. 1.
 *
 * Everything is computed from its definition: one weight at a time, fp64
 * accumulation, no blocking, no group factoring, no reordering.  Only the test
 * suite, the smoke check and the CPU-baseline leg of the benchmark may load this
 * file; the product path never does.  It shares no code with the CUDA library.
 *
 * Readings of the paper taken here (each is also listed in the design notes):
 *   R1  Eq. 2 prints the integer range as [0 .. 2^B]; B bits hold the 2^B codes
 *       0 .. 2^B-1, which is what is used.
 *   R2  Groups are g consecutive weights along the input (reduction) dimension of
 *       each output row; every group has one fp16 scale s and one fp16 zero z and
 *       a weight dequantises to w = (q - z) * s.
 *   R3  Eq. 5 prints {w0 = 0, w1 = 1 | w1/w0 < mu}, which would zero the primary;
 *       the text of Sec. 2.3.1 says only the primary is kept.  Read: when
 *       w1/w0 < mu (strict) the secondary is dropped and the primary weight becomes 1.
 *   R4  Routing weights are the full softmax over all experts restricted to the
 *       top-2 and renormalised to sum to 1 (Mixtral's gate).
 *   R5  Top-2 ties are broken towards the lower expert index.  Selection is
 *       decided on the logits rounded to fp32 (the precision the GPU decides in).
 *   R6  Mask byte 1 (or any value other than 0 and 2): the token is protected and
 *       never pruned (Sec. 2.3.2).  Mask byte 2: the token is dropped, all its
 *       experts are masked (Sec. 3.2, Fig. 9): weights (0, 0), no expert
 *       evaluated, its layer output is zero; pruned = 2 records it.
 *   R7  A 1-bit code is B~ = (sign(W)+1)/2 (Appendix A.2); it dequantises with the
 *       same formula using z = 1/2 and s = 2*alpha, giving w = +-alpha.
 *   R8  bits == 16 means the expert is not quantised: dense weights are used.
 *   R9  Routing weights are carried in fp32 from the gate to the combine.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* One weight matrix of one expert, [rows, cols] row-major, groups along cols.
 * bits in {1,2,3} uses codes/scale/zero; bits == 16 uses dense (R8). */
typedef struct {
    int rows, cols, group, bits;
    const uint8_t *codes;  /* [rows*cols], one code per byte, 0 .. 2^bits-1 */
    const float *scale;    /* [rows, cols/group]  (fp16 values, exactly converted) */
    const float *zero;     /* [rows, cols/group]  (fp16 values, exactly converted) */
    const float *dense;    /* [rows*cols]         (bits == 16 only) */
} mco_mat;

/* ---------------------------------------------------------------- dequant -- */

/* Sec. 2.1 (Eq. 2 grid, R1/R2) and App. A.2 (R7): the real value of weight (r, k). */
double mco_weight(const mco_mat *m, int r, int k)
{
    if (m->bits == 16)
        return (double)m->dense[(size_t)r * m->cols + k];
    int ng = m->cols / m->group;
    int gi = k / m->group;
    double q = (double)m->codes[(size_t)r * m->cols + k];
    double z = (double)m->zero[(size_t)r * ng + gi];
    double s = (double)m->scale[(size_t)r * ng + gi];
    return (q - z) * s;
}

/* The dequantised matrix in fp32, as the GPU materialises it: (float)q minus
 * (float)z, times (float)s, each step in fp32 (Sec. 2.1, R2).  Used to compare a
 * device dequantisation dump bit-exactly. */
void mco_dequant_f32(const mco_mat *m, float *out)
{
    int ng = m->cols / m->group;
    for (int r = 0; r < m->rows; ++r)
        for (int k = 0; k < m->cols; ++k) {
            if (m->bits == 16) {
                out[(size_t)r * m->cols + k] = m->dense[(size_t)r * m->cols + k];
                continue;
            }
            int gi = k / m->group;
            float q = (float)m->codes[(size_t)r * m->cols + k];
            float z = m->zero[(size_t)r * ng + gi];
            float s = m->scale[(size_t)r * ng + gi];
            float d = q - z;
            out[(size_t)r * m->cols + k] = d * s;
        }
}

/* y[r] = sum_k W[r,k] * x[k], fp64, one weight at a time. */
void mco_gemv(const mco_mat *m, const double *x, double *y)
{
    for (int r = 0; r < m->rows; ++r) {
        double acc = 0.0;
        for (int k = 0; k < m->cols; ++k)
            acc += mco_weight(m, r, k) * x[k];
        y[r] = acc;
    }
}

/* ------------------------------------------------------------------ expert -- */

/* The Mixtral expert E_i of Eq. 1: E(x) = W2 (silu(W1 x) * (W3 x)),
 * silu(a) = a / (1 + exp(-a)).  w1, w3: [F, H]; w2: [H, F].  fp64 throughout. */
void mco_expert(const mco_mat *w1, const mco_mat *w3, const mco_mat *w2,
                const double *x, double *out)
{
    int F = w1->rows;
    double *a1 = (double *)malloc(sizeof(double) * F);
    double *a3 = (double *)malloc(sizeof(double) * F);
    mco_gemv(w1, x, a1);
    mco_gemv(w3, x, a3);
    for (int f = 0; f < F; ++f) {
        double g = a1[f];
        double silu = g / (1.0 + exp(-g));
        a1[f] = silu * a3[f];
    }
    mco_gemv(w2, a1, out);
    free(a1);
    free(a3);
}

/* ----------------------------------------------------------------- routing -- */

/* Gate logits of Eq. 1: l[t,e] = sum_h x[t,h] * Wg[e,h], fp64. */
void mco_gate_logits(const float *x, const float *wg, int T, int H, int E, double *logits)
{
    for (int t = 0; t < T; ++t)
        for (int e = 0; e < E; ++e) {
            double acc = 0.0;
            for (int h = 0; h < H; ++h)
                acc += (double)x[(size_t)t * H + h] * (double)wg[(size_t)e * H + h];
            logits[(size_t)t * E + e] = acc;
        }
}

/*
 * Eq. 1 top-2 selection + softmax weights (R4, R5), then Eq. 5 ODP (R3) with the
 * token protection of Sec. 2.3.2 (R6).
 *   idx[t,0] = primary (largest logit), idx[t,1] = secondary.
 *   w[t,0..1] = renormalised softmax weights; (1, 0) when pruned.
 *   pruned[t] = 1 when the secondary was dropped.
 * mu is the per-layer threshold of Eq. 5; mu <= 0 never prunes (strict <).
 * protect may be NULL (nothing protected).
 */
void mco_route(const float *x, const float *wg, int T, int H, int E, double mu,
               const uint8_t *protect, int32_t *idx, float *w, uint8_t *pruned)
{
    double *l = (double *)malloc(sizeof(double) * (size_t)T * E);
    mco_gate_logits(x, wg, T, H, E, l);
    for (int t = 0; t < T; ++t) {
        const double *lt = l + (size_t)t * E;
        /* R5: decide on fp32-rounded logits, lower index wins ties. */
        int e0 = 0;
        for (int e = 1; e < E; ++e)
            if ((float)lt[e] > (float)lt[e0]) e0 = e;
        int e1 = (e0 == 0) ? 1 : 0;
        for (int e = 0; e < E; ++e)
            if (e != e0 && (float)lt[e] > (float)lt[e1]) e1 = e;
        /* R4: full softmax, keep the two, renormalise. */
        double mx = lt[e0], z = 0.0;
        for (int e = 0; e < E; ++e) z += exp(lt[e] - mx);
        double p0 = exp(lt[e0] - mx) / z;
        double p1 = exp(lt[e1] - mx) / z;
        double w0 = p0 / (p0 + p1);
        double w1 = p1 / (p0 + p1);
        /* Eq. 5 (R3) unless protected; a dropped token keeps no expert (R6). */
        const int drop = protect ? (protect[t] == 2) : 0;
        const int prot = protect ? (protect[t] != 0 && !drop) : 0;
        int prune = (!prot) && (w1 / w0 < mu);
        if (prune) { w0 = 1.0; w1 = 0.0; }
        if (drop) { w0 = 0.0; w1 = 0.0; prune = 2; }
        idx[2 * t + 0] = e0;
        idx[2 * t + 1] = e1;
        w[2 * t + 0] = (float)w0;
        w[2 * t + 1] = (float)w1;
        pruned[t] = (uint8_t)prune;
    }
    free(l);
}

/*
 * The token -> expert correspondence of Eq. 1 as a permutation: every kept
 * (token, slot) pair, grouped by expert, ascending token inside an expert.
 * offsets[E+1] (exclusive prefix counts), perm[P] with entry = 2*token + slot.
 * Returns P.  A pruned token's slot 1 is not a pair; a dropped token (pruned 2)
 * has no pair.
 */
int mco_permute(const int32_t *idx, const uint8_t *pruned, int T, int E,
                int32_t *offsets, int32_t *perm)
{
    int n = 0;
    offsets[0] = 0;
    for (int e = 0; e < E; ++e) {
        for (int t = 0; t < T; ++t)
            for (int slot = 0; slot < 2; ++slot) {
                if ((slot == 1 && pruned[t]) || pruned[t] == 2) continue;
                if (idx[2 * t + slot] == e) perm[n++] = 2 * t + slot;
            }
        offsets[e + 1] = n;
    }
    return n;
}

/* ------------------------------------------------------------------- layer -- */

/*
 * One MoE layer, Eq. 1 with Eq. 5: y_t = sum over kept slots of w * E_{idx}(x_t).
 * mats[3*e + m] for m = 0 (w1), 1 (w3), 2 (w2).
 * Only the tokens listed in `tokens` (n_tok of them) get an output row; routing
 * outputs are produced for all T tokens.  y is [n_tok, H] fp64.
 */
void mco_moe_layer(const float *x, const float *wg, int T, int H, int E,
                   const mco_mat *mats, double mu, const uint8_t *protect,
                   const int32_t *tokens, int n_tok,
                   int32_t *idx, float *w, uint8_t *pruned, double *y)
{
    mco_route(x, wg, T, H, E, mu, protect, idx, w, pruned);
    double *xt = (double *)malloc(sizeof(double) * H);
    double *eo = (double *)malloc(sizeof(double) * H);
    for (int i = 0; i < n_tok; ++i) {
        int t = tokens[i];
        for (int h = 0; h < H; ++h) xt[h] = (double)x[(size_t)t * H + h];
        double *yt = y + (size_t)i * H;
        for (int h = 0; h < H; ++h) yt[h] = 0.0;
        for (int slot = 0; slot < 2; ++slot) {
            if ((slot == 1 && pruned[t]) || pruned[t] == 2) continue;
            int e = idx[2 * t + slot];
            mco_expert(&mats[3 * e + 0], &mats[3 * e + 1], &mats[3 * e + 2], xt, eo);
            double wt = (double)w[2 * t + slot];
            for (int h = 0; h < H; ++h) yt[h] += wt * eo[h];
        }
    }
    free(xt);
    free(eo);
}

/* RMSNorm between stacked layers: x / sqrt(mean(x^2) + eps) * gamma, fp64. */
void mco_rmsnorm(const double *x, const float *gamma, int H, double eps, double *out)
{
    double ss = 0.0;
    for (int h = 0; h < H; ++h) ss += x[h] * x[h];
    double inv = 1.0 / sqrt(ss / H + eps);
    for (int h = 0; h < H; ++h) out[h] = x[h] * inv * (double)gamma[h];
}
