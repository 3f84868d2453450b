"""PMQ calibration through the library (Sec. 2.2): the expert errors eps_{i,j} of
Sec. 2.2.2 measured with the library's own kernels, the expert significance of
Sec. 2.2.1 from its routing, and the Eq. 4 allocation (mc_pmq_allocate).

eps_{i,j} = || F(theta) - F(theta[e_i -> Q(e_i, j)]) ||_F is the layer output
with only expert i quantised to j bits against the unquantised layer.  The gate
is not quantised, so the routing is the same in both layers, and by the linearity
of Eq. 1 in the expert outputs the difference is sum over the tokens routed to i
of w_i(t) (E_i^Q(x_t) - E_i(x_t)).  Each E_i(x_t) comes from mc_moe_forward on a
two-expert layer that holds expert i twice behind a zero gate: both logits are 0,
both slots get weight 1/2 and the combine returns E_i(x_t) itself (rounded to the
layer's bf16 output).  The unquantised expert runs as a 16-bit expert.  What is
done on the host is the weighting by the routing weights and the norm of a
[T, H] difference (offline calibration, not the layer's hot path).

The quantisation function Q (GPTQ in the paper) is the caller's: it passes, per
expert and bit width, the canonical codes / scale / zero the library packs.
"""
from __future__ import annotations

import numpy as np

from . import Shape, expert_significance, moe_forward, pack_experts, pmq_allocate, route


def _expert_on_tokens(x, H, F, group, bits, mats):
    """E(x_t) for every row of x (device bf16 [T, H]) of one expert given as
    canonical (codes, scale, zero) triples for w1, w3, w2 (bits 16: fp16 weights
    in `codes`, scale / zero None), through a two-expert layer holding it twice."""
    import torch
    shape = Shape(2, H, F, group)
    codes = [m[0] for m in mats] * 2
    scales = [m[1] for m in mats] * 2
    zeros = [m[2] for m in mats] * 2
    packed = pack_experts(shape, [bits, bits], codes, scales, zeros, device=x.device)
    gate = torch.zeros((2, H), dtype=torch.bfloat16, device=x.device)
    return moe_forward(x, gate, shape, [bits, bits], packed)


def expert_error(x, gate_w, shape: Shape, dense, quantized, mu: float = 0.0, protect=None):
    """eps [E, 3] (fp64): eps[i][j-1] of Sec. 2.2.2 over the calibration tokens x
    (device bf16 [T, H]) routed by gate_w (device bf16 [E, H]) at threshold mu.
    dense[e] = (w1, w3, w2) fp16 arrays ([F,H], [F,H], [H,F]); quantized[e][j-1] =
    three (codes, scale, zero) triples of expert e quantised to j bits."""
    import torch
    r = route(x, gate_w, shape, mu, protect)
    idx = r["idx"].cpu().numpy()
    w = r["w"].cpu().numpy().astype(np.float64)
    pr = r["pruned"].cpu().numpy()
    keep = np.stack([pr != 2, pr == 0], axis=1)
    eps = np.zeros((shape.E, 3))
    for i in range(shape.E):
        wi = np.where((idx == i) & keep, w, 0.0).sum(axis=1)  # w_i(t), 0 when not routed
        if not wi.any():
            continue
        dm = [(np.ascontiguousarray(m, dtype=np.float16), None, None) for m in dense[i]]
        y16 = _expert_on_tokens(x, shape.H, shape.F, shape.group, 16, dm).float().cpu().numpy().astype(np.float64)
        for j in range(3):
            yq = _expert_on_tokens(x, shape.H, shape.F, shape.group, j + 1,
                                   quantized[i][j]).float().cpu().numpy().astype(np.float64)
            eps[i, j] = float(np.linalg.norm(wi[:, None] * (yq - y16)))
    torch.cuda.synchronize()
    return eps


def calibrate(x, gate_w, shape: Shape, dense, quantized, bits_total: int, mu: float = 0.0, protect=None,
              alpha: float = 1.0, beta: float = 1.0, gamma: float = 2.0):
    """The PMQ bit table of one layer: significance (phi, w) from the library's
    routing of the calibration tokens (Sec. 2.2.1), eps from `expert_error`
    (Sec. 2.2.2), Eq. 4 solved exactly by mc_pmq_allocate.  Returns a dict with
    bits (int8 [E]), objective, eps, phi, wact."""
    r = route(x, gate_w, shape, mu, protect)
    phi, wact = expert_significance(r["idx"].cpu().numpy(), r["w"].cpu().numpy(), r["pruned"].cpu().numpy(),
                                    shape.E)
    eps = expert_error(x, gate_w, shape, dense, quantized, mu, protect)
    bits, obj = pmq_allocate(phi, wact, eps, bits_total, alpha, beta, gamma)
    return {"bits": bits, "objective": obj, "eps": eps, "phi": phi, "wact": wact}
