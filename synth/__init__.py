"""Seeded synthetic inputs for the MC MoE layer.

This module is shared by the tests, the benchmark and the smoke check: it is the
only code both the CUDA path and the CPU oracle see.  It draws random numbers and
converts number formats; it contains none of the layer's arithmetic (no gate, no
dequantisation, no expert, no pruning rule).

Workload shapes follow the Mixtral-8x7b MoE block (H = 4096, E = 8, top-2; the
paper's model table) with the SwiGLU width F = 14336 and the synthetic recipes
below:

* activations x ~ N(0, 1), rounded to bf16;
* gate weight Wg ~ N(0, 0.02), rounded to bf16 (optionally tilted along a shared
  direction so that expert loads are skewed);
* expert weights N(0, 0.02) quantised per group by ``rtn_quantize`` (round to
  nearest min-max for b = 2, 3; the sign rule of the paper's appendix for b = 1)
  in the named single-layer configurations; or, for the small test layers, the
  32-layer stack and the Mixtral-8x22b layer, codes drawn uniformly in
  [0, 2**b - 1] per weight (b = the expert's bit width), one fp16 scale per group
  with the magnitude a min-max quantiser gives an N(0, 0.02) group, an fp16 zero
  that is an integer in the code range for b >= 2 and 1/2 for b = 1 (the binary
  format of the paper's appendix); ``zero_mode="fractional"`` draws arbitrary
  fp16 zeros instead;
* protect masks choose a seeded subset of tokens.
"""
from __future__ import annotations

import concurrent.futures as cf
import os
from dataclasses import dataclass, field

import numpy as np

MIXTRAL_H = 4096
MIXTRAL_F = 14336
MIXTRAL_E = 8
# Mixtral-8x22b (Tab. model): H 6144, 8 experts; F is not in the paper: 16384
MIXTRAL22_H = 6144
MIXTRAL22_F = 16384


# ----------------------------------------------------------------- formats --

def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even float32 -> bf16, returned as uint16 bit patterns."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact bf16 (uint16 bits) -> float32."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def fp16_bits(a: np.ndarray) -> np.ndarray:
    """float16 array -> its uint16 bit patterns."""
    return np.ascontiguousarray(a, dtype=np.float16).view(np.uint16)


# ------------------------------------------------------------------ layout --

@dataclass
class Layer:
    """All inputs of one MoE layer, host side.

    x      uint16 [T, H]  bf16 bits        gate  uint16 [E, H] bf16 bits
    bits   int8 [E]                         group int
    codes  list over E of 3 uint8 arrays: w1 [F, H], w3 [F, H], w2 [H, F]
    scale, zero  list over E of 3 float16 arrays [rows, cols/group]
    protect uint8 [T] or None; mu float (Eq. 5 threshold; 0 = no pruning)
    """
    T: int
    H: int
    F: int
    E: int
    group: int
    bits: np.ndarray
    x: np.ndarray
    gate: np.ndarray
    codes: list
    scale: list
    zero: list
    protect: np.ndarray | None = None
    mu: float = 0.0
    meta: dict = field(default_factory=dict)

    def x_f32(self):
        return bf16_bits_to_f32(self.x)

    def gate_f32(self):
        return bf16_bits_to_f32(self.gate)

    def mat_shape(self, m: int):
        return (self.F, self.H) if m < 2 else (self.H, self.F)

    def mean_bits(self) -> float:
        return float(np.mean(self.bits))


def _rng(seed, *stream):
    return np.random.default_rng([int(seed)] + [int(s) for s in stream])


def gaussian_bf16(seed, stream, shape, std=1.0):
    r = _rng(seed, *stream)
    return f32_to_bf16_bits((r.standard_normal(shape, dtype=np.float32) * np.float32(std)))


def expert_matrix(seed, e, m, rows, cols, group, bits, zero_mode="integer"):
    """Codes, fp16 scale, fp16 zero for matrix m (0=w1, 1=w3, 2=w2) of expert e;
    for bits = 16 (the unquantised fp16 baseline) the fp16 weights ~ N(0, 0.02)
    and no scale / zero."""
    if bits == 16:
        w = (_rng(seed, 3000 + e, m).standard_normal((rows, cols), dtype=np.float32) * np.float32(0.02))
        return w.astype(np.float16), None, None
    r = _rng(seed, 1000 + e, m)
    n = rows * cols
    raw = np.frombuffer(r.bytes(n), dtype=np.uint8)
    codes = (raw & np.uint8((1 << bits) - 1)).reshape(rows, cols)
    ng = cols // group
    levels = (1 << bits) - 1
    # scale magnitude of a min-max quantiser on an N(0, 0.02) group of this size:
    # the expected range of g normals is ~ 2 * 2.6 sigma at g = 64..128.
    jitter = r.uniform(0.8, 1.25, size=(rows, ng)).astype(np.float32)
    if bits == 1:
        # binary format: s = 2 * alpha with alpha ~ mean |w| = 0.8 * 0.02; z = 1/2
        scale = (np.float32(2 * 0.8 * 0.02) * jitter).astype(np.float16)
        zero = np.full((rows, ng), 0.5, np.float16)
    else:
        scale = (np.float32(5.2 * 0.02 / levels) * jitter).astype(np.float16)
        if zero_mode == "integer":
            lo, hi = levels // 2, (levels + 1) // 2
            zero = r.integers(lo, hi + 1, size=(rows, ng)).astype(np.float16)
        elif zero_mode == "fractional":
            zero = r.uniform(0.0, float(levels), size=(rows, ng)).astype(np.float16)
        else:
            raise ValueError(zero_mode)
    return codes, scale, zero


def expert_weights_f32(seed, e, m, rows, cols, std=0.02):
    """The unquantised weights of matrix m (0=w1, 1=w3, 2=w2) of expert e:
    N(0, std) float32 [rows, cols], from their own seeded stream."""
    return _rng(seed, 4000 + e, m).standard_normal((rows, cols), dtype=np.float32) * np.float32(std)


def rtn_quantize(w, bits, group):
    """Quantiser of the synthetic expert weights (input generation: the paper
    quantises with GPTQ, Sec. 2.2.2, which needs calibration data and trained
    weights; this stands in for it), per group of `group` consecutive columns:
      b = 2, 3  round-to-nearest min-max: s = fp16((max - min) / (2^b - 1)), 1 if
                max = min; z = clip(rint(-min / s), 0, 2^b - 1), an integer stored
                in fp16; q = clip(rint(w / s + z), 0, 2^b - 1), ties to even;
      b = 1     the sign rule of App. A.2 with sign(0) = +1: q = (w >= 0), z = 1/2,
                s = fp16(2 * mean |w|) of the group (App. A.2's scale is per matrix;
                per group refines it in the same storage format).
    Returns (codes uint8 [rows, cols], scale fp16 [rows, cols/group], zero fp16)."""
    w = np.asarray(w, np.float32)
    rows, cols = w.shape
    ng = cols // group
    wg = w.reshape(rows, ng, group)
    if bits == 1:
        scale = (np.float32(2.0) * np.abs(wg).mean(axis=2, dtype=np.float32)).astype(np.float16)
        zero = np.full((rows, ng), 0.5, np.float16)
        return (w >= 0).astype(np.uint8), scale, zero
    levels = np.float32((1 << bits) - 1)
    mn, mx = wg.min(axis=2), wg.max(axis=2)
    scale = ((mx - mn) / levels).astype(np.float16)
    scale[scale == 0] = np.float16(1.0)
    s = scale.astype(np.float32)
    z = np.clip(np.rint(-mn / s), 0, levels)
    q = np.clip(np.rint(wg / s[:, :, None] + z[:, :, None]), 0, levels).astype(np.uint8)
    return q.reshape(rows, cols), scale, z.astype(np.float16)


def bit_table(seed, E, total, lo=1, hi=3):
    """A seeded per-expert bit table with the given sum, values in [lo, hi], with at
    least one 3-bit and one 2-bit expert (the constraints of the paper's Eq. 4)."""
    r = _rng(seed, 7)
    for _ in range(100000):
        b = r.integers(lo, hi + 1, size=E)
        if b.sum() == total and (b == 3).any() and (b == 2).any():
            return b.astype(np.int8)
    raise ValueError("no table")


def make_layer(T, H, F, E, group, bits, seed, *, gate_std=0.02, mu=0.0,
               protect_frac=0.0, zero_mode="integer", skew=None, experts=True, quant="direct"):
    """One layer of synthetic inputs.

    ``skew``: None, or (c, beta) -- x gets +c along a seeded unit direction u and
    gate row e gets +beta*(e - (E-1)/2)/((E-1)/2) * u, which tilts expert loads.
    ``experts=False`` skips the expert weights (routing-only tests).
    ``quant``: "direct" draws the codes uniformly with scales and zeros of a
    quantised N(0, 0.02) group's magnitude (``expert_matrix``); "rtn" draws the
    weights N(0, 0.02) and quantises them (``rtn_quantize``).  The matrices are
    generated on parallel host threads, each from its own seeded stream.
    """
    bits = np.asarray(bits, dtype=np.int8)
    assert bits.shape == (E,)
    xr = _rng(seed, 1).standard_normal((T, H), dtype=np.float32)
    gr = _rng(seed, 2).standard_normal((E, H), dtype=np.float32) * np.float32(gate_std)
    if skew is not None:
        c, beta = skew
        u = _rng(seed, 3).standard_normal(H).astype(np.float32)
        u /= np.linalg.norm(u)
        xr = xr + np.float32(c) * u[None, :]
        tilt = np.float32(beta) * (np.arange(E, dtype=np.float32) - (E - 1) / 2) / ((E - 1) / 2)
        gr = gr + tilt[:, None] * u[None, :]
    meta = {}
    if skew is not None:
        meta["skew_dir"] = u
        meta["skew_c"] = float(skew[0])
    x = f32_to_bf16_bits(xr)
    gate = f32_to_bf16_bits(gr)
    codes, scale, zero = [], [], []
    if experts:
        def one(em):
            e, m = em
            rows, cols = (F, H) if m < 2 else (H, F)
            if quant == "rtn" and int(bits[e]) != 16:
                return rtn_quantize(expert_weights_f32(seed, e, m, rows, cols), int(bits[e]), group)
            if quant not in ("direct", "rtn"):
                raise ValueError(quant)
            return expert_matrix(seed, e, m, rows, cols, group, int(bits[e]), zero_mode)
        jobs = [(e, m) for e in range(E) for m in range(3)]
        with cf.ThreadPoolExecutor(max(1, min(len(jobs), 8, os.cpu_count() or 1))) as ex:
            mats = list(ex.map(one, jobs))
        for e in range(E):
            codes.append([mats[3 * e + m][0] for m in range(3)])
            scale.append([mats[3 * e + m][1] for m in range(3)])
            zero.append([mats[3 * e + m][2] for m in range(3)])
    protect = None
    if protect_frac > 0:
        r = _rng(seed, 4)
        n = int(round(protect_frac * T))
        protect = np.zeros(T, np.uint8)
        protect[r.choice(T, size=n, replace=False)] = 1
    return Layer(T, H, F, E, group, bits, x, gate, codes, scale, zero, protect, float(mu), meta)


def resample_x_rows(layer: Layer, rows, seed, attempt):
    """Redraw the listed activation rows (same recipe, new stream)."""
    rows = np.asarray(rows, dtype=np.int64)
    if rows.size == 0:
        return
    r = _rng(seed, 5, attempt)
    new = r.standard_normal((rows.size, layer.H), dtype=np.float32)
    skew = layer.meta.get("skew_dir")
    if skew is not None:
        new = new + np.float32(layer.meta["skew_c"]) * skew[None, :]
    layer.x[rows] = f32_to_bf16_bits(new)


def dense_expert_weights(seed, e, H, F, std=0.02):
    """bf16 dense (unquantised, 16-bit) weights w1 [F,H], w3 [F,H], w2 [H,F]."""
    out = []
    for m in range(3):
        rows, cols = (F, H) if m < 2 else (H, F)
        out.append(gaussian_bf16(seed, (2000 + e, m), (rows, cols), std))
    return out


# ------------------------------------------------------------ named configs --

def config_tiny(seed=1235):
    """Tiny single layer: H 256, F 512, 8 experts, 64 tokens, group 64,
    bits [3,2,2,1,3,2,2,3], mu 0.3, 25% of tokens protected; expert weights
    N(0, 0.02) quantised by ``rtn_quantize``."""
    return make_layer(64, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], seed,
                      mu=0.3, protect_frac=0.25, quant="rtn")


def config_decode(T=16, seed=1236, bits_total=20):
    """Mixtral-8x7b-shaped decode layer: H 4096, F 14336, 8 experts, group 128,
    bits from {1,2,3} with sum 20 (mean 2.5, nearest feasible to 2.54), ODP off;
    expert weights N(0, 0.02) quantised by ``rtn_quantize``."""
    bits = bit_table(seed, 8, bits_total)
    return make_layer(T, MIXTRAL_H, MIXTRAL_F, MIXTRAL_E, 128, bits, seed, quant="rtn")


def importance_protect(x_bits, frac, seed):
    """Protect mask of the ODP workload: the top `frac` of tokens by a seeded
    importance surrogate, the L1 norm of the token's activations times a uniform
    draw standing in for its attention mass (ties to the lower index).  Input
    generation only: the mask is an input of the layer."""
    x = bf16_bits_to_f32(x_bits)
    score = np.abs(x).sum(axis=1, dtype=np.float64) * _rng(seed, 5).random(x.shape[0])
    n = int(np.ceil(frac * x.shape[0]))
    order = np.lexsort((np.arange(x.shape[0]), -score))  # score descending, index ascending
    protect = np.zeros(x.shape[0], np.uint8)
    protect[order[:n]] = 1
    return protect


def importance_mask(x_bits, protect_frac, drop_frac, seed):
    """Token mask with the Sec. 3.2 (Fig. 9) drop: the top `protect_frac` of tokens
    by the importance surrogate of `importance_protect` get 1 (protected), the
    bottom `drop_frac` get 2 (all experts masked), ties to the lower index.  Input
    generation only."""
    x = bf16_bits_to_f32(x_bits)
    score = np.abs(x).sum(axis=1, dtype=np.float64) * _rng(seed, 5).random(x.shape[0])
    order = np.lexsort((np.arange(x.shape[0]), -score))  # score descending, index ascending
    mask = np.zeros(x.shape[0], np.uint8)
    n_p = int(np.ceil(protect_frac * x.shape[0]))
    n_d = int(np.ceil(drop_frac * x.shape[0]))
    mask[order[:n_p]] = 1
    if n_d:
        mask[order[-n_d:]] = 2
    return mask


def config_odp(T=256, seed=1238, bits_total=20, protect_frac=0.10):
    """Mixtral-8x7b-shaped layer for ODP: 256 tokens, 10% protected by the
    importance surrogate, bits with sum 20 / 16 / 13 (mean 2.5 / 2.0 / 1.6).  The
    prune threshold mu is set by the caller from the layer's own routing (the
    value that prunes ~15% of the unprotected tokens' secondary experts); expert
    weights N(0, 0.02) quantised by ``rtn_quantize``."""
    bits = bit_table(seed, 8, bits_total)
    L = make_layer(T, MIXTRAL_H, MIXTRAL_F, MIXTRAL_E, 128, bits, seed, quant="rtn")
    L.protect = importance_protect(L.x, protect_frac, seed)
    return L


def config_stack(T=32, layers=32, seed=1239, bits_total=20, protect_frac=0.10, H=MIXTRAL_H, F=MIXTRAL_F,
                 E=MIXTRAL_E, group=128, gate_std=0.02):
    """A stack of `layers` pre-norm MoE layers (h <- h + MoE(RMSNorm(h)), RMSNorm
    weight 1): one seeded expert-weight set shared by every layer (the caller
    stores one device copy per layer, so each layer streams its own weights),
    a distinct seeded gate per layer, 10% of tokens protected by the importance
    surrogate.  Returns (layer, gates): `layer` carries x, the experts and the
    protect mask; gates[l] is layer l's gate (bf16 bits [E, H])."""
    bits = bit_table(seed, E, bits_total)
    L = make_layer(T, H, F, E, group, bits, seed, gate_std=gate_std)
    L.protect = importance_protect(L.x, protect_frac, seed)
    gates = [gaussian_bf16(seed, (6, l), (E, H), gate_std) for l in range(layers)]
    return L, gates


def config_decode_fp16(T=16, seed=1236):
    """The decode layer of config_decode with every expert unquantised (fp16
    weights, bits = 16): the baseline PMQ is compared with (Tab. 3's fp16)."""
    return make_layer(T, MIXTRAL_H, MIXTRAL_F, MIXTRAL_E, 128, [16] * MIXTRAL_E, seed)


def config_decode_22b(T=16, seed=1241, bits_total=20):
    """Mixtral-8x22b-shaped decode layer: H 6144, F 16384, 8 experts, group 128,
    bits from {1,2,3} with sum 20 (mean 2.5), ODP off."""
    bits = bit_table(seed, 8, bits_total)
    return make_layer(T, MIXTRAL22_H, MIXTRAL22_F, MIXTRAL_E, 128, bits, seed)


def config_prefill(T=4096, seed=1237, bits_total=20, skew=(3.0, 0.9)):
    """Mixtral-8x7b-shaped prefill layer with skewed expert loads, ODP off; expert
    weights N(0, 0.02) quantised by ``rtn_quantize``."""
    bits = bit_table(seed, 8, bits_total)
    return make_layer(T, MIXTRAL_H, MIXTRAL_F, MIXTRAL_E, 128, bits, seed, skew=skew, quant="rtn")


def causal_attention(nh, L, seed, temp=1.0):
    """Seeded synthetic attention probabilities fp32 [nh, L, L] (query i, key j):
    a causal softmax of standard normal scores times `temp`, one head at a time.
    Input generation for the token-importance step (Eq. 6)."""
    rng = _rng(seed, 6)
    out = np.empty((nh, L, L), np.float32)
    tri = np.tril(np.ones((L, L), bool))
    for h in range(nh):
        s = rng.standard_normal((L, L)) * temp
        s = np.where(tri, s, -np.inf)
        e = np.exp(s - s.max(axis=1, keepdims=True))
        out[h] = e / e.sum(axis=1, keepdims=True)
    return out
