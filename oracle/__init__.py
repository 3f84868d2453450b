"""CPU oracle for the MC compressed MoE layer -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The product
library never imports it, and it imports nothing from the product library.

The arithmetic lives in ``mc_oracle.c`` (plain C, fp64, one weight at a time);
this module compiles it with gcc on first use and marshals numpy arrays.  Every
function states the passage of the paper it follows:

* ``gate_logits`` / ``route``   -- Sec. 2.1 Eq. 1 (top-2 gate), Sec. 2.3.1 Eq. 5
  (ODP), Sec. 2.3.2 (token protection).
* ``permute``                   -- the token/expert correspondence of Eq. 1.
* ``gemv`` / ``dequant_f32``    -- Sec. 2.1 (Eq. 2 integer grid), App. A.2 (1-bit).
* ``expert``                    -- the Mixtral SwiGLU expert E_i of Eq. 1.
* ``moe_layer``                 -- Eq. 1 with Eq. 5.
* ``rmsnorm``                   -- the normalisation between stacked layers.
* ``token_importance`` / ``select_top`` -- Sec. 2.3.2 Eq. 6 and the protect mask
  of the most important tokens; ``odp_threshold`` -- the Eq. 5 threshold as a
  quantile (the median in Sec. 2.3.1) of w1/w0 over calibration tokens.
* ``expert_significance`` / ``pmq_allocate`` -- Sec. 2.2.1 (phi, w) and the
  Eq. 4 integer program by brute force; ``expert_error`` -- the eps_{i,j} of
  Sec. 2.2.2 (layer output with one expert quantised against the unquantised
  layer).
* ``stack``                     -- pre-norm residual layers h <- h + MoE(RMSNorm(h)),
  each result rounded to bf16 where the stacked workload stores bf16.

Parity status: every function is pinned by ``tests/test_oracle_pins.py`` (closed
forms, library routines, brute force and invariants); none is "parity unpinned".
"""
from __future__ import annotations

import itertools

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mc_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libmc_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the C oracle with gcc (-O2, no fast-math, no vectorised reassociation)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-fno-fast-math",
                               "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _SO)
    return _SO


class _Mat(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int), ("cols", ctypes.c_int), ("group", ctypes.c_int),
                ("bits", ctypes.c_int),
                ("codes", ctypes.c_void_p), ("scale", ctypes.c_void_p),
                ("zero", ctypes.c_void_p), ("dense", ctypes.c_void_p)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            # MC_ORACLE_SO: load that build of mc_oracle.c instead (the mutant
            # tests point it at deliberately broken copies)
            lib = ctypes.CDLL(os.environ.get("MC_ORACLE_SO") or build())
            P = ctypes.c_void_p
            I = ctypes.c_int
            D = ctypes.c_double
            lib.mco_weight.restype = D
            lib.mco_weight.argtypes = [ctypes.POINTER(_Mat), I, I]
            lib.mco_dequant_f32.argtypes = [ctypes.POINTER(_Mat), P]
            lib.mco_gemv.argtypes = [ctypes.POINTER(_Mat), P, P]
            lib.mco_expert.argtypes = [ctypes.POINTER(_Mat)] * 3 + [P, P]
            lib.mco_gate_logits.argtypes = [P, P, I, I, I, P]
            lib.mco_route.argtypes = [P, P, I, I, I, D, P, P, P, P]
            lib.mco_permute.restype = I
            lib.mco_permute.argtypes = [P, P, I, I, P, P]
            lib.mco_moe_layer.argtypes = [P, P, I, I, I, P, D, P, P, I, P, P, P, P]
            lib.mco_rmsnorm.argtypes = [P, P, I, D, P]
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


class QMat:
    """One expert matrix [rows, cols]; groups of ``group`` along cols.

    ``codes`` uint8 [rows, cols] (0 .. 2**bits-1), ``scale``/``zero`` fp16 or fp32
    [rows, cols/group]; or ``bits=16`` with ``dense`` [rows, cols].
    """

    def __init__(self, rows, cols, group, bits, codes=None, scale=None, zero=None, dense=None):
        self.rows, self.cols, self.group, self.bits = int(rows), int(cols), int(group), int(bits)
        if bits == 16:
            self.dense = _f32(dense).reshape(rows, cols)
            self.codes = self.scale = self.zero = None
        else:
            self.codes = np.ascontiguousarray(codes, dtype=np.uint8).reshape(rows, cols)
            self.scale = _f32(np.asarray(scale).astype(np.float32)).reshape(rows, cols // group)
            self.zero = _f32(np.asarray(zero).astype(np.float32)).reshape(rows, cols // group)
            self.dense = None

    def c(self):
        return _Mat(self.rows, self.cols, self.group, self.bits,
                    _ptr(self.codes), _ptr(self.scale), _ptr(self.zero), _ptr(self.dense))


def weight(m: QMat, r: int, k: int) -> float:
    """Sec. 2.1 / App. A.2: the real value (q - z) * s of one weight (fp64)."""
    cm = m.c()
    return _load().mco_weight(ctypes.byref(cm), int(r), int(k))


def dequant_f32(m: QMat) -> np.ndarray:
    """Sec. 2.1: the whole matrix dequantised in fp32, ((float)q - (float)z) * (float)s."""
    out = np.empty((m.rows, m.cols), np.float32)
    cm = m.c()
    _load().mco_dequant_f32(ctypes.byref(cm), _ptr(out))
    return out


def gemv(m: QMat, x) -> np.ndarray:
    """y = W x with W dequantised one weight at a time, fp64."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty(m.rows, np.float64)
    cm = m.c()
    _load().mco_gemv(ctypes.byref(cm), _ptr(x), _ptr(y))
    return y


def expert(w1: QMat, w3: QMat, w2: QMat, x) -> np.ndarray:
    """Mixtral SwiGLU expert of Eq. 1: W2 (silu(W1 x) * W3 x), fp64."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(w2.rows, np.float64)
    a, b, c = w1.c(), w3.c(), w2.c()
    _load().mco_expert(ctypes.byref(a), ctypes.byref(b), ctypes.byref(c), _ptr(x), _ptr(out))
    return out


def gate_logits(x, wg) -> np.ndarray:
    """Eq. 1 gate: l = x Wg^T in fp64.  x [T,H], wg [E,H] (bf16 values as fp32)."""
    x, wg = _f32(x), _f32(wg)
    T, H = x.shape
    E = wg.shape[0]
    out = np.empty((T, E), np.float64)
    _load().mco_gate_logits(_ptr(x), _ptr(wg), T, H, E, _ptr(out))
    return out


def route(x, wg, mu: float, protect=None):
    """Eq. 1 top-2 + renormalised softmax weights, Eq. 5 ODP, Sec. 2.3.2 protection
    and the Sec. 3.2 (Fig. 9) token drop: protect byte 0 = prunable, 2 = dropped
    (weights (0, 0), no expert: pruned = 2), any other value = protected.

    Returns (idx int32 [T,2], w float32 [T,2], pruned uint8 [T]).
    """
    x, wg = _f32(x), _f32(wg)
    T, H = x.shape
    E = wg.shape[0]
    idx = np.empty((T, 2), np.int32)
    w = np.empty((T, 2), np.float32)
    pr = np.empty(T, np.uint8)
    prot = None if protect is None else np.ascontiguousarray(protect, dtype=np.uint8)
    _load().mco_route(_ptr(x), _ptr(wg), T, H, E, float(mu), _ptr(prot),
                      _ptr(idx), _ptr(w), _ptr(pr))
    return idx, w, pr


def permute(idx, pruned, E: int):
    """Kept (token, slot) pairs grouped by expert, ascending token: (offsets[E+1], perm[P])."""
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    pruned = np.ascontiguousarray(pruned, dtype=np.uint8)
    T = idx.shape[0]
    offsets = np.empty(E + 1, np.int32)
    perm = np.empty(2 * T, np.int32)
    n = _load().mco_permute(_ptr(idx), _ptr(pruned), T, E, _ptr(offsets), _ptr(perm))
    return offsets, perm[:n].copy()


def moe_layer(x, wg, mats, mu: float, protect=None, tokens=None):
    """Eq. 1 with Eq. 5 for the tokens listed (default all).

    ``mats`` is a list of E triples (w1, w3, w2) of QMat.  Returns
    (y fp64 [n_tok, H], idx, w, pruned).
    """
    x, wg = _f32(x), _f32(wg)
    T, H = x.shape
    E = wg.shape[0]
    flat = (_Mat * (3 * E))()
    for e in range(E):
        for m in range(3):
            flat[3 * e + m] = mats[e][m].c()
    toks = np.arange(T, dtype=np.int32) if tokens is None else np.ascontiguousarray(tokens, dtype=np.int32)
    y = np.empty((len(toks), H), np.float64)
    idx = np.empty((T, 2), np.int32)
    w = np.empty((T, 2), np.float32)
    pr = np.empty(T, np.uint8)
    prot = None if protect is None else np.ascontiguousarray(protect, dtype=np.uint8)
    _load().mco_moe_layer(_ptr(x), _ptr(wg), T, H, E, ctypes.cast(flat, ctypes.c_void_p),
                          float(mu), _ptr(prot), _ptr(toks), len(toks),
                          _ptr(idx), _ptr(w), _ptr(pr), _ptr(y))
    return y, idx, w, pr


def rmsnorm(x, gamma, eps: float = 1e-5) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * gamma for one vector, fp64."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    g = _f32(gamma)
    out = np.empty_like(x)
    _load().mco_rmsnorm(_ptr(x), _ptr(g), x.shape[0], float(eps), _ptr(out))
    return out


def bf16_round(a) -> np.ndarray:
    """Round to the nearest bf16 (ties to even), returned as fp64."""
    f = np.ascontiguousarray(a, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint32) << 16
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def stack(x, gates, mats, mus, protect=None, eps: float = 1e-5, gamma=None):
    """Pre-norm residual stack for the rows of x (bf16 values): per layer l,
    xn = bf16(RMSNorm(h)), y = bf16(MoE_l(xn)) with gate l and threshold mus[l],
    h = bf16(h + y).  Every token's trajectory is independent.  Returns
    (h after the last layer fp64 [T, H], per-layer (idx, w, pruned, layer input xn))."""
    h = bf16_round(x)
    T, H = h.shape
    g = np.ones(H, np.float32) if gamma is None else gamma
    routes = []
    for wg, mu in zip(gates, mus):
        xn = bf16_round(np.stack([rmsnorm(h[t], g, eps) for t in range(T)]))
        y, idx, w, pr = moe_layer(xn, wg, mats, mu, protect)
        h = bf16_round(h + bf16_round(y))
        routes.append((idx, w, pr, xn))
    return h, routes



def token_importance(t, attn, protect_frac: float):
    """Sec. 2.3.2, Eq. 6, in fp64: I_j = ||t_j||_1 * (sum_{i=j}^{L-1} Abar[i, j]) / (L - j)
    (0-based j; Abar = mean of the heads' attention probabilities attn[h, i, j],
    query i, key j; the mean attention key j receives from the queries that see it),
    and the protect mask of the ceil(protect_frac * L) most important tokens
    (``select_top``; the product taken within 1e-6 of an integer as that integer).  t [L, H] (bf16 values), attn [nh, L, L].  Returns
    (importance fp64 [L], mask uint8 [L])."""
    t = np.asarray(t, np.float64)
    A = np.asarray(attn, np.float64)
    nh, L, _ = A.shape
    Abar = A.sum(axis=0) / nh
    imp = np.empty(L, np.float64)
    for j in range(L):
        imp[j] = np.abs(t[j]).sum() * Abar[j:, j].sum() / (L - j)
    # ceil(frac * L), a product within 1e-6 of an integer counting as that integer
    # (frac arrives as fp32: 0.3 * 10 must give 3)
    n = int(np.ceil(float(np.float32(protect_frac)) * L - 1e-6))
    return imp, select_top(imp, n)


def select_top(imp, n: int):
    """Mask of the n tokens of largest importance, ties to the lower index."""
    imp = np.asarray(imp)
    order = sorted(range(len(imp)), key=lambda j: (-imp[j], j))
    mask = np.zeros(len(imp), np.uint8)
    mask[order[:max(0, min(n, len(imp)))]] = 1
    return mask


def odp_threshold(w, mask=None, q: float = 0.5) -> float:
    """Sec. 2.3.1: the Eq. 5 threshold as the q-quantile (0.5: the median the
    paper uses) of w1/w0 over the tokens that can be pruned (mask 0) and have a
    positive primary weight; linear between order statistics."""
    w = np.asarray(w, np.float64)
    keep = w[:, 0] > 0
    if mask is not None:
        keep &= np.asarray(mask) == 0
    r = np.sort(w[keep, 1] / w[keep, 0])
    pos = q * (len(r) - 1)
    lo = int(np.floor(pos))
    hi = min(lo + 1, len(r) - 1)
    return float(r[lo] + (pos - lo) * (r[hi] - r[lo]))


def expert_significance(idx, w, pruned, E: int):
    """Sec. 2.2.1: phi_i = n_i / N (activations of expert i per calibration token)
    and w_i = (sum of its routing weights) / N, N = the number of tokens; a pruned
    secondary (pruned 1) or a dropped token (pruned 2) is not an activation."""
    idx = np.asarray(idx)
    w = np.asarray(w, np.float64)
    T = idx.shape[0]
    pr = np.zeros(T, np.uint8) if pruned is None else np.asarray(pruned)
    phi, wact = np.zeros(E), np.zeros(E)
    for t in range(T):
        for s in range(2):
            if (s == 1 and pr[t]) or pr[t] == 2:
                continue
            phi[idx[t, s]] += 1
            wact[idx[t, s]] += w[t, s]
    return phi / T, wact / T


def expert_error(x, wg, dense_mats, quant_mats, mu: float = 0.0, protect=None):
    """Sec. 2.2.2: eps[i][j-1] = || F(theta) - F(theta[e_i -> Q(e_i, j)]) ||_F over
    the calibration tokens x [T, H]: the layer output (Eq. 1 with Eq. 5 at mu) with
    every expert unquantised, against the same layer with only expert i replaced by
    its j-bit quantisation; the gate is not quantised, so the routing is the same.
    dense_mats[e] = (w1, w3, w2) QMats with bits 16, quant_mats[e][j-1] = expert e
    quantised to j bits.  Returns eps fp64 [E, 3]."""
    E = len(dense_mats)
    y16, *_ = moe_layer(x, wg, dense_mats, mu, protect)
    eps = np.zeros((E, 3))
    for i in range(E):
        for j in range(3):
            mats = list(dense_mats)
            mats[i] = quant_mats[i][j]
            yq, *_ = moe_layer(x, wg, mats, mu, protect)
            eps[i, j] = float(np.linalg.norm(yq - y16))
    return eps


def pmq_allocate(phi, wact, eps, bits_total: int, alpha=1.0, beta=1.0, gamma=2.0):
    """Eq. 4 (Sec. 2.2.2) by brute force: every assignment x of {1, 2, 3} bits with
    sum = bits_total, at least one 3-bit and one 2-bit expert, minimising
    sum_i phi_i^alpha w_i^beta (eps_{i, x_i})^gamma.  Ties: the assignment met
    first when expert 0's width varies fastest.  Returns (bits, objective) or None
    when no assignment is feasible."""
    E = len(phi)
    best = None
    for combo in itertools.product((1, 2, 3), repeat=E):
        b = combo[::-1]  # expert 0 varies fastest
        if sum(b) != bits_total or 3 not in b or 2 not in b:
            continue
        obj = sum(phi[i] ** alpha * wact[i] ** beta * float(eps[i][b[i] - 1]) ** gamma for i in range(E))
        if best is None or obj < best[1]:
            best = (np.array(b, np.int8), obj)
    return best
