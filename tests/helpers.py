"""Shared helpers for the GPU parity tests: device copies of synthetic inputs, the
oracle's matrices, routing-margin conditioning and the output tolerance."""
from __future__ import annotations

import concurrent.futures as cf
import os

import numpy as np

import oracle
import synth

# Output tolerance (fixed by the build's target): relative Frobenius error and
# max-abs error relative to max |ref| against the fp64 oracle.
REL_FRO = 5e-3
MAX_ABS = 2e-2


def flat(L, attr):
    a = getattr(L, attr)
    return [a[e][m] for e in range(L.E) for m in range(3)]


def oracle_mats(L):
    def one(e, m):
        if int(L.bits[e]) == 16:  # unquantised fp16 expert
            return oracle.QMat(*L.mat_shape(m), L.group, 16, dense=np.asarray(L.codes[e][m], np.float32))
        return oracle.QMat(*L.mat_shape(m), L.group, int(L.bits[e]), L.codes[e][m], L.scale[e][m], L.zero[e][m])
    return [[one(e, m) for m in range(3)] for e in range(L.E)]


def to_dev(L):
    import torch
    x = torch.from_numpy(L.x.view(np.int16).copy()).view(torch.bfloat16).cuda()
    g = torch.from_numpy(L.gate.view(np.int16).copy()).view(torch.bfloat16).cuda()
    p = None if L.protect is None else torch.from_numpy(L.protect.copy()).cuda()
    return x, g, p


def condition_routing(L, mu=0.0, margin=1e-3, seed=99, max_rounds=50):
    """Redraw activation rows whose fp64 logits sit within `margin` of a top-2
    tie (first/second or second/third) or of the ODP threshold, so that the fp32
    decisions of the GPU and the oracle cannot differ by rounding."""
    thr = -np.log(mu) if mu > 0 else np.inf
    for rnd in range(max_rounds):
        lg = oracle.gate_logits(L.x_f32(), L.gate_f32())
        srt = -np.sort(-lg, axis=1)
        bad = (srt[:, 0] - srt[:, 1] <= margin) | (srt[:, 1] - srt[:, 2] <= margin)
        if np.isfinite(thr):
            bad |= np.abs((srt[:, 0] - srt[:, 1]) - thr) <= margin
        rows = np.nonzero(bad)[0]
        if rows.size == 0:
            return L
        synth.resample_x_rows(L, rows, seed, rnd)
    raise RuntimeError("could not condition routing margins")


def oracle_layer(L, mats, tokens=None, threads=None):
    """Oracle outputs for the listed tokens, one token per host thread."""
    toks = list(range(L.T)) if tokens is None else list(tokens)
    xf, gf = L.x_f32(), L.gate_f32()
    if threads is None:
        threads = min(len(toks), os.cpu_count() or 1)
    if threads <= 1 or len(toks) <= 1:
        y, idx, w, pr = oracle.moe_layer(xf, gf, mats, L.mu, L.protect, tokens=toks)
        return y, idx, w, pr
    _, idx, w, pr = oracle.moe_layer(xf, gf, mats, L.mu, L.protect, tokens=[])
    with cf.ThreadPoolExecutor(threads) as ex:
        rows = list(ex.map(lambda t: oracle.moe_layer(xf, gf, mats, L.mu, L.protect, tokens=[t])[0][0], toks))
    return np.stack(rows), idx, w, pr


def errors(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    rel = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    mx = np.abs(got - ref).max() / max(np.abs(ref).max(), 1e-30)
    return rel, mx


def assert_close(got, ref, what=""):
    rel, mx = errors(got, ref)
    print("[parity] %s rel_fro=%.3e max_abs/max=%.3e" % (what, rel, mx))
    assert rel <= REL_FRO and mx <= MAX_ABS, "%s rel_fro=%.3e max_abs/max=%.3e" % (what, rel, mx)
    return rel, mx


def boundary_tokens(L, mu=None, blocks=(16, 128)):
    """Tokens whose outputs cover the edges of the expert kernels' work units at a
    full shape: for every expert, the first and the last pair of its first and of
    its last (ragged) block of `block` pairs, for each block size the kernels use
    (16-pair GEMV chunks, 128-pair GEMM token blocks).  The pairs come from the
    oracle's routing and permutation (pairs grouped by expert, ascending token).
    Every sampled token's output spans all W1|W3 row blocks and every W2 row
    block and column split."""
    mu = L.mu if mu is None else mu
    idx, _, pr = oracle.route(L.x_f32(), L.gate_f32(), mu, L.protect)
    off, perm = oracle.permute(idx, pr, L.E)
    toks = set()
    for e in range(L.E):
        a, b = int(off[e]), int(off[e + 1])
        if a == b:
            continue
        for blk in blocks:
            last = a + ((b - 1 - a) // blk) * blk  # first pair of the last block
            for q in (a, min(a + blk, b) - 1, last, b - 1):
                toks.add(int(perm[q]) >> 1)
    return sorted(toks)
