"""Pins for the CPU oracle: each test checks the oracle against something other than
itself -- a closed form from the paper, a library routine (numpy / torch), brute
force on tiny inputs, or an invariant the method fixes.  No GPU needed.

Together they are chosen so that a plausible slip in the oracle (a dropped term, a
wrong sign or index, a transposed operand, a swapped slot, a wrong tie-break, a
non-strict threshold) fails at least one of them; ``test_oracle_mutants.py``
checks exactly that by compiling deliberately broken copies of the oracle.
"""
import itertools

import numpy as np
import pytest
import torch

import oracle
import synth


def _rand_layer(T=12, H=32, F=48, E=4, group=16, bits=(1, 2, 3, 2), seed=7, **kw):
    return synth.make_layer(T, H, F, E, group, list(bits), seed, **kw)


def _mats(L):
    return [[oracle.QMat(*L.mat_shape(m), L.group, int(L.bits[e]), L.codes[e][m],
                         L.scale[e][m], L.zero[e][m]) for m in range(3)] for e in range(L.E)]


# ------------------------------------------------------------------ gate ----

def test_gate_logits_equal_library_matmul():
    L = _rand_layer(T=9, H=40, E=5, bits=(1, 2, 3, 2, 1))
    got = oracle.gate_logits(L.x_f32(), L.gate_f32())
    want = L.x_f32().astype(np.float64) @ L.gate_f32().astype(np.float64).T
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)
    # orientation: logits[t, e] uses row e of the gate (a transposed gate fails)
    assert got.shape == (9, 5)


def test_top2_matches_full_sort():
    """Eq. 1 top-2 against a stable sort of the fp32-rounded logits (library)."""
    L = _rand_layer(T=200, H=24, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False, gate_std=0.3)
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), mu=0.0)
    lg = oracle.gate_logits(L.x_f32(), L.gate_f32()).astype(np.float32)
    order = np.argsort(-lg, axis=1, kind="stable")  # ties -> lower index first
    np.testing.assert_array_equal(idx, order[:, :2].astype(np.int32))
    assert not pr.any()


def test_top2_tie_breaks_to_lower_index():
    # identical gate rows give identical logits: lower index must win both slots
    x = np.ones((1, 4), np.float32)
    wg = np.array([[0, 0, 0, 0], [1, 1, 1, 1], [1, 1, 1, 1], [1, 1, 1, 1]], np.float32)
    idx, w, _ = oracle.route(x, wg, mu=0.0)
    assert idx.tolist() == [[1, 2]]
    np.testing.assert_allclose(w, [[0.5, 0.5]], rtol=1e-7)


def test_weights_are_renormalised_softmax():
    """Weights = library softmax over all experts, restricted to top-2, renormalised."""
    L = _rand_layer(T=64, H=24, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False, gate_std=0.3)
    idx, w, _ = oracle.route(L.x_f32(), L.gate_f32(), mu=0.0)
    lg = torch.tensor(oracle.gate_logits(L.x_f32(), L.gate_f32()))
    p = torch.softmax(lg, dim=1).numpy()
    sel = np.take_along_axis(p, idx.astype(np.int64), axis=1)
    np.testing.assert_allclose(w, sel / sel.sum(1, keepdims=True), rtol=2e-7, atol=1e-7)
    np.testing.assert_allclose(w.sum(1), 1.0, rtol=1e-6)
    assert (w[:, 0] >= w[:, 1]).all()  # slot 0 is the primary


# ------------------------------------------------------------------- ODP ----

def _ratios(L):
    lg = torch.tensor(oracle.gate_logits(L.x_f32(), L.gate_f32()))
    p = torch.softmax(lg, dim=1)
    top = torch.topk(p, 2, dim=1).values.numpy()
    return top[:, 1] / top[:, 0]


def test_mu_zero_is_plain_top2():
    """Eq. 5 uses a strict '<' and w1/w0 > 0, so mu = 0 prunes nothing."""
    L = _rand_layer(T=80, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False, gate_std=0.5)
    i0, w0, p0 = oracle.route(L.x_f32(), L.gate_f32(), mu=0.0)
    assert not p0.any()
    i1, w1, p1 = oracle.route(L.x_f32(), L.gate_f32(), mu=-1.0)
    np.testing.assert_array_equal(i0, i1)
    np.testing.assert_array_equal(w0, w1)


def test_mu_above_one_prunes_every_unprotected_token():
    """w1/w0 <= 1 always, so mu > 1 prunes all but protected tokens (Sec. 2.3.2)."""
    L = _rand_layer(T=80, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False,
                    gate_std=0.5, protect_frac=0.25)
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), mu=1.0001, protect=L.protect)
    np.testing.assert_array_equal(pr, 1 - L.protect)
    # pruned: primary weight exactly 1, secondary exactly 0 (Eq. 5 as read)
    np.testing.assert_array_equal(w[pr == 1], np.tile([1.0, 0.0], (int(pr.sum()), 1)).astype(np.float32))
    # protected tokens keep the renormalised pair
    np.testing.assert_allclose(w[pr == 0].sum(1), 1.0, rtol=1e-6)
    assert (w[pr == 0][:, 1] > 0).all()


def test_prune_set_is_ratio_below_mu():
    """The pruned set is exactly {t unprotected : w1/w0 < mu}, checked on both sides
    of several tokens' own ratios (a flipped ratio or a lost protection fails)."""
    L = _rand_layer(T=60, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False,
                    gate_std=0.6, protect_frac=0.2)
    ratio = _ratios(L)
    for t in range(0, 60, 7):
        for mu, flip in ((float(ratio[t]) * (1 - 1e-9), False), (float(ratio[t]) * (1 + 1e-9), True)):
            _, _, pr = oracle.route(L.x_f32(), L.gate_f32(), mu=mu, protect=L.protect)
            want = (ratio < mu) & (L.protect == 0)
            np.testing.assert_array_equal(pr.astype(bool), want)
            # just below its own ratio a token is kept; just above it is pruned
            assert pr[t] == (flip and not L.protect[t])
    # monotone in mu
    counts = [oracle.route(L.x_f32(), L.gate_f32(), mu=m)[2].sum() for m in (0.1, 0.3, 0.5, 0.7, 0.9)]
    assert counts == sorted(counts)


def test_dropped_tokens_keep_no_expert():
    """Mask byte 2 drops the token (Sec. 3.2, Fig. 9): weights (0, 0), pruned = 2,
    the same top-2 indices as without the drop, no pair in the permutation; the
    other tokens route exactly as before."""
    L = _rand_layer(T=40, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False,
                    gate_std=0.6, protect_frac=0.2)
    base = oracle.route(L.x_f32(), L.gate_f32(), mu=0.5, protect=L.protect)
    mask = L.protect.copy()
    dropped = [3, 11, 25, int(np.flatnonzero(L.protect)[0])]  # a protected token can be dropped too
    mask[dropped] = 2
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), mu=0.5, protect=mask)
    np.testing.assert_array_equal(idx, base[0])
    keep = np.setdiff1d(np.arange(40), dropped)
    np.testing.assert_array_equal(w[keep], base[1][keep])
    np.testing.assert_array_equal(pr[keep], base[2][keep])
    assert (pr[dropped] == 2).all() and (w[dropped] == 0).all()
    offsets, perm = oracle.permute(idx, pr, 8)
    assert not set(perm.tolist()) & {2 * t + s for t in dropped for s in range(2)}
    assert offsets[-1] == 80 - int(pr.astype(int).sum())


# ----------------------------------------------------------- permutation ----

def test_permutation_brute_force():
    L = _rand_layer(T=50, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False,
                    gate_std=0.6, protect_frac=0.2)
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), mu=0.5, protect=L.protect)
    offsets, perm = oracle.permute(idx, pr, 8)
    pairs = sorted((int(idx[t, s]), t, s) for t in range(50) for s in range(2)
                   if not (s == 1 and pr[t]))
    assert perm.tolist() == [2 * t + s for (_, t, s) in pairs]
    for e in range(8):
        assert offsets[e + 1] - offsets[e] == sum(1 for p in pairs if p[0] == e)
    assert offsets[0] == 0 and offsets[-1] == 100 - pr.sum()


# ---------------------------------------------------------------- dequant ---

def test_dequant_closed_form_grid_points():
    """Eq. 2 grid: a weight that lies on the grid of its group comes back exactly."""
    r = np.random.default_rng(3)
    for bits in (2, 3):
        rows, cols, g = 6, 64, 16
        s = r.uniform(0.01, 0.05, (rows, cols // g)).astype(np.float16)
        z = r.integers(0, 2 ** bits, (rows, cols // g)).astype(np.float16)
        q = r.integers(0, 2 ** bits, (rows, cols)).astype(np.uint8)
        m = oracle.QMat(rows, cols, g, bits, q, s, z)
        d = oracle.dequant_f32(m)
        for rr, kk in [(0, 0), (5, 63), (3, 17), (2, 31), (4, 48)]:
            gi = kk // g
            want = (int(q[rr, kk]) - float(z[rr, gi])) * float(s[rr, gi])
            assert d[rr, kk] == np.float32(want)
            assert oracle.weight(m, rr, kk) == pytest.approx(want, rel=0, abs=0)
    # the largest code is 2^b - 1 (R1): code 7 at 3 bits, zero 0, scale 1 -> 7
    m = oracle.QMat(1, 8, 8, 3, np.full((1, 8), 7, np.uint8), np.ones((1, 1), np.float16),
                    np.zeros((1, 1), np.float16))
    assert oracle.dequant_f32(m)[0, 0] == 7.0


def test_one_bit_sign_transform_round_trip():
    """App. A.2: B~ = (sign(W)+1)/2 with sign(0)=+1, stored 1-bit; dequant with z=1/2,
    s=2*alpha returns alpha*sign(W) exactly."""
    r = np.random.default_rng(4)
    rows, cols, g = 5, 32, 32
    W = r.standard_normal((rows, cols)).astype(np.float32) * 0.02
    W[0, 3] = 0.0  # sign(0) = +1
    B = np.where(W >= 0, 1.0, -1.0)
    Bt = ((B + 1) / 2).astype(np.uint8)
    alpha = np.abs(W).mean(axis=1, keepdims=True).astype(np.float16)
    m = oracle.QMat(rows, cols, g, 1, Bt, (2 * alpha.astype(np.float32)).astype(np.float16),
                    np.full((rows, 1), 0.5, np.float16))
    d = oracle.dequant_f32(m)
    np.testing.assert_array_equal(d, (alpha.astype(np.float32) * B).astype(np.float32))
    assert d[0, 3] > 0


def test_one_bit_gemv_is_eq10_mac_free_form():
    """Eq. 10: s*xB = s*(sum_{B~=1} x - sum_{B~=0} x), per group."""
    r = np.random.default_rng(5)
    rows, cols, g = 7, 96, 32
    Bt = r.integers(0, 2, (rows, cols)).astype(np.uint8)
    alpha = r.uniform(0.01, 0.03, (rows, cols // g)).astype(np.float16)
    m = oracle.QMat(rows, cols, g, 1, Bt, (2 * alpha.astype(np.float32)).astype(np.float16),
                    np.full((rows, cols // g), 0.5, np.float16))
    x = r.standard_normal(cols)
    y = oracle.gemv(m, x)
    for rr in range(rows):
        want = 0.0
        for gi in range(cols // g):
            sl = slice(gi * g, (gi + 1) * g)
            xs, bs = x[sl], Bt[rr, sl]
            want += float(alpha[rr, gi]) * (xs[bs == 1].sum() - xs[bs == 0].sum())
        assert y[rr] == pytest.approx(want, rel=1e-12, abs=1e-12)


def test_gemv_group_factored_identity():
    """sum_k x_k (q_k - z) s = s (sum_k q_k x_k - z sum_k x_k) per group."""
    r = np.random.default_rng(6)
    for bits, g in [(2, 16), (3, 32), (1, 64)]:
        rows, cols = 5, 128
        q = r.integers(0, 2 ** bits, (rows, cols)).astype(np.uint8)
        s = r.uniform(0.01, 0.05, (rows, cols // g)).astype(np.float16)
        z = r.uniform(0, 2 ** bits - 1, (rows, cols // g)).astype(np.float16)
        m = oracle.QMat(rows, cols, g, bits, q, s, z)
        x = r.standard_normal(cols)
        y = oracle.gemv(m, x)
        qx = (q.astype(np.float64) * x).reshape(rows, cols // g, g).sum(-1)
        X = x.reshape(cols // g, g).sum(-1)
        want = (s.astype(np.float64) * (qx - z.astype(np.float64) * X[None, :])).sum(-1)
        np.testing.assert_allclose(y, want, rtol=1e-11, atol=1e-12)


def test_gemv_equals_library_matmul_of_dequantised():
    L = _rand_layer()
    m = _mats(L)[2][0]
    x = np.random.default_rng(8).standard_normal(m.cols)
    np.testing.assert_allclose(oracle.gemv(m, x), oracle.dequant_f32(m).astype(np.float64) @ x,
                               rtol=1e-10, atol=1e-12)


# ----------------------------------------------------------------- expert ---

def _torch_expert(W1, W3, W2, x):
    x = torch.as_tensor(x, dtype=torch.float64)
    a = torch.nn.functional.silu(x @ torch.as_tensor(W1, dtype=torch.float64).T)
    b = x @ torch.as_tensor(W3, dtype=torch.float64).T
    return ((a * b) @ torch.as_tensor(W2, dtype=torch.float64).T).numpy()


def test_expert_16bit_is_textbook_swiglu():
    """bits = 16: the expert is the unquantised Mixtral FFN, W2 (silu(W1 x) * W3 x)."""
    H, F = 24, 40
    W = [synth.bf16_bits_to_f32(w) for w in synth.dense_expert_weights(9, 0, H, F, std=0.2)]
    ms = [oracle.QMat(*w.shape, 8, 16, dense=w) for w in W]
    x = np.random.default_rng(9).standard_normal(H)
    np.testing.assert_allclose(oracle.expert(*ms, x), _torch_expert(*W, x), rtol=1e-10, atol=1e-12)


def test_expert_operands_not_swapped():
    """w1 carries the silu, w3 does not: swapping them changes the result."""
    L = _rand_layer()
    m = _mats(L)[0]
    x = np.random.default_rng(10).standard_normal(L.H)
    D = [oracle.dequant_f32(mm).astype(np.float64) for mm in m]
    np.testing.assert_allclose(oracle.expert(*m, x), _torch_expert(D[0], D[1], D[2], x), rtol=1e-9, atol=1e-12)
    assert not np.allclose(_torch_expert(D[1], D[0], D[2], x), _torch_expert(D[0], D[1], D[2], x))


# ------------------------------------------------------------------ layer ---

def _brute_layer(L, mats, mu, protect):
    """Every expert on every token (library matmuls), then Eq. 1 / Eq. 5 by hand."""
    D = [[oracle.dequant_f32(mm).astype(np.float64) for mm in me] for me in mats]
    lg = torch.tensor(oracle.gate_logits(L.x_f32(), L.gate_f32()))
    p = torch.softmax(lg, dim=1).numpy()
    y = np.zeros((L.T, L.H))
    for t in range(L.T):
        outs = [_torch_expert(*D[e], L.x_f32()[t]) for e in range(L.E)]
        best = None
        for a, b in itertools.permutations(range(L.E), 2):  # exhaustive pair search
            key = (np.float32(lg[t, a]), np.float32(lg[t, b]), -a, -b)
            if np.float32(lg[t, a]) < np.float32(lg[t, b]) or (
                    np.float32(lg[t, a]) == np.float32(lg[t, b]) and a > b):
                continue
            if best is None or key > best[0]:
                best = (key, a, b)
        _, a, b = best
        # routing weights are carried in fp32 between the gate and the combine
        wa = float(np.float32(p[t, a] / (p[t, a] + p[t, b])))
        wb = float(np.float32(p[t, b] / (p[t, a] + p[t, b])))
        if protect is not None and protect[t] == 2:  # dropped token: no expert (Sec. 3.2)
            continue
        prot = protect is not None and protect[t]
        if not prot and wb / wa < mu:
            y[t] = outs[a]
        else:
            y[t] = wa * outs[a] + wb * outs[b]
    return y


@pytest.mark.parametrize("mu", [0.0, 0.8])
@pytest.mark.parametrize("drop", [False, True])
def test_layer_brute_force_tiny(mu, drop):
    L = _rand_layer(T=10, H=16, F=24, E=4, group=8, bits=(1, 2, 3, 2), seed=11,
                    gate_std=0.5, protect_frac=0.3)
    if drop:  # two unprotected tokens dropped (Sec. 3.2, Fig. 9)
        L.protect[np.flatnonzero(L.protect == 0)[[1, 4]]] = 2
    mats = _mats(L)
    y, idx, w, pr = oracle.moe_layer(L.x_f32(), L.gate_f32(), mats, mu, L.protect)
    if mu > 0:
        assert 0 < (pr == 1).sum() < L.T  # the case exercises both branches
    np.testing.assert_allclose(y, _brute_layer(L, mats, mu, L.protect), rtol=1e-9, atol=1e-12)


def test_layer_token_subset_matches_full():
    L = _rand_layer(T=10, H=16, F=24, E=4, group=8, seed=12, gate_std=0.5)
    mats = _mats(L)
    y, *_ = oracle.moe_layer(L.x_f32(), L.gate_f32(), mats, 0.5)
    ys, *_ = oracle.moe_layer(L.x_f32(), L.gate_f32(), mats, 0.5, tokens=[7, 2])
    np.testing.assert_array_equal(ys, y[[7, 2]])


def test_layer_all_16bit_equals_unquantised_moe():
    """All experts at 16 bits reproduce the unquantised Mixtral block (torch)."""
    T, H, F, E = 6, 16, 32, 4
    L = _rand_layer(T=T, H=H, F=F, E=E, experts=False, gate_std=0.5, seed=13)
    W = [[synth.bf16_bits_to_f32(w) for w in synth.dense_expert_weights(13, e, H, F, std=0.2)]
         for e in range(E)]
    mats = [[oracle.QMat(*w.shape, 8, 16, dense=w) for w in We] for We in W]
    y, idx, w, pr = oracle.moe_layer(L.x_f32(), L.gate_f32(), mats, 0.0)
    xt = torch.tensor(L.x_f32(), dtype=torch.float64)
    logits = xt @ torch.tensor(L.gate_f32(), dtype=torch.float64).T
    top = torch.topk(torch.softmax(logits, 1), 2, dim=1)
    ww = (top.values / top.values.sum(1, keepdim=True)).float().double()
    want = np.zeros((T, H))
    for t in range(T):
        for s in range(2):
            e = int(top.indices[t, s])
            want[t] += float(ww[t, s]) * _torch_expert(*W[e], L.x_f32()[t])
    np.testing.assert_allclose(y, want, rtol=1e-9, atol=1e-12)


def test_rmsnorm_textbook():
    x = np.random.default_rng(14).standard_normal(64)
    g = np.random.default_rng(15).uniform(0.5, 1.5, 64).astype(np.float32)
    xt = torch.tensor(x)
    want = (xt * torch.rsqrt((xt * xt).mean() + 1e-5) * torch.tensor(g, dtype=torch.float64)).numpy()
    np.testing.assert_allclose(oracle.rmsnorm(x, g), want, rtol=1e-12)


# -------------------------------------------------------------- stacking ----

def test_bf16_round_matches_library_cast():
    x = np.concatenate([np.random.default_rng(16).standard_normal(2000) * 10.0 ** np.arange(-4, 4).repeat(250),
                        [1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 0.0]])
    want = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(oracle.bf16_round(x), want)


def test_stack_with_zero_experts_is_identity():
    """Experts whose every weight is zero (codes equal to the zero point) add
    nothing: any number of layers returns the bf16 input."""
    L = _rand_layer(bits=(2, 2, 2, 2))
    for e in range(L.E):
        for m in range(3):
            L.codes[e][m][:] = 1
            L.zero[e][m][:] = 1.0
    gates = [synth.gaussian_bf16(3, (l,), (L.E, L.H), 0.1) for l in range(3)]
    h, _ = oracle.stack(L.x_f32(), [synth.bf16_bits_to_f32(g) for g in gates], _mats(L), [0.0, 0.3, 0.0])
    np.testing.assert_array_equal(h, L.x_f32().astype(np.float64))


def test_stack_composes_layer_by_layer():
    L = _rand_layer(T=6, bits=(3, 1, 2, 2))
    gates = [synth.bf16_bits_to_f32(synth.gaussian_bf16(4, (l,), (L.E, L.H), 0.1)) for l in range(2)]
    mats = _mats(L)
    both, routes = oracle.stack(L.x_f32(), gates, mats, [0.2, 0.0], L.protect)
    first, r0 = oracle.stack(L.x_f32(), gates[:1], mats, [0.2], L.protect)
    second, r1 = oracle.stack(first, gates[1:], mats, [0.0], L.protect)
    np.testing.assert_array_equal(both, second)
    np.testing.assert_array_equal(routes[1][0], r1[0][0])


def test_stack_one_layer_is_residual_of_normalised_layer():
    """One layer with every rounding written out: bf16(x + bf16(MoE(bf16(RMSNorm x))))."""
    L = _rand_layer(T=5, bits=(2, 3, 1, 2))
    g = synth.bf16_bits_to_f32(synth.gaussian_bf16(5, (0,), (L.E, L.H), 0.1))
    x = L.x_f32().astype(np.float64)
    rms = np.sqrt((x * x).mean(axis=1, keepdims=True) + 1e-5)
    xn = torch.tensor(x / rms, dtype=torch.float32).to(torch.bfloat16).double().numpy()
    y, *_ = oracle.moe_layer(xn, g, _mats(L), 0.0)
    yb = torch.tensor(y, dtype=torch.float32).to(torch.bfloat16).double().numpy()
    want = torch.tensor(x + yb, dtype=torch.float32).to(torch.bfloat16).double().numpy()
    h, _ = oracle.stack(L.x_f32(), [g], _mats(L), [0.0])
    np.testing.assert_array_equal(h, want)


# ---------------------------------------------------- token importance (N2) ---

def _causal_softmax(nh, L, seed, temp=1.0):
    rng = np.random.default_rng(seed)
    s = rng.standard_normal((nh, L, L)) * temp
    s = np.where(np.tril(np.ones((L, L), bool))[None], s, -np.inf)
    e = np.exp(s - s.max(axis=2, keepdims=True))
    return e / e.sum(axis=2, keepdims=True)


def test_importance_uniform_causal_attention_is_harmonic():
    """Every query spreads evenly over the keys it sees (A[i, j] = 1/(i+1), j <= i):
    the attention key j receives is H_L - H_j (harmonic numbers), so Eq. 6 gives
    I_j = ||t_j||_1 (H_L - H_j) / (L - j)."""
    L, H = 37, 8
    t = np.random.default_rng(40).standard_normal((L, H))
    A = np.tril(np.ones((L, L))) / np.arange(1, L + 1)[:, None]
    imp, _ = oracle.token_importance(t, A[None], 0.0)
    harm = np.concatenate([[0.0], np.cumsum(1.0 / np.arange(1, L + 1))])
    want = np.abs(t).sum(1) * (harm[L] - harm[:L]) / (L - np.arange(L))
    np.testing.assert_allclose(imp, want, rtol=1e-12)


def test_importance_one_hot_attention_and_ties():
    """All queries attend to key 0 only: I_0 = ||t_0||_1, every other token 0; the
    mask takes token 0, then the zero-importance tokens by ascending index."""
    L = 10
    t = np.random.default_rng(41).standard_normal((L, 4)) + 3.0
    A = np.zeros((1, L, L))
    A[0, :, 0] = 1.0
    imp, mask = oracle.token_importance(t, A, 0.3)
    np.testing.assert_allclose(imp, np.r_[np.abs(t[0]).sum(), np.zeros(L - 1)], rtol=1e-12)
    assert mask.tolist() == [1, 1, 1] + [0] * (L - 3)


def test_importance_is_linear_in_the_heads_and_uses_l1():
    """Eq. 6 is linear in A and in the l1 norm: two heads give the mean of the
    one-head importances; scaling a token scales its importance by |c|; the sign
    of its entries does not matter."""
    L, H = 20, 6
    t = np.random.default_rng(42).standard_normal((L, H))
    A = _causal_softmax(2, L, 43)
    both, _ = oracle.token_importance(t, A, 0.0)
    one = [oracle.token_importance(t, A[h:h + 1], 0.0)[0] for h in range(2)]
    np.testing.assert_allclose(both, 0.5 * (one[0] + one[1]), rtol=1e-12)
    t2 = t.copy()
    t2[5] *= -3.0
    imp2, _ = oracle.token_importance(t2, A, 0.0)
    np.testing.assert_allclose(imp2[5], 3.0 * both[5], rtol=1e-12)
    np.testing.assert_allclose(np.delete(imp2, 5), np.delete(both, 5), rtol=1e-12)


def test_importance_mask_size_and_brute_force():
    """The mask holds ceil(frac * L) tokens, each at least as important as any
    unmasked one (lower index on ties), checked against an exhaustive count."""
    L = 30
    t = np.random.default_rng(44).standard_normal((L, 5))
    A = _causal_softmax(3, L, 45)
    for frac in (0.0, 0.02, 0.1, 0.5, 1.0):
        imp, mask = oracle.token_importance(t, A, frac)
        n = int(np.ceil(float(np.float32(frac)) * L - 1e-6))
        assert mask.sum() == n
        for j in range(L):
            better = sum(1 for i in range(L) if imp[i] > imp[j] or (imp[i] == imp[j] and i < j))
            assert mask[j] == (better < n)


def test_odp_threshold_is_quantile_of_prunable_ratios():
    """q = 0.5 is the median of w1/w0 over the prunable tokens (Sec. 2.3.1), the
    quantile follows numpy's linear rule, protected / dropped tokens are left out,
    and mu = the q-quantile prunes (strictly below it) about a q share."""
    L = _rand_layer(T=101, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False, gate_std=0.5)
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), mu=0.0)
    r = w[:, 1].astype(np.float64) / w[:, 0]
    assert oracle.odp_threshold(w, None, 0.5) == pytest.approx(np.median(r), rel=1e-12)
    for q in (0.0, 0.15, 0.9, 1.0):
        assert oracle.odp_threshold(w, None, q) == pytest.approx(np.quantile(r, q), rel=1e-12)
    mask = np.zeros(101, np.uint8)
    mask[::3] = 1
    mask[1::7] = 2
    assert oracle.odp_threshold(w, mask, 0.5) == pytest.approx(np.median(r[mask == 0]), rel=1e-12)
    mu = oracle.odp_threshold(w, None, 0.15)
    _, _, pr = oracle.route(L.x_f32(), L.gate_f32(), mu=mu)
    assert abs(pr.mean() - 0.15) <= 1.0 / 101 + 1e-12


# ---------------------------------------------------- PMQ allocation (N3) ---

def test_pmq_tiny_by_hand():
    """E = 3, budget 6: only the 6 permutations of (1, 2, 3) are feasible (2,2,2
    has no 3-bit expert); the objective of each written out by hand."""
    phi, w = [0.5, 1.0, 0.5], [0.2, 0.6, 0.2]
    eps = [[4.0, 2.0, 1.0], [3.0, 2.0, 0.5], [5.0, 1.0, 0.2]]
    best, arg = None, None
    for b in itertools.permutations((1, 2, 3)):
        obj = sum(phi[i] * w[i] * eps[i][b[i] - 1] ** 2 for i in range(3))
        if best is None or obj < best - 1e-15:
            best, arg = obj, b
    bits, obj = oracle.pmq_allocate(phi, w, eps, 6)
    assert tuple(bits) == arg and obj == pytest.approx(best, rel=1e-12)


def test_pmq_invariances_and_exchange():
    """Scaling every eps by c > 0 keeps the allocation; with alpha = beta = 0 only
    eps matters; of two experts with the same eps row (falling with the bit
    width) the more significant one never gets fewer bits."""
    rng = np.random.default_rng(46)
    E = 6
    phi, w = rng.uniform(0.1, 0.6, E), rng.uniform(0.05, 0.3, E)
    eps = np.sort(rng.uniform(0.1, 5.0, (E, 3)), axis=1)[:, ::-1]  # 1 bit worst
    b0, _ = oracle.pmq_allocate(phi, w, eps, 13)
    b1, _ = oracle.pmq_allocate(phi, w, 3.7 * eps, 13)
    np.testing.assert_array_equal(b0, b1)
    b2, _ = oracle.pmq_allocate(np.ones(E), np.ones(E), eps, 13, alpha=0.0, beta=0.0)
    b3, _ = oracle.pmq_allocate(phi, w, eps, 13, alpha=0.0, beta=0.0)
    np.testing.assert_array_equal(b2, b3)
    eps2 = eps.copy()
    eps2[1] = eps2[0]
    phi2 = phi.copy()
    phi2[0], phi2[1] = 0.9, 0.2  # expert 0 more significant than expert 1
    for total in (10, 12, 14):
        b, _ = oracle.pmq_allocate(phi2, w * 0 + 0.2, eps2, total)
        assert b[0] >= b[1]


def test_pmq_infeasible_budget():
    assert oracle.pmq_allocate([1, 1], [1, 1], [[1, 1, 1]] * 2, 6) is None  # (3,3) has no 2-bit expert
    assert oracle.pmq_allocate([1, 1, 1], [1, 1, 1], [[1, 1, 1]] * 3, 10) is None  # > 3 bits each


def test_expert_significance_sums():
    """phi sums to the activations per token (2 - pruned secondaries - 2 x dropped,
    over T) and w to the non-dropped share (each kept token's weights sum to 1)."""
    L = _rand_layer(T=90, E=8, bits=(1, 2, 3, 2, 1, 2, 3, 3), experts=False, gate_std=0.5, protect_frac=0.1)
    mask = L.protect.copy()
    mask[[3, 30, 60]] = 2
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), 0.5, mask)
    phi, wact = oracle.expert_significance(idx, w, pr, 8)
    n_pruned, n_drop = int((pr == 1).sum()), int((pr == 2).sum())
    assert phi.sum() == pytest.approx((2 * 90 - n_pruned - 2 * n_drop) / 90, rel=1e-12)
    assert wact.sum() == pytest.approx((90 - n_drop) / 90, rel=1e-6)
    for e in range(8):  # brute force count
        n = sum(1 for t in range(90) for s in range(2) if idx[t, s] == e and not ((s and pr[t]) or pr[t] == 2))
        assert phi[e] == pytest.approx(n / 90, rel=1e-12)


# ------------------------------------------------------- eps_{i,j} (N3) ----

def _eps_setup(T=10, H=32, F=48, E=4, group=16, seed=51):
    """Unquantised weights N(0, 0.02) (fp16 values) and their 1/2/3-bit quantisations."""
    L = synth.make_layer(T, H, F, E, group, [2] * E, seed, gate_std=0.3, experts=False)
    dense, quant = [], []
    for e in range(E):
        ws = [synth.expert_weights_f32(seed, e, m, *L.mat_shape(m)).astype(np.float16).astype(np.float32)
              for m in range(3)]
        dense.append([oracle.QMat(*L.mat_shape(m), group, 16, dense=ws[m]) for m in range(3)])
        quant.append([[oracle.QMat(*L.mat_shape(m), group, j, *synth.rtn_quantize(ws[m], j, group))
                       for m in range(3)] for j in (1, 2, 3)])
    return L, dense, quant


def test_expert_error_is_the_routing_weighted_expert_difference():
    """Sec. 2.2.2's eps_{i,j} (two whole layers per (i, j)) equals, by the linearity
    of Eq. 1 in the expert outputs with the routing unchanged, the F-norm of
    w_i(t) (E_i^Q(x_t) - E_i^16(x_t)) over the tokens, built from the routing
    weights and the single-expert function instead."""
    L, dense, quant = _eps_setup()
    eps = oracle.expert_error(L.x_f32(), L.gate_f32(), dense, quant)
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), 0.0)
    x = L.x_f32().astype(np.float64)
    for i in range(L.E):
        for j in range(3):
            rows = []
            for t in range(L.T):
                wi = sum(float(w[t, s]) for s in range(2) if idx[t, s] == i)
                d = oracle.expert(*quant[i][j], x[t]) - oracle.expert(*dense[i], x[t])
                rows.append(wi * d)
            assert eps[i, j] == pytest.approx(np.linalg.norm(np.stack(rows)), rel=1e-9, abs=1e-12)


def test_expert_error_invariants():
    """An expert no token is routed to has eps = 0; a 'quantisation' equal to the
    dense expert gives eps = 0; doubling an expert's W2 (dense and quantised alike)
    doubles its eps and leaves the others'."""
    L, dense, quant = _eps_setup(seed=52)
    idx, _, _ = oracle.route(L.x_f32(), L.gate_f32(), 0.0)
    unused = [e for e in range(L.E) if e not in set(idx.reshape(-1).tolist())]
    eps = oracle.expert_error(L.x_f32(), L.gate_f32(), dense, quant)
    for e in unused:
        assert np.all(eps[e] == 0.0)
    same = [[dense[e]] * 3 for e in range(L.E)]
    assert np.all(oracle.expert_error(L.x_f32(), L.gate_f32(), dense, same) == 0.0)
    i = int(idx[0, 0])
    d2 = [list(m) for m in dense]
    q2 = [[list(m) for m in qe] for qe in quant]
    d2[i][2] = oracle.QMat(*L.mat_shape(2), L.group, 16, dense=2.0 * dense[i][2].dense)
    for j in range(3):
        c, s_, z = quant[i][j][2].codes, quant[i][j][2].scale, quant[i][j][2].zero
        q2[i][j][2] = oracle.QMat(*L.mat_shape(2), L.group, j + 1, c, 2.0 * s_, z)
    eps2 = oracle.expert_error(L.x_f32(), L.gate_f32(), d2, q2)
    np.testing.assert_allclose(eps2[i], 2.0 * eps[i], rtol=1e-9)
    others = [e for e in range(L.E) if e != i]
    np.testing.assert_allclose(eps2[others], eps[others], rtol=1e-12)


def test_odp_threshold_is_strict_at_equality():
    """Eq. 5 prunes when w1/w0 < mu, strictly.  Two identical gate rows give a
    token bit-equal top-2 logits, so w0 = w1 and w1/w0 = 1 exactly: at mu = 1 the
    secondary is kept (weights 1/2, 1/2), just above 1 it is pruned."""
    L = _rand_layer(T=6, H=24, E=4, experts=False)
    g = L.gate_f32().copy()
    g[1] = g[0]
    x = np.abs(L.x_f32()) + 0.1  # logits of experts 0 and 1 the largest
    g[0] = g[1] = 0.5
    g[2:] = -0.5
    idx, w, pr = oracle.route(x, g, 1.0)
    assert (idx[:, 0] == 0).all() and (idx[:, 1] == 1).all()
    assert (w[:, 0] == w[:, 1]).all() and (pr == 0).all()
    _, w2, pr2 = oracle.route(x, g, np.nextafter(1.0, 2.0))
    assert (pr2 == 1).all() and (w2[:, 0] == 1.0).all() and (w2[:, 1] == 0.0).all()
