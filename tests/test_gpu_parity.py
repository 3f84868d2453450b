"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the same
seeded inputs.  Routing indices, prune flags, the permutation and the unpacked
codes must be bit-exact; layer outputs must be within rel-Frobenius 5e-3 and
max-abs 2e-2 * max|ref| of the fp64 oracle."""
import copy

import numpy as np
import pytest

import oracle
import synth
from helpers import (assert_close, condition_routing, errors, flat, oracle_layer, oracle_mats, to_dev)

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def mc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2410_06270_gb300 import build
    build.build()
    import paper_2410_06270_gb300 as m
    m.load()
    m.set_debug(0, 1_000_000_000)
    return m


def _pack(mc, L):
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    return shape, mc.pack_experts(shape, L.bits, flat(L, "codes"), flat(L, "scale"), flat(L, "zero"))


def _check_routing(mc, L, idx, w, pr, offsets=None, perm=None):
    oidx, ow, opr = oracle.route(L.x_f32(), L.gate_f32(), L.mu, L.protect)
    np.testing.assert_array_equal(idx.cpu().numpy(), oidx)
    np.testing.assert_array_equal(pr.cpu().numpy(), opr)
    np.testing.assert_allclose(w.cpu().numpy(), ow, rtol=2e-6, atol=2e-6)
    if offsets is not None:
        ooff, operm = oracle.permute(oidx, opr, L.E)
        np.testing.assert_array_equal(offsets.cpu().numpy(), ooff)
        np.testing.assert_array_equal(perm.cpu().numpy()[: ooff[-1]], operm)


# -------------------------------------------------------------- routing ----

def _with_drops(L, n, seed):
    """Drop n unprotected tokens (mask byte 2, Sec. 3.2 Fig. 9); returns their indices."""
    free = np.flatnonzero(L.protect == 0) if L.protect is not None else np.arange(L.T)
    if L.protect is None:
        L.protect = np.zeros(L.T, np.uint8)
    dropped = np.random.default_rng(seed).choice(free, size=n, replace=False)
    L.protect[dropped] = 2
    return np.sort(dropped)


@pytest.mark.parametrize("case", ["tiny", "odp", "odp_heavy", "many_tokens", "e16", "ragged_h", "drop_small",
                                  "drop"])
def test_route_bit_exact(mc, case):
    if case == "tiny":
        L = synth.config_tiny()
    elif case == "odp":
        L = synth.make_layer(200, 256, 128, 8, 64, [2] * 8, 31, gate_std=0.15, mu=0.3, protect_frac=0.25,
                             experts=False)
    elif case == "odp_heavy":
        L = synth.make_layer(300, 512, 128, 8, 128, [2] * 8, 32, gate_std=0.1, mu=0.8, protect_frac=0.1,
                             experts=False)
    elif case == "many_tokens":
        L = synth.make_layer(5000, 256, 128, 8, 64, [2] * 8, 33, gate_std=0.1, mu=0.5, protect_frac=0.02,
                             experts=False)
    elif case == "e16":
        L = synth.make_layer(100, 384, 128, 16, 128, [2] * 16, 34, gate_std=0.1, mu=0.6, experts=False)
    elif case == "ragged_h":  # H = 384 is a multiple of 128 but not of 256
        L = synth.make_layer(77, 384, 128, 8, 64, [2] * 8, 35, gate_std=0.1, mu=0.4, protect_frac=0.3,
                             experts=False)
    else:  # token drop: T = 48 takes the single-launch routing, T = 200 the two-launch one
        T = 48 if case == "drop_small" else 200
        L = synth.make_layer(T, 256, 128, 8, 64, [2] * 8, 37, gate_std=0.15, mu=0.3, protect_frac=0.1,
                             experts=False)
        dropped = _with_drops(L, T // 8, 38)
    condition_routing(L, L.mu)
    x, g, p = to_dev(L)
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    out = mc.route(x, g, shape, L.mu, p)
    torch.cuda.synchronize()
    _check_routing(mc, L, out["idx"], out["w"], out["pruned"], out["offsets"], out["perm"])
    if case != "tiny":
        assert 0 < int((out["pruned"] == 1).sum()) < L.T
    if case.startswith("drop"):
        np.testing.assert_array_equal(np.flatnonzero(out["pruned"].cpu().numpy() == 2), dropped)


@pytest.mark.parametrize("T", [1, 5, 17, 32, 33, 48, 64])
def test_single_launch_routing_places_like_the_two_launch_one(mc, T):
    """mc_moe_forward routes T <= 64 tokens in one launch whose last CTA places
    the pairs with one warp (ballots per 32-pair slice, a warp scan over the
    experts); debug bit 2 sends mc_route through that launch.  Offsets and the
    stable permutation must equal the oracle's and the two-launch placement's,
    with ODP pruning, protected tokens and dropped tokens in the batch."""
    L = synth.make_layer(T, 256, 128, 8, 64, [2] * 8, 90 + T, gate_std=0.15, mu=0.4, protect_frac=0.2,
                         experts=False)
    if T >= 5:
        _with_drops(L, max(1, T // 10), 91 + T)
    condition_routing(L, L.mu)
    x, g, p = to_dev(L)
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    two = mc.route(x, g, shape, L.mu, p)
    mc.set_debug(4, 0)
    try:
        for _ in range(3):  # the arrival word is back at zero after every call
            one = mc.route(x, g, shape, L.mu, p)
            torch.cuda.synchronize()
            _check_routing(mc, L, one["idx"], one["w"], one["pruned"], one["offsets"], one["perm"])
            for k in ("idx", "w", "pruned", "offsets"):
                assert torch.equal(one[k], two[k]), k
            n = int(two["offsets"][-1])
            assert torch.equal(one["perm"][:n], two["perm"][:n])
    finally:
        mc.set_debug(0, 1_000_000_000)


def test_route_mu_zero_and_above_one(mc):
    L = synth.make_layer(64, 256, 128, 8, 64, [2] * 8, 36, gate_std=0.2, protect_frac=0.25, experts=False)
    condition_routing(L, 0.0)
    x, g, p = to_dev(L)
    shape = mc.Shape(8, 256, 128, 64)
    a = mc.route(x, g, shape, 0.0, p)
    assert int(a["pruned"].sum()) == 0 and int(a["offsets"][-1]) == 2 * L.T
    b = mc.route(x, g, shape, 1.5, p)
    np.testing.assert_array_equal(b["pruned"].cpu().numpy(), 1 - L.protect)
    assert int(b["offsets"][-1]) == 2 * L.T - int((1 - L.protect).sum())


# ------------------------------------------------------------ unpacking ----

@pytest.mark.parametrize("group", [64, 128])
def test_device_unpack_bit_exact(mc, group):
    L = synth.make_layer(2, 256, 384, 4, group, [1, 2, 3, 2], 41, zero_mode="fractional")
    shape, packed = _pack(mc, L)
    mc.pack_verify(shape, L.bits, packed)
    for e in range(4):
        for m in range(3):
            c, s, z = mc.unpack_experts(shape, L.bits, packed, e, m)
            torch.cuda.synchronize()
            np.testing.assert_array_equal(c.cpu().numpy(), L.codes[e][m])
            np.testing.assert_array_equal(s.cpu().numpy().view(np.uint16), L.scale[e][m].view(np.uint16))
            np.testing.assert_array_equal(z.cpu().numpy().view(np.uint16), L.zero[e][m].view(np.uint16))


# ---------------------------------------------------------------- layer ----

def _forward_and_check(mc, L, tokens=None, path=None):
    condition_routing(L, L.mu)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    ws = mc.alloc_workspace(shape, L.T)
    old = mc.set_path(path) if path is not None else None
    try:
        y, r = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, workspace=ws, routing=True)
        mc.check_status(ws)
    finally:
        if old is not None:
            mc.set_path(old)
    torch.cuda.synchronize()
    _check_routing(mc, L, r["idx"], r["w"], r["pruned"])
    mats = oracle_mats(L)
    ref, *_ = oracle_layer(L, mats, tokens)
    got = y.float().cpu().numpy()
    if tokens is not None:
        got = got[list(tokens)]
    return assert_close(got, ref, "T=%d H=%d F=%d E=%d g=%d bits=%s mu=%g" % (
        L.T, L.H, L.F, L.E, L.group, list(map(int, L.bits)), L.mu))


def test_forward_tiny_config(mc):
    """H 256, F 512, 8 experts, 64 tokens, group 64, bits [3,2,2,1,3,2,2,3],
    mu 0.3, 25% of tokens protected."""
    _forward_and_check(mc, synth.config_tiny())


@pytest.mark.parametrize("T", [1, 2, 3, 8, 9, 16, 17, 40])
def test_forward_token_counts(mc, T):
    """Empty experts, one token, full n-tiles, ragged n-tiles and the chunked path."""
    L = synth.make_layer(T, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 50 + T, gate_std=0.1, mu=0.5,
                         protect_frac=0.25)
    _forward_and_check(mc, L)


@pytest.mark.parametrize("bits", [[1] * 4, [2] * 4, [3] * 4, [1, 3, 1, 3]])
@pytest.mark.parametrize("group", [64, 128])
def test_forward_bit_widths_and_groups(mc, bits, group):
    L = synth.make_layer(12, 512, 384, 4, group, bits, 60 + group + sum(bits), gate_std=0.1)
    _forward_and_check(mc, L)


def test_forward_fractional_zeros(mc):
    """Arbitrary fp16 zero points (HQQ-style storage), not only integer ones."""
    L = synth.make_layer(16, 384, 640, 8, 128, [3, 2, 1, 2, 3, 2, 1, 3], 70, gate_std=0.1,
                         zero_mode="fractional", mu=0.4, protect_frac=0.1)
    _forward_and_check(mc, L)


def test_forward_odd_row_blocks(mc):
    """H / 128 odd: the last W2 CTA has a single row stream."""
    L = synth.make_layer(10, 384, 256, 8, 64, [2, 3, 1, 2, 2, 3, 1, 2], 71, gate_std=0.1)
    _forward_and_check(mc, L)


def test_forward_sixteen_experts(mc):
    L = synth.make_layer(24, 256, 256, 16, 64, [1, 2, 3] * 5 + [2], 72, gate_std=0.1, mu=0.5)
    _forward_and_check(mc, L)


@pytest.mark.parametrize("T", [1, 4, 16])
def test_forward_mixtral_decode(mc, T):
    """Mixtral-8x7b-shaped decode layer (H 4096, F 14336, group 128, mean 2.5
    bits), outputs and routing on every token."""
    L = synth.config_decode(T=T)
    _forward_and_check(mc, L, tokens=list(range(T)))


def test_forward_mixtral_8x22b_decode(mc):
    """Mixtral-8x22b-shaped decode layer (H 6144, F 16384, group 128, mean 2.5
    bits), outputs on sampled tokens, routing on all tokens."""
    _forward_and_check(mc, synth.config_decode_22b(T=16), tokens=[0, 9, 15])


def test_forward_is_deterministic(mc):
    L = synth.make_layer(16, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 80, gate_std=0.1)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    y1 = mc.moe_forward(x, g, shape, L.bits, packed)
    y2 = mc.moe_forward(x, g, shape, L.bits, packed)
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))


@pytest.mark.parametrize("T", [40, 300])
def test_forward_token_drop(mc, T):
    """Dropped tokens (mask byte 2) get a zero output and the rest match the
    oracle; T = 40 takes the GEMV path, T = 300 the GEMM path."""
    L = synth.make_layer(T, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 84, gate_std=0.1, mu=0.3,
                         protect_frac=0.1)
    dropped = _with_drops(L, max(2, T // 20), 85)
    condition_routing(L, L.mu)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    y, r = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, routing=True)
    torch.cuda.synchronize()
    _check_routing(mc, L, r["idx"], r["w"], r["pruned"])
    got = y.float().cpu().numpy()
    assert (got[dropped] == 0).all()
    ref, *_ = oracle_layer(L, oracle_mats(L))
    assert_close(got, ref, "token drop T=%d" % T)


def test_one_workspace_serves_every_token_count(mc):
    """A workspace sized for 40 tokens serves calls with 1, 3, 16, 40 and again 1
    and 3 tokens: the words a call counts on (the single-launch routing's arrival
    count) sit at offsets that do not depend on T, so a call never finds another
    T's data there.  Every output matches the oracle and, bit for bit, a call
    with a fresh workspace of its own T."""
    ws = mc.alloc_workspace(mc.Shape(8, 256, 512, 64), 40)
    for T in (1, 3, 16, 40, 1, 3):
        L = synth.make_layer(T, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 87 + T, gate_std=0.1, mu=0.4,
                             protect_frac=0.2)
        condition_routing(L, L.mu)
        shape, packed = _pack(mc, L)
        x, g, p = to_dev(L)
        y = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, workspace=ws)
        y_fresh = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p)
        mc.check_status(ws)
        torch.cuda.synchronize()
        ref, *_ = oracle_layer(L, oracle_mats(L))
        assert_close(y.float().cpu().numpy(), ref, "shared workspace T=%d" % T)
        assert torch.equal(y, y_fresh), "shared vs fresh workspace, T=%d" % T


@pytest.mark.parametrize("T,path", [(8, 1), (40, 1), (8, 2), (130, 0)])
def test_forward_every_token_dropped(mc, T, path):
    """The degenerate batch: every token dropped (mask byte 2).  No pair reaches
    an expert, every expert kernel runs with zero work items, and the output is
    exactly zero; on the GEMV and the GEMM paths (T = 130 takes the GEMM
    automatically)."""
    L = synth.make_layer(T, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 86, gate_std=0.1, mu=0.3)
    L.protect = np.full(T, 2, np.uint8)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    prev = mc.set_path(path)
    try:
        y = torch.full_like(x, 7.0)
        y, r = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, y=y, routing=True)
        ws = mc.alloc_workspace(shape, T)
        y2 = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, workspace=ws)
        mc.check_status(ws)
        torch.cuda.synchronize()
    finally:
        mc.set_path(prev)
    assert (r["pruned"] == 2).all()
    assert (r["w"] == 0).all()
    assert (y.float() == 0).all() and (y2.float() == 0).all()


@pytest.mark.parametrize("T", [16, 300])
def test_forward_same_without_programmatic_launch(mc, T):
    """Kernels launched without programmatic dependent launch (each one starts
    only after the one before it ended) give bit-identical outputs; T = 300
    takes the GEMM path."""
    L = synth.make_layer(T, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 81, gate_std=0.1, mu=0.3,
                         protect_frac=0.1)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    y_on = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p)
    mc.set_debug(2, 0)
    try:
        y_off = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p)
    finally:
        mc.set_debug(0, 1_000_000_000)
    torch.cuda.synchronize()
    assert torch.equal(y_on.view(torch.int16), y_off.view(torch.int16))


def test_profile_events_inside_a_captured_graph(mc):
    """Profiling events captured into a CUDA graph are recorded again by every
    replay: each read reports the latest replay's launches and keeps the records
    until profile_clear."""
    L = synth.make_layer(16, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 82, gate_std=0.1)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    ws = mc.alloc_workspace(shape, L.T)
    y = torch.empty_like(x)
    mc.moe_forward(x, g, shape, L.bits, packed, y=y, workspace=ws)
    torch.cuda.synchronize()
    mc.profile_clear()
    mc.profile_select(["gemv_w13", "gemv_w2"])
    mc.profile_enable(True)
    gr = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(gr, stream=s):
            mc.moe_forward(x, g, shape, L.bits, packed, y=y, workspace=ws)
    torch.cuda.current_stream().wait_stream(s)
    mc.profile_enable(False)
    mc.profile_select(None)
    try:
        for _ in range(2):
            gr.replay()
            pr = mc.profile_read()
            assert set(pr) == {"gemv_w13", "gemv_w2"}
            assert all(n == 1 and ms > 0 for ms, n in pr.values())
    finally:
        mc.profile_clear()
    torch.cuda.synchronize()
    assert mc.profile_read() == {}


# ---------------------------------------------------------- device faults ----

@pytest.mark.parametrize("T", [4, 20])
def test_bounded_wait_reports_timeout_and_context_survives(mc, T):
    """Both GEMV kernels (one consumer group below 16 tokens, two from 16)."""
    L = synth.make_layer(T, 256, 256, 8, 64, [2] * 8, 90, gate_std=0.1)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    ws = mc.alloc_workspace(shape, L.T)
    mc.set_debug(1, 20_000_000)  # producer issues nothing; waits give up after 20 ms
    try:
        mc.moe_forward(x, g, shape, L.bits, packed, workspace=ws)
        with pytest.raises(mc.MCError) as ei:
            mc.check_status(ws)
        assert ei.value.code == mc.ERR_TIMEOUT
    finally:
        mc.set_debug(0, 1_000_000_000)
    y = mc.moe_forward(x, g, shape, L.bits, packed, workspace=ws)
    mc.check_status(ws)
    torch.cuda.synchronize()
    assert torch.isfinite(y.float()).all()


@pytest.mark.parametrize("T,path", [(4, "auto"), (20, "auto"), (20, "gemm")])
def test_corrupt_pack_header_is_reported(mc, T, path):
    """The packed header is checked once per call (by the kernel that prepares the
    activations) and the expert kernels copy nothing unless its verdict says the
    buffer matches; the verdict is rewritten by every call, so a good call after
    a bad one runs normally.  Both expert paths: the GEMV kernels (single-group
    at 4 tokens, two-group at 20) and the GEMM."""
    L = synth.make_layer(T, 256, 256, 8, 64, [2] * 8, 91, gate_std=0.1)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    bad = packed.clone()
    bad[0] ^= 0xFF
    with pytest.raises(mc.MCError) as ei:
        mc.pack_verify(shape, L.bits, bad)
    assert ei.value.code == mc.ERR_BAD_PACK
    old = mc.set_path(mc.PATH_GEMM if path == "gemm" else mc.PATH_AUTO)
    try:
        ws = mc.alloc_workspace(shape, L.T)
        y_good = mc.moe_forward(x, g, shape, L.bits, packed, workspace=ws).clone()
        mc.check_status(ws)
        mc.moe_forward(x, g, shape, L.bits, bad, workspace=ws)
        with pytest.raises(mc.MCError) as ei:
            mc.check_status(ws)
        assert ei.value.code == mc.ERR_BAD_PACK
        # the next call with the right buffer is not affected by the bad one
        y_again = mc.moe_forward(x, g, shape, L.bits, packed, workspace=ws)
        mc.check_status(ws)
        assert torch.equal(y_again, y_good)
        # a bit table that disagrees with the buffer is reported the same way, both
        # when the wrong entry is a routed expert's and when it only shifts the
        # offsets of the experts after it (expert 0 untouched by these tokens)
        idx, _, _ = oracle.route(L.x_f32(), L.gate_f32(), 0.0)
        touched = sorted(set(idx.reshape(-1).tolist()))
        shifting = [e for e in range(L.E) if e not in touched and any(t > e for t in touched)]
        for e in [touched[0]] + shifting[:1]:
            other = np.array(L.bits).copy()
            other[e] = 3 if other[e] != 3 else 1
            mc.moe_forward(x, g, shape, other, packed, workspace=ws)
            with pytest.raises(mc.MCError) as ei:
                mc.check_status(ws)
            assert ei.value.code == mc.ERR_BAD_PACK
    finally:
        mc.set_path(old)


def test_activation_outside_fp16_range_is_reported(mc):
    L = synth.make_layer(4, 256, 256, 8, 64, [2] * 8, 92, gate_std=0.1)
    L.x[2, 17] = synth.f32_to_bf16_bits(np.array([1e6], np.float32))[0]
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    ws = mc.alloc_workspace(shape, L.T)
    mc.moe_forward(x, g, shape, L.bits, packed, workspace=ws)
    with pytest.raises(mc.MCError) as ei:
        mc.check_status(ws)
    assert ei.value.code == mc.ERR_RANGE


# ------------------------------------------------------------- rmsnorm ----

@pytest.mark.parametrize("H", [4096, 16384, 1001])
def test_rmsnorm_and_add(mc, H):
    """RMSNorm against the oracle (16-byte rows up to H 16384 take the vector
    kernel, H 1001 the scalar one), in place too; the residual add exactly."""
    r = np.random.default_rng(5)
    xs = synth.f32_to_bf16_bits(r.standard_normal((6, H)).astype(np.float32) * 3)
    gs = synth.f32_to_bf16_bits(r.uniform(0.5, 1.5, H).astype(np.float32))
    x = torch.from_numpy(xs.view(np.int16)).view(torch.bfloat16).cuda()
    g = torch.from_numpy(gs.view(np.int16)).view(torch.bfloat16).cuda()
    y = mc.rmsnorm(x, g, 1e-5).float().cpu().numpy()
    for t in range(6):
        ref = oracle.rmsnorm(synth.bf16_bits_to_f32(xs[t]), synth.bf16_bits_to_f32(gs), 1e-5)
        rel, mx = errors(y[t], ref)
        assert rel < 4e-3 and mx < 8e-3
    xi = x.clone()
    mc.rmsnorm(xi, g, 1e-5, out=xi)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(xi.float().cpu().numpy(), y)
    s = mc.add(x, x).float().cpu().numpy()
    np.testing.assert_array_equal(s, 2 * synth.bf16_bits_to_f32(xs))
    s1 = mc.add(x.view(-1)[1:], x.view(-1)[1:]).float().cpu().numpy()  # odd length, unaligned: scalar kernel
    np.testing.assert_array_equal(s1, 2 * synth.bf16_bits_to_f32(xs).reshape(-1)[1:])
    if H % 8 == 0:
        # an unaligned row takes the scalar kernel, which sums in the vector
        # kernel's order for H % 8 == 0: the same bits
        buf = torch.empty(6 * H + 8, dtype=torch.bfloat16, device="cuda")
        xu = buf[1:1 + 6 * H].view(6, H)
        xu.copy_(x)
        yu = mc.rmsnorm(xu, g, 1e-5).float().cpu().numpy()
        np.testing.assert_array_equal(yu, y)


@pytest.mark.parametrize("path", [1, 2])
@pytest.mark.parametrize("group", [64, 128])
def test_forward_both_expert_paths(mc, path, group):
    """The mma.sync GEMV kernels (path 1) and the tcgen05 grouped GEMM (path 2,
    token blocks far from full here) against the oracle on the same layer."""
    L = synth.make_layer(20, 384, 512, 8, group, [3, 2, 1, 3, 2, 2, 1, 3], 95 + group, gate_std=0.1, mu=0.4,
                         protect_frac=0.2, zero_mode="fractional")
    _forward_and_check(mc, L, path=path)


# ------------------------------------------------- unquantised experts (N1) --

@pytest.mark.parametrize("T", [5, 40])
def test_forward_fp16_experts(mc, T):
    """Every expert unquantised (bits 16: fp16 weights, no scale / zero), the
    baseline of the mixed-bit layer: routing bit-exact, outputs against the
    oracle's dense experts; T = 40 has 9..16-pair chunks; W2 with an odd number
    of row blocks (H = 384)."""
    L = synth.make_layer(T, 384, 512, 8, 128, [16] * 8, 86, gate_std=0.1, mu=0.3, protect_frac=0.2)
    _forward_and_check(mc, L)


def test_forward_fp16_experts_mixtral(mc):
    """The Mixtral-8x7b decode layer with fp16 experts (the bench's baseline
    workload), sampled tokens."""
    _forward_and_check(mc, synth.config_decode_fp16(T=16), tokens=[0, 8, 15])


def test_fp16_experts_refuse_the_tensor_core_paths(mc):
    L = synth.make_layer(8, 256, 256, 8, 128, [16] * 8, 87, gate_std=0.1)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    old = mc.set_path(mc.PATH_GEMM)
    try:
        with pytest.raises(mc.MCError) as ei:
            mc.moe_forward(x, g, shape, L.bits, packed)
        assert ei.value.code == mc.ERR_UNSUPPORTED
    finally:
        mc.set_path(old)


# ------------------------------------------------------------ fp16 range --

def _heavy_tailed(L, seed, nch=4, lo=100.0, hi=1000.0):
    """A few activation channels at |x| in [lo, hi] (outlier features), the rest
    N(0, 1): the decode path's group fold starts each accumulator at -(O + z X),
    with field offsets of up to 2^10 per weight, so its fp32 cancellation grows
    with sum |x|."""
    r = np.random.default_rng(seed)
    xf = L.x_f32().copy()
    ch = r.choice(L.H, size=nch, replace=False)
    xf[:, ch] = (r.uniform(lo, hi, (L.T, nch)) * r.choice([-1.0, 1.0], (L.T, nch))).astype(np.float32)
    L.x = synth.f32_to_bf16_bits(xf)
    return ch


def _max_abs_h(L, mats):
    """Largest |silu(W1 x) * (W3 x)| over every token and expert (fp64, from the
    oracle's dequantised weights): the fp16 intermediate the kernels form."""
    x = L.x_f32().astype(np.float64)
    mx = 0.0
    for e in range(L.E):
        a1 = x @ oracle.dequant_f32(mats[e][0]).astype(np.float64).T
        a3 = x @ oracle.dequant_f32(mats[e][1]).astype(np.float64).T
        mx = max(mx, float(np.abs(a1 / (1.0 + np.exp(-a1)) * a3).max()))
    return mx


@pytest.mark.parametrize("T,path", [(12, 1), (12, 2), (300, 0)])
def test_forward_heavy_tailed_activations(mc, T, path):
    """Outlier channels at |x| ~ 100-1000 on both expert paths (GEMV; GEMM forced
    at 12 tokens and automatic at 300), against the oracle at the usual output
    tolerance; expert weights N(0, 0.02) quantised per group (the configs'
    recipe), so that h stays inside the fp16 range (checked first)."""
    L = synth.make_layer(T, 512, 384, 8, 128, [3, 2, 1, 3, 2, 2, 1, 3], 960 + T + path, gate_std=0.02,
                         quant="rtn")
    _heavy_tailed(L, 961 + T)
    condition_routing(L, L.mu)
    _heavy_tailed(L, 961 + T)  # resampled rows get their outlier channels back
    hmax = _max_abs_h(L, oracle_mats(L))
    print("[heavy] max |h| = %.4g" % hmax)
    assert hmax < 32768.0
    tokens = None if T <= 16 else [0, 1, 77, 150, 299]
    _forward_and_check(mc, L, tokens=tokens, path=path)


@pytest.mark.parametrize("T,path", [(8, 1), (8, 2)])
def test_h_outside_fp16_range_is_reported(mc, T, path):
    """x inside the fp16 range but h = silu(W1 x) * (W3 x) outside it: the W1,W3
    epilogue (GEMV and GEMM) records MC_ERR_RANGE in the status word, the call
    returns, and the same workspace serves a normal call afterwards."""
    L = synth.make_layer(T, 256, 256, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 970, gate_std=0.1)
    xf = L.x_f32() * np.float32(60.0)
    L.x = synth.f32_to_bf16_bits(xf)
    condition_routing(L)
    big = copy.deepcopy(L)
    for e in range(L.E):
        for m in range(2):
            big.scale[e][m] = (big.scale[e][m].astype(np.float32) * 200.0).astype(np.float16)
    shape, packed = _pack(mc, big)
    x, g, p = to_dev(big)
    ws = mc.alloc_workspace(shape, T)
    old = mc.set_path(path)
    try:
        mc.moe_forward(x, g, shape, big.bits, packed, 0.0, p, workspace=ws)
        with pytest.raises(mc.MCError) as ei:
            mc.check_status(ws)
        assert ei.value.code == mc.ERR_RANGE
        # the normal layer on the same workspace is reported clean and correct
        shape, packed = _pack(mc, L)
        y = mc.moe_forward(x, g, shape, L.bits, packed, 0.0, p, workspace=ws)
        mc.check_status(ws)
    finally:
        mc.set_path(old)
    ref, *_ = oracle_layer(L, oracle_mats(L))
    assert_close(y.float().cpu().numpy(), ref, "normal call after a range error")
