"""GPU parity of the stacked workload: pre-norm residual MoE layers
(h <- h + MoE_l(RMSNorm(h)), per-layer gates and ODP thresholds, protected
tokens) through mc_stack_forward against the oracle's stack; the Mixtral-8x7b
stack of 32 layers against the oracle layer by layer with teacher forcing; and
the stack captured into one CUDA graph equal, bit for bit, to the eager call (at
the Mixtral-8x7b shape too)."""
import os

import numpy as np
import pytest

import oracle
import synth
from helpers import assert_close, errors, flat, oracle_mats

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


def _dev_bf16(bits):
    return torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).cuda()


def _setup(mc, L, gates, mus, copies=True):
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    packed = mc.pack_experts(shape, L.bits, flat(L, "codes"), flat(L, "scale"), flat(L, "zero"))
    layers = len(gates)
    packs = [packed.clone() for _ in range(layers)] if copies else [packed] * layers
    args = mc.StackArgs([_dev_bf16(g) for g in gates], [L.bits] * layers, packs, mus)
    gamma = torch.ones((layers, L.H), dtype=torch.bfloat16, device="cuda")
    ws = mc.stack_workspace(shape, L.T)
    prot = None if L.protect is None else torch.from_numpy(L.protect.copy()).cuda()
    return shape, args, gamma, ws, prot


def _margins_ok(gates_f, routes, mus, margin=1e-3):
    """Tokens whose top-2 and ODP decisions are unambiguous at every layer."""
    ok = None
    for wg, (idx, w, pr, xn), mu in zip(gates_f, routes, mus):
        lg = oracle.gate_logits(xn, wg)
        srt = -np.sort(-lg, axis=1)
        good = (srt[:, 0] - srt[:, 1] > margin) & (srt[:, 1] - srt[:, 2] > margin)
        if mu > 0:
            good &= np.abs((srt[:, 0] - srt[:, 1]) + np.log(mu)) > margin
        ok = good if ok is None else ok & good
    return np.nonzero(ok)[0]


def test_stack_small_vs_oracle(mc):
    layers = 4
    L, gates = synth.config_stack(T=48, layers=layers, seed=401, H=256, F=512, E=8, group=64, gate_std=0.1)
    gates_f = [synth.bf16_bits_to_f32(g) for g in gates]
    mats = oracle_mats(L)
    _, r0 = oracle.stack(L.x_f32(), gates_f, mats, [0.0] * layers, L.protect)
    mus = []
    for (idx, w, pr, xn) in r0:
        ratio = w[:, 1].astype(np.float64) / w[:, 0]
        mus.append(float(np.quantile(ratio[L.protect == 0], 0.15)))
    ref, routes = oracle.stack(L.x_f32(), gates_f, mats, mus, L.protect)
    tokens = _margins_ok(gates_f, routes, mus)
    assert len(tokens) >= L.T // 2
    shape, args, gamma, ws, prot = _setup(mc, L, gates, mus)
    h = _dev_bf16(L.x)
    mc.stack_forward(h, shape, args, gamma, ws, prot)
    mc.check_status(ws)
    torch.cuda.synchronize()
    x0 = L.x_f32().astype(np.float64)
    got = h.float().cpu().numpy().astype(np.float64)
    # the layers' accumulated contribution h_L - x on the unambiguous tokens
    assert_close((got - x0)[tokens], (ref - x0)[tokens], "stack of %d layers, %d/%d tokens" % (
        layers, len(tokens), L.T))


@pytest.mark.parametrize("shape_name", ["small", "mixtral"])
def test_stack_graph_replay_equals_eager(mc, shape_name):
    if shape_name == "small":
        L, gates = synth.config_stack(T=32, layers=6, seed=402, H=256, F=512, E=8, group=64, gate_std=0.1)
        copies = True
    else:
        L, gates = synth.config_stack(T=32, layers=4, seed=403)
        copies = False
    mus = [0.2] * len(gates)
    shape, args, gamma, ws, prot = _setup(mc, L, gates, mus, copies=copies)
    h_eager = _dev_bf16(L.x)
    mc.stack_forward(h_eager, shape, args, gamma, ws, prot)
    torch.cuda.synchronize()
    h_graph = _dev_bf16(L.x)
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            mc.stack_forward(h_graph, shape, args, gamma, ws, prot)
    torch.cuda.current_stream().wait_stream(s)
    h_graph.copy_(_dev_bf16(L.x))
    g.replay()
    torch.cuda.synchronize()
    mc.check_status(ws)
    assert torch.equal(h_eager.view(torch.int16), h_graph.view(torch.int16))


def test_stack_fused_pre_norm_equals_separate_launches(mc):
    """With 16-byte aligned h and gamma each layer's RMSNorm runs in its routing
    launch and its residual add in its combine; an unaligned h (or gamma) takes
    mc_rmsnorm, the layer and mc_add as separate launches.  The results are bit
    for bit the same, with random (non-unit) gamma."""
    L, gates = synth.config_stack(T=24, layers=5, seed=405, H=256, F=512, E=8, group=64, gate_std=0.1)
    mus = [0.2] * len(gates)
    shape, args, gamma, ws, prot = _setup(mc, L, gates, mus, copies=True)
    rng = np.random.default_rng(405)
    gvals = torch.from_numpy((1.0 + 0.25 * rng.standard_normal(gamma.shape)).astype(np.float32)).to(torch.bfloat16)
    gamma.copy_(gvals.cuda())
    n = L.T * L.H
    h_fused = _dev_bf16(L.x)
    mc.stack_forward(h_fused, shape, args, gamma, ws, prot)
    # h two bytes past an aligned address: the separate-launch path
    buf = torch.empty(n + 8, dtype=torch.bfloat16, device="cuda")
    h_sep = buf[1:1 + n].view(L.T, L.H)
    h_sep.copy_(_dev_bf16(L.x))
    assert h_sep.data_ptr() % 16 != 0
    mc.stack_forward(h_sep, shape, args, gamma, ws, prot)
    # aligned h, unaligned gamma: separate RMSNorm, residual add in the combine
    gbuf = torch.empty(gamma.numel() + 8, dtype=torch.bfloat16, device="cuda")
    g_un = gbuf[1:1 + gamma.numel()].view(gamma.shape)
    g_un.copy_(gamma)
    h_gun = _dev_bf16(L.x)
    mc.stack_forward(h_gun, shape, args, g_un, ws, prot)
    torch.cuda.synchronize()
    mc.check_status(ws)
    assert torch.equal(h_fused.view(torch.int16), h_sep.view(torch.int16))
    assert torch.equal(h_fused.view(torch.int16), h_gun.view(torch.int16))


def test_stack_same_without_programmatic_launch(mc):
    """The stack with every kernel launched without programmatic dependent
    launch is bit-identical to the default (overlapped launches)."""
    L, gates = synth.config_stack(T=32, layers=6, seed=404, H=256, F=512, E=8, group=64, gate_std=0.1)
    mus = [0.2] * len(gates)
    shape, args, gamma, ws, prot = _setup(mc, L, gates, mus, copies=True)
    h_on = _dev_bf16(L.x)
    mc.stack_forward(h_on, shape, args, gamma, ws, prot)
    mc.set_debug(2, 0)
    try:
        h_off = _dev_bf16(L.x)
        mc.stack_forward(h_off, shape, args, gamma, ws, prot)
    finally:
        mc.set_debug(0, 1_000_000_000)
    torch.cuda.synchronize()
    mc.check_status(ws)
    assert torch.equal(h_on.view(torch.int16), h_off.view(torch.int16))


def test_stack_mixtral_teacher_forced(mc):
    """The stack workload at the Mixtral-8x7b shape (32 layers, 32 tokens, H 4096,
    F 14336, bits sum 20, ODP on with per-layer mu dropping the secondary expert
    of 15% of the unprotected tokens, 10% of tokens protected), checked layer by
    layer with teacher forcing: the oracle's layer l consumes the GPU's own bf16
    input to layer l (its RMSNorm output), so that every layer is compared on
    the same inputs however far the trajectories drift apart.
      - The layer-by-layer calls (mc_rmsnorm, mc_moe_forward, mc_add) reproduce
        mc_stack_forward bit for bit, so these are the stack's own layers.
      - Routing (top-2, weights, prune flags) against the oracle on every token
        whose fp64 logits lie more than 1e-4 from a top-2 tie or from the ODP
        threshold; the others are reported and excluded.
      - Every layer's output y_l on two tokens per layer (64 in all, every token
        twice), within the output tolerance.
      - The end-to-end drift of the whole stack against the oracle's own
        trajectory on two tokens is printed, not gated (Eq. 1 per layer; the
        paper's Mixtral models have 32 MoE layers)."""
    import concurrent.futures as cf
    layers, T = 32, 32
    L, gates = synth.config_stack(T=T, layers=layers)
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    packed = mc.pack_experts(shape, L.bits, flat(L, "codes"), flat(L, "scale"), flat(L, "zero"))
    gw = [_dev_bf16(g) for g in gates]
    gamma = torch.ones((layers, L.H), dtype=torch.bfloat16, device="cuda")
    prot = torch.from_numpy(L.protect.copy()).cuda()
    ws = mc.alloc_workspace(shape, T)
    # layer by layer, with the stack's per-layer thresholds from its own trajectory
    h = _dev_bf16(L.x)
    mus, xns, ys, routes = [], [], [], []
    for l in range(layers):
        xn = mc.rmsnorm(h, gamma[l])
        r0 = mc.route(xn, gw[l], shape, 0.0, prot)
        w0 = r0["w"].cpu().numpy().astype(np.float64)
        mus.append(float(np.quantile((w0[:, 1] / w0[:, 0])[L.protect == 0], 0.15)))
        y, r = mc.moe_forward(xn, gw[l], shape, L.bits, packed, mus[-1], prot, workspace=ws, routing=True)
        mc.check_status(ws)
        h = mc.add(h, y)
        xns.append(xn.view(torch.int16).cpu().numpy().view(np.uint16))
        ys.append(y.float().cpu().numpy().astype(np.float64))
        routes.append((r["idx"].cpu().numpy(), r["w"].cpu().numpy(), r["pruned"].cpu().numpy()))
    # the same layers through mc_stack_forward, bit for bit
    args = mc.StackArgs(gw, [L.bits] * layers, [packed] * layers, mus)
    hs = _dev_bf16(L.x)
    mc.stack_forward(hs, shape, args, gamma, mc.stack_workspace(shape, T), prot)
    torch.cuda.synchronize()
    assert torch.equal(hs.view(torch.int16), h.view(torch.int16))

    mats = oracle_mats(L)
    gates_f = [synth.bf16_bits_to_f32(g) for g in gates]
    excluded, jobs = 0, []
    for l in range(layers):
        xf = synth.bf16_bits_to_f32(xns[l])
        lg = oracle.gate_logits(xf, gates_f[l])
        srt = -np.sort(-lg, axis=1)
        clear = (srt[:, 0] - srt[:, 1] > 1e-4) & (srt[:, 1] - srt[:, 2] > 1e-4) & \
                (np.abs((srt[:, 0] - srt[:, 1]) + np.log(mus[l])) > 1e-4)
        excluded += int((~clear).sum())
        oidx, ow, opr = oracle.route(xf, gates_f[l], mus[l], L.protect)
        gidx, gwt, gpr = routes[l]
        np.testing.assert_array_equal(gidx[clear], oidx[clear], err_msg="layer %d top-2" % l)
        np.testing.assert_array_equal(gpr[clear], opr[clear], err_msg="layer %d prune flags" % l)
        np.testing.assert_allclose(gwt[clear], ow[clear], rtol=2e-6, atol=2e-6, err_msg="layer %d weights" % l)
        assert 0 < int((opr == 1).sum()) and int((opr[L.protect == 1] == 1).sum()) == 0
        toks = [t for t in ((2 * l) % T, (2 * l + 1) % T) if clear[t]]
        jobs += [(l, t, xf) for t in toks]
    print("[stack32] routing compared on %d of %d token-layers (%d within 1e-4 of a tie or the threshold)" % (
        layers * T - excluded, layers * T, excluded))
    assert excluded <= layers * T // 20

    def one(job):
        l, t, xf = job
        yo, *_ = oracle.moe_layer(xf, gates_f[l], mats, mus[l], L.protect, tokens=[t])
        return yo[0]

    with cf.ThreadPoolExecutor(os.cpu_count() or 4) as ex:
        refs = list(ex.map(one, jobs))
    for l in range(layers):
        sel = [i for i, j in enumerate(jobs) if j[0] == l]
        if sel:
            got = np.stack([ys[l][jobs[i][1]] for i in sel])
            assert_close(got, np.stack([refs[i] for i in sel]), "stack32 layer %d (teacher forced)" % l)
    got_all = np.concatenate([ys[jobs[i][0]][jobs[i][1]][None] for i in range(len(jobs))])
    rel, mx = errors(got_all, np.stack(refs))
    print("[stack32] all %d sampled layer outputs: rel_fro=%.3e max_abs/max=%.3e" % (len(jobs), rel, mx))

    # end-to-end drift of the whole stack on two tokens (reported only)
    drift_toks = [0, T - 1]

    def traj(t):
        return oracle.stack(L.x_f32()[t:t + 1], gates_f, mats, mus, L.protect[t:t + 1])[0][0]

    with cf.ThreadPoolExecutor(len(drift_toks)) as ex:
        h_ref = np.stack(list(ex.map(traj, drift_toks)))
    x0 = L.x_f32().astype(np.float64)[drift_toks]
    h_got = h.float().cpu().numpy().astype(np.float64)[drift_toks]
    rel, mx = errors(h_got - x0, h_ref - x0)
    print("[stack32] end-to-end drift after %d layers on tokens %s: rel_fro=%.3e max_abs/max=%.3e (not gated)" % (
        layers, drift_toks, rel, mx))
