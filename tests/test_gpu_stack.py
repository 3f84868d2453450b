"""GPU parity of the stacked workload: pre-norm residual MoE layers
(h <- h + MoE_l(RMSNorm(h)), per-layer gates and ODP thresholds, protected
tokens) through mc_stack_forward against the oracle's stack; and the stack
captured into one CUDA graph equal, bit for bit, to the eager call (at the
Mixtral-8x7b shape too)."""
import numpy as np
import pytest

import oracle
import synth
from helpers import assert_close, flat, oracle_mats

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
