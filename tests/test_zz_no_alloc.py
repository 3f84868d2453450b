"""mc_moe_forward_static (the layer with the library's fixed device scratch, no
workspace) against mc_moe_forward on the same inputs, two calls in a row, within
the output tolerance of the parity tests, and against the oracle; its size limit;
and its bounded device waits (the mc_set_debug hook that starves the weight
producer makes them expire, and the caller's status word reports it).  The file
name sorts last so that it also runs after every other GPU test in one session."""
import numpy as np
import pytest

import synth
from helpers import assert_close, condition_routing, flat, oracle_layer, oracle_mats, to_dev

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


def _as_f32(y):
    return y.float().cpu().numpy().astype(np.float64)


def _static_twice_vs_workspace(mc, L, tokens=None):
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    ref = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p)
    # every buffer the no-allocation call writes exists before it runs
    y1, y2 = torch.empty_like(x), torch.empty_like(x)
    status = torch.zeros(1, dtype=torch.int32, device=x.device)
    mc.moe_forward_static(x, g, shape, L.bits, packed, L.mu, p, y=y1, status=status)
    mc.moe_forward_static(x, g, shape, L.bits, packed, L.mu, p, y=y2)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    r = _as_f32(ref)
    assert_close(_as_f32(y1), r, "static call 1 vs workspace")
    assert_close(_as_f32(y2), r, "static call 2 vs workspace")
    # and directly against the oracle (sampled tokens at the Mixtral shape)
    toks = list(range(L.T)) if tokens is None else list(tokens)
    ref_o, *_ = oracle_layer(L, oracle_mats(L), tokens=toks)
    assert_close(_as_f32(y2)[toks], ref_o, "static call vs oracle")


def test_static_matches_workspace_forward_odp(mc):
    """Small layer with ODP pruning and protected tokens, group 64, mixed bits."""
    L = synth.make_layer(64, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 1241, gate_std=0.1, mu=0.3,
                         protect_frac=0.25)
    condition_routing(L, mu=L.mu)
    _static_twice_vs_workspace(mc, L)


def test_static_matches_workspace_forward_decode(mc):
    """Mixtral-8x7b-shaped decode layer, 16 tokens (oracle on three of them)."""
    _static_twice_vs_workspace(mc, synth.config_decode(T=16), tokens=[0, 7, 15])


def test_static_bounded_waits_report_timeout(mc):
    """With the weight producer starved (mc_set_debug bit 0, 20 ms bound) every
    consumer wait of the static call runs out; the caller's status word gets
    MC_ERR_TIMEOUT, the call returns, and the next call on the same context is
    correct again."""
    L = synth.make_layer(24, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 1243, gate_std=0.1)
    condition_routing(L)
    shape, packed = _pack(mc, L)
    x, g, p = to_dev(L)
    status = torch.zeros(1, dtype=torch.int32, device=x.device)
    y = torch.empty_like(x)
    mc.set_debug(1, 20_000_000)
    try:
        mc.moe_forward_static(x, g, shape, L.bits, packed, 0.0, p, y=y, status=status)
        torch.cuda.synchronize()
    finally:
        mc.set_debug(0, 1_000_000_000)
    assert int(status.item()) == mc.ERR_TIMEOUT
    status.zero_()
    mc.moe_forward_static(x, g, shape, L.bits, packed, 0.0, p, y=y, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ref, *_ = oracle_layer(L, oracle_mats(L))
    assert_close(_as_f32(y), ref, "static call after an expired wait")


def test_static_rejects_T_beyond_scratch(mc):
    """At the Mixtral-8x7b shape the 16 MiB scratch holds T <= 96."""
    shape = mc.Shape(8, 4096, 14336, 128)
    bits = [2, 2, 3, 3, 1, 3, 3, 3]
    T = 97
    x = torch.zeros((T, 4096), dtype=torch.bfloat16, device="cuda")
    g = torch.zeros((8, 4096), dtype=torch.bfloat16, device="cuda")
    packed = torch.zeros(256, dtype=torch.uint8, device="cuda")
    with pytest.raises(mc.MCError) as ei:
        mc.moe_forward_static(x, g, shape, bits, packed)
    assert ei.value.code == mc.ERR_INVALID_ARG
    assert "static scratch" in str(ei.value)
