"""GPU parity of the prefill expert path (tcgen05 grouped GEMM, token blocks of
128 pairs, A operand dequantised into tensor memory) against the CPU oracle:
ragged token blocks, empty and overloaded experts, an odd number of W2 row
blocks, both group sizes, fractional zeros, ODP with protected tokens, the
automatic path switch, and the Mixtral-8x7b-shaped prefill layer on sampled
tokens."""
import numpy as np
import pytest

import synth
from helpers import assert_close, boundary_tokens, condition_routing, flat, oracle_layer, oracle_mats, to_dev

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

PATH_GEMM = 2  # mc_set_path: the tcgen05 grouped GEMM


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


def _run(mc, L, path, tokens=None):
    condition_routing(L, L.mu)
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    packed = mc.pack_experts(shape, L.bits, flat(L, "codes"), flat(L, "scale"), flat(L, "zero"))
    x, g, p = to_dev(L)
    ws = mc.alloc_workspace(shape, L.T)
    old = mc.set_path(path)
    try:
        y = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, workspace=ws)
        mc.check_status(ws)
    finally:
        mc.set_path(old)
    torch.cuda.synchronize()
    got = y.float().cpu().numpy()
    return got if tokens is None else got[list(tokens)]


def _check(mc, L, path=PATH_GEMM, tokens=None):
    got = _run(mc, L, path, tokens)
    ref, *_ = oracle_layer(L, oracle_mats(L), tokens)
    return assert_close(got, ref, "prefill path=%d T=%d H=%d F=%d g=%d bits=%s mu=%g" % (
        path, L.T, L.H, L.F, L.group, list(map(int, L.bits)), L.mu))


@pytest.mark.parametrize("group", [64, 128])
def test_prefill_small_layer(mc, group):
    """H 384 (three W2 row blocks: one pair plus a lone block), ragged blocks."""
    L = synth.make_layer(300, 384, 512, 8, group, [3, 2, 1, 3, 2, 2, 1, 3], 301 + group, gate_std=0.1, mu=0.4,
                         protect_frac=0.2, zero_mode="fractional")
    _check(mc, L)


@pytest.mark.parametrize("bits", [[1] * 8, [2] * 8, [3] * 8])
def test_prefill_single_bit_width(mc, bits):
    L = synth.make_layer(260, 256, 256, 8, 64, bits, 320 + bits[0], gate_std=0.1)
    _check(mc, L)


def test_prefill_skewed_loads(mc):
    """Skewed routing: some experts get several full 128-pair blocks, some none."""
    L = synth.make_layer(700, 256, 384, 8, 128, [3, 3, 2, 2, 1, 2, 3, 1], 330, gate_std=0.05, skew=(3.0, 0.9))
    _check(mc, L)


def test_prefill_sixteen_experts(mc):
    L = synth.make_layer(400, 256, 256, 16, 64, [1, 2, 3] * 5 + [2], 340, gate_std=0.1, mu=0.5)
    _check(mc, L)


def test_automatic_switch_agrees_with_gemv(mc):
    """T = 256 (512 pairs; the GEMM from 240 pairs) takes the GEMM automatically;
    the GEMV path on the same inputs agrees with it and with the oracle."""
    L = synth.make_layer(256, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 350, gate_std=0.1, mu=0.3,
                         protect_frac=0.1)
    auto = _run(mc, L, 0)
    gemv = _run(mc, L, 1)
    ref, *_ = oracle_layer(L, oracle_mats(L))
    assert_close(auto, ref, "automatic path")
    assert_close(gemv, ref, "GEMV path")
    assert_close(auto, gemv.astype(np.float64), "automatic vs GEMV")


def test_prefill_mixtral_shape(mc):
    """Mixtral-8x7b-shaped prefill layer, 4096 tokens with skewed expert loads
    (the prefill workload), outputs checked on the tokens of every expert's
    first and last pair in its first and last (ragged) 128-pair token block,
    from the oracle's permutation, plus the first and last token."""
    L = synth.config_prefill(T=4096)
    tokens = sorted(set(boundary_tokens(L, 0.0, blocks=(128,)) + [0, L.T - 1]))
    assert len(tokens) >= 2 * L.E
    _check(mc, L, path=0, tokens=tokens)
