"""GPU parity of the ODP workload: a Mixtral-8x7b-shaped layer of 256 tokens with
10% of tokens protected by the importance surrogate and mu set to drop the
secondary expert of ~15% of the unprotected tokens (Eq. 5, Sec. 2.3.2), at the
three bit budgets (sum 20 / 16 / 13).  Routing, prune flags and the permutation
bit-exact on all tokens; outputs on sampled tokens (protected, pruned and kept
ones, and the edges of every expert's work chunks and token blocks) against the
oracle, on the automatic (GEMM) path and on the GEMV path."""
import numpy as np
import pytest

import oracle
import synth
from helpers import assert_close, boundary_tokens, condition_routing, flat, oracle_layer, oracle_mats, to_dev

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


def _odp_layer(bits_total):
    L = synth.config_odp(T=256, bits_total=bits_total)
    _, w, _ = oracle.route(L.x_f32(), L.gate_f32(), 0.0, L.protect)
    ratio = w[:, 1].astype(np.float64) / w[:, 0]
    L.mu = float(np.quantile(ratio[L.protect == 0], 0.15))
    condition_routing(L, L.mu)
    return L


@pytest.mark.parametrize("bits_total", [20, 16, 13])
def test_odp_layer(mc, bits_total):
    L = _odp_layer(bits_total)
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    packed = mc.pack_experts(shape, L.bits, flat(L, "codes"), flat(L, "scale"), flat(L, "zero"))
    x, g, p = to_dev(L)
    ws = mc.alloc_workspace(shape, L.T)
    oidx, ow, opr = oracle.route(L.x_f32(), L.gate_f32(), L.mu, L.protect)
    pruned = np.nonzero(opr)[0]
    prot = np.nonzero(L.protect)[0]
    kept = np.nonzero((opr == 0) & (L.protect == 0))[0]
    assert 0.05 * L.T < len(pruned) < 0.25 * L.T
    # protected, pruned and kept tokens, and the edges of every expert's 16-pair
    # GEMV chunks and 128-pair GEMM token blocks (from the oracle's permutation)
    tokens = sorted(set(pruned[:2].tolist() + prot[:2].tolist() + kept[:2].tolist() + boundary_tokens(L)))
    mats = oracle_mats(L)
    ref, *_ = oracle_layer(L, mats, tokens)
    for path in (0, 1):
        old = mc.set_path(path)
        try:
            y, r = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, workspace=ws, routing=True)
            mc.check_status(ws)
        finally:
            mc.set_path(old)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(r["idx"].cpu().numpy(), oidx)
        np.testing.assert_array_equal(r["pruned"].cpu().numpy(), opr)
        np.testing.assert_allclose(r["w"].cpu().numpy(), ow, rtol=2e-6, atol=2e-6)
        got = y.float().cpu().numpy()[tokens]
        assert_close(got, ref, "ODP bits sum %d path %d mu %.4g (%d pruned, %d protected)" % (
            bits_total, path, L.mu, len(pruned), len(prot)))
