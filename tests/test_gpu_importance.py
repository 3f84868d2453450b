"""GPU parity of the token-importance producer (Sec. 2.3.2, Eq. 6) and the protect
mask it writes, against the CPU oracle: importance values within fp32 rounding of
the fp64 oracle; the mask bit-exact against the oracle's selection rule applied to
the GPU's own fp32 importances (the decision is taken in the kernel's precision)
and against the oracle's mask where the importances are well separated; ties,
empty and full masks, ragged L; the mask driving the ODP layer."""
import numpy as np
import pytest

import oracle
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


def _causal_softmax(nh, L, seed, temp=1.0):
    rng = np.random.default_rng(seed)
    s = rng.standard_normal((nh, L, L)) * temp
    s = np.where(np.tril(np.ones((L, L), bool))[None], s, -np.inf)
    e = np.exp(s - s.max(axis=2, keepdims=True))
    return (e / e.sum(axis=2, keepdims=True)).astype(np.float32)


def _tokens(L, H, seed):
    x = np.random.default_rng(seed).standard_normal((L, H)).astype(np.float32)
    xb = torch.from_numpy(x).to(torch.bfloat16)
    return xb.float().numpy().astype(np.float64), xb.cuda()


def _run(mc, L, H, nh, frac, seed, attn=None):
    t64, t = _tokens(L, H, seed)
    A = _causal_softmax(nh, L, seed + 1) if attn is None else attn
    imp, mask = mc.token_importance(t, torch.from_numpy(A).cuda(), frac)
    torch.cuda.synchronize()
    return t64, A, imp.cpu().numpy(), mask.cpu().numpy()


@pytest.mark.parametrize("L,H,nh,frac", [(300, 256, 4, 0.02), (300, 256, 4, 0.1), (1, 128, 2, 0.5),
                                         (33, 64, 1, 0.0), (33, 64, 1, 1.0), (2048, 128, 8, 0.02),
                                         (1024, 64, 2, 0.3), (1025, 64, 2, 0.3)])
def test_importance_and_mask(mc, L, H, nh, frac):
    t64, A, imp, mask = _run(mc, L, H, nh, frac, 500 + L + nh)
    ref, ref_mask = oracle.token_importance(t64, A.astype(np.float64), frac)
    np.testing.assert_allclose(imp, ref, rtol=2e-5, atol=1e-30)
    n = int(np.ceil(float(np.float32(frac)) * L - 1e-6))
    np.testing.assert_array_equal(mask, oracle.select_top(imp, n))
    # the importances are well separated here: the fp64 oracle picks the same tokens
    order = np.sort(ref)[::-1]
    if 0 < n < L and (order[n - 1] - order[n]) > 1e-4 * order[n - 1]:
        np.testing.assert_array_equal(mask, ref_mask)


def test_mask_ties_go_to_lower_indices(mc):
    """One-hot attention on key 0: every other token has importance 0, so the mask
    is token 0 then the lowest indices."""
    L = 97
    A = np.zeros((2, L, L), np.float32)
    A[:, :, 0] = 1.0
    t64, _, imp, mask = _run(mc, L, 64, 2, 0.05, 600, attn=A)
    assert imp[0] > 0 and (imp[1:] == 0).all()
    n = int(np.ceil(float(np.float32(0.05)) * L - 1e-6))
    assert np.flatnonzero(mask).tolist() == list(range(n))


def test_mask_drives_the_odp_layer(mc):
    """The produced mask protects its tokens in the ODP layer: routing bit-exact
    against the oracle with the same mask, outputs within the layer tolerance."""
    L = synth.make_layer(48, 256, 512, 8, 64, [3, 2, 2, 1, 3, 2, 2, 3], 610, gate_std=0.1, mu=0.6)
    x, g, _ = to_dev(L)
    A = _causal_softmax(4, L.T, 611)
    _, mask = mc.token_importance(x, torch.from_numpy(A).cuda(), 0.25)
    L.protect = mask.cpu().numpy()
    assert L.protect.sum() == 12
    condition_routing(L, L.mu)
    x, g, p = to_dev(L)
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    packed = mc.pack_experts(shape, L.bits, flat(L, "codes"), flat(L, "scale"), flat(L, "zero"))
    y, r = mc.moe_forward(x, g, shape, L.bits, packed, L.mu, p, routing=True)
    torch.cuda.synchronize()
    oidx, ow, opr = oracle.route(L.x_f32(), L.gate_f32(), L.mu, L.protect)
    np.testing.assert_array_equal(r["pruned"].cpu().numpy(), opr)
    assert not opr[L.protect == 1].any()
    ref, *_ = oracle_layer(L, oracle_mats(L))
    assert_close(y.float().cpu().numpy(), ref, "layer with the produced mask")


def test_invalid_arguments(mc):
    t = torch.zeros((4, 64), dtype=torch.bfloat16, device="cuda")
    A = torch.zeros((1, 4, 4), dtype=torch.float32, device="cuda")
    with pytest.raises(mc.MCError) as ei:
        mc.token_importance(t, A, 1.5)
    assert ei.value.code == mc.ERR_INVALID_ARG
