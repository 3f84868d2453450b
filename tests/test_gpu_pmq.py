"""PMQ calibration through the library (Sec. 2.2, N3): eps_{i,j} of Sec. 2.2.2
measured with the library's kernels (`paper_2410_06270_gb300.pmq`) against the
oracle's definition (the whole layer with one expert quantised, against the
unquantised layer), and the Eq. 4 bit table they lead to."""
import numpy as np
import pytest

import oracle
import synth
from helpers import to_dev

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


@pytest.mark.parametrize("T", [48, 160])
def test_pmq_eps_and_allocation_match_the_oracle(mc, T):
    """A layer of H 256, F 512, 8 experts, group 64 with weights N(0, 0.02) and
    their 1/2/3-bit quantisations (round-to-nearest / sign rule); T calibration
    tokens (160: the experts' 2-expert layers take the GEMM path).  eps within
    4% of the oracle's (the library's layer outputs are bf16; the differences are
    5-60% of the expert outputs), and the library's bit table optimal within 2%
    under the oracle's eps."""
    from paper_2410_06270_gb300 import pmq
    H, F, E, g, seed = 256, 512, 8, 64, 77
    L = synth.make_layer(T, H, F, E, g, [2] * E, seed, gate_std=0.1, experts=False)
    dense, quant, dmats, qmats = [], [], [], []
    for e in range(E):
        ws = [synth.expert_weights_f32(seed, e, m, *L.mat_shape(m)).astype(np.float16) for m in range(3)]
        qs = [[synth.rtn_quantize(ws[m].astype(np.float32), j, g) for m in range(3)] for j in (1, 2, 3)]
        dense.append(ws)
        quant.append(qs)
        dmats.append([oracle.QMat(*L.mat_shape(m), g, 16, dense=ws[m].astype(np.float32)) for m in range(3)])
        qmats.append([[oracle.QMat(*L.mat_shape(m), g, j + 1, *qs[j][m]) for m in range(3)] for j in range(3)])
    shape = mc.Shape(E, H, F, g)
    x, gw, _ = to_dev(L)
    res = pmq.calibrate(x, gw, shape, dense, quant, bits_total=16)
    eps_o = oracle.expert_error(L.x_f32(), L.gate_f32(), dmats, qmats)
    print("[pmq] eps library / oracle:\n", np.round(res["eps"], 4), "\n", np.round(eps_o, 4))
    np.testing.assert_allclose(res["eps"], eps_o, rtol=4e-2, atol=1e-6)
    # significance from the library's routing equals the oracle's counting
    idx, w, pr = oracle.route(L.x_f32(), L.gate_f32(), 0.0)
    phi_o, wact_o = oracle.expert_significance(idx, w, pr, E)
    np.testing.assert_allclose(res["phi"], phi_o, rtol=1e-12)
    np.testing.assert_allclose(res["wact"], wact_o, rtol=1e-5)
    bits_o, obj_o = oracle.pmq_allocate(phi_o, wact_o, eps_o, 16)
    b = res["bits"]
    obj_lib_under_o = sum(phi_o[i] * wact_o[i] * eps_o[i][b[i] - 1] ** 2 for i in range(E))
    print("[pmq] bits library %s oracle %s; objective %.6g vs optimum %.6g" % (
        list(map(int, b)), list(map(int, bits_o)), obj_lib_under_o, obj_o))
    assert b.sum() == 16 and (b == 3).any() and (b == 2).any()
    assert obj_lib_under_o <= obj_o * 1.02
