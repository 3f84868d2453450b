"""The oracle against the hand-computed worked examples in
tests/golden/worked_examples.txt (Eq. 1 / Eq. 5 routing with protection and
drop, Eq. 2 dequantisation, Eq. 6 token importance and mask, Eq. 4 allocation).
CPU only."""
import os

import numpy as np
import pytest

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))


def _blocks():
    out, cur = {}, None
    with open(os.path.join(HERE, "golden", "worked_examples.txt")) as f:
        for raw in f:
            line = raw.split("#", 1)[0].strip()
            if not line:
                continue
            if line.startswith("[") and line.endswith("]"):
                cur = out.setdefault(line[1:-1], {})
                continue
            key, vals = line.split(":", 1)
            cur[key.strip()] = np.array([float(v) for v in vals.split()], np.float64)
    return out


G = _blocks()


def _route(mu, mask):
    g = G["route"]
    E, H = len(g["logits"]), 8
    x = np.zeros((1, H), np.float32)
    x[0, 0] = 1.0  # logits = column 0 of the gate
    wg = np.zeros((E, H), np.float32)
    wg[:, 0] = g["logits"]
    return oracle.route(x, wg, mu, np.array([mask], np.uint8))


def test_route_worked_example():
    g = G["route"]
    idx, w, pr = _route(float(g["mu_keep"][0]), 0)
    assert idx[0].tolist() == g["idx"].astype(int).tolist() and pr[0] == 0
    np.testing.assert_allclose(w[0], g["w_kept"], rtol=1e-6)
    idx, w, pr = _route(float(g["mu_prune"][0]), 0)
    assert pr[0] == 1 and w[0].tolist() == g["w_pruned"].tolist()
    idx, w, pr = _route(float(g["mu_prune"][0]), 1)  # protected: kept at the same mu
    assert pr[0] == 0
    np.testing.assert_allclose(w[0], g["w_kept"], rtol=1e-6)
    idx, w, pr = _route(float(g["mu_keep"][0]), 2)  # dropped
    assert pr[0] == 2 and w[0].tolist() == g["w_dropped"].tolist()


def test_dequant_worked_example():
    g = G["dequant"]
    codes = g["codes"].astype(np.uint8)[None, :]
    m = oracle.QMat(1, 4, 4, 2, codes, np.float16([[g["scale"][0]]]), np.float16([[g["zero"][0]]]))
    got = [oracle.weight(m, 0, k) for k in range(4)]
    assert got == g["weights"].tolist()
    assert oracle.dequant_f32(m)[0].tolist() == g["weights"].tolist()


@pytest.mark.parametrize("frac,key", [(1.0 / 3.0, "mask_third"), (0.5, "mask_half")])
def test_importance_worked_example(frac, key):
    g = G["importance"]
    A = g["attn"].reshape(1, 3, 3)
    t = g["tokens"].reshape(3, 2)
    imp, mask = oracle.token_importance(t, A, frac)
    np.testing.assert_allclose(imp, g["importance"], rtol=1e-15)
    assert mask.tolist() == g[key].astype(int).tolist()


def test_pmq_worked_example():
    g = G["pmq"]
    bits, obj = oracle.pmq_allocate(g["phi"], g["wact"], g["eps"].reshape(3, 3), int(g["budget"][0]))
    assert list(bits) == g["bits"].astype(int).tolist()
    assert obj == pytest.approx(g["objective"][0], rel=1e-12)
