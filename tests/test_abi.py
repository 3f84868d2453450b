"""Host-side tests of the C-ABI library (no GPU): it loads, exports every symbol
include/mc.h declares, packs and unpacks bit-exactly, and rejects bad arguments
before touching the device."""
import ctypes
import os
import re

import numpy as np
import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def mc():
    from paper_2410_06270_gb300 import build
    build.build()
    import paper_2410_06270_gb300 as m
    m.load()
    return m


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "mc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mc_[a-z0-9_]+)\s*\(", src)))


def test_exports_every_declared_symbol(mc):
    names = _declared_functions()
    assert len(names) >= 15
    lib = ctypes.CDLL(mc.LIB_PATH)
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def _flat(L, attr):
    a = getattr(L, attr)
    return [a[e][m] for e in range(L.E) for m in range(3)]


@pytest.mark.parametrize("group,bits", [(64, [3, 2, 2, 1, 3, 2, 2, 3]), (128, [1, 2, 3, 1]),
                                        (128, [3, 3, 2, 2])])
def test_pack_unpack_round_trip(mc, group, bits):
    E = len(bits)
    L = synth.make_layer(4, 256, 384, E, group, bits, seed=21, zero_mode="fractional")
    shape = mc.Shape(E, L.H, L.F, group)
    packed = mc.pack_experts_host(shape, L.bits, _flat(L, "codes"), _flat(L, "scale"), _flat(L, "zero"))
    assert packed.nbytes == mc.packed_size(shape, L.bits)
    for e in range(E):
        for m in range(3):
            rows, cols = L.mat_shape(m)
            c, s, z = mc.unpack_experts_host(packed, e, m, rows, cols, group)
            np.testing.assert_array_equal(c, L.codes[e][m])
            np.testing.assert_array_equal(s.view(np.uint16), L.scale[e][m].view(np.uint16))
            np.testing.assert_array_equal(z.view(np.uint16), L.zero[e][m].view(np.uint16))


def test_packed_size_is_bits_plus_metadata(mc):
    # per weight: b bits + 4 bytes per group (fp16 scale + zero), plus header/padding
    E, H, F, g = 8, 4096, 14336, 128
    bits = [3, 3, 3, 3, 3, 2, 2, 1]
    n = mc.packed_size(mc.Shape(E, H, F, g), bits)
    want = sum(3 * H * F * b / 8 + 3 * H * F / g * 4 for b in bits)
    assert want <= n <= want + 4096 + 24 * 256


def test_pack_rejects_code_out_of_range(mc):
    L = synth.make_layer(2, 128, 128, 2, 64, [2, 3], seed=3)
    L.codes[0][1][5, 7] = 4  # > 2^2 - 1
    with pytest.raises(mc.MCError) as ei:
        mc.pack_experts_host(mc.Shape(2, 128, 128, 64), L.bits, _flat(L, "codes"), _flat(L, "scale"),
                             _flat(L, "zero"))
    assert ei.value.code == mc.ERR_INVALID_ARG
    assert "expert 0 matrix 1" in str(ei.value)


@pytest.mark.parametrize("shape,bits,code", [
    ((8, 4096, 14336, 32), [2] * 8, -1),      # group not 64/128
    ((8, 4000, 14336, 128), [2] * 8, -1),     # H not a multiple of 128
    ((8, 4096, 14300, 128), [2] * 8, -1),     # F not a multiple of 128
    ((17, 4096, 14336, 128), [2] * 17, -2),   # too many experts
    ((8, 4096, 14336, 128), [2, 2, 2, 4, 2, 2, 2, 2], -2),   # 4-bit expert
    ((8, 4096, 14336, 128), [2, 2, 2, 0, 2, 2, 2, 2], -2),
])
def test_bad_shapes_and_bits(mc, shape, bits, code):
    s = mc.Shape(*shape)
    b = np.asarray(bits, np.int8)
    assert mc.load().mc_packed_size(ctypes.byref(s), b.ctypes.data) == 0
    with pytest.raises(mc.MCError) as ei:
        mc.packed_size(s, b)
    ws = mc.load().mc_moe_forward(None, None, 4, ctypes.byref(s), b.ctypes.data, None, 0.0, None, None, None, 0,
                                  None, None, None, None)
    assert ws == code


def test_top_k_other_than_two_is_unsupported(mc):
    s = mc.Shape(8, 4096, 14336, 128, 1)
    assert mc.load().mc_moe_workspace_size(ctypes.byref(s), 4) == 0
    assert "top" in mc.last_error()


def test_forward_argument_checks_before_any_device_work(mc):
    lib = mc.load()
    s = mc.Shape(8, 256, 512, 64)
    b = np.asarray([3, 2, 2, 1, 3, 2, 2, 3], np.int8)
    fake = ctypes.c_void_p(0x100000)  # never dereferenced: validation fails first
    odd = ctypes.c_void_p(0x100008)
    # T < 0
    assert lib.mc_moe_forward(fake, fake, -1, ctypes.byref(s), b.ctypes.data, fake, 0.0, None, fake, fake, 1 << 30,
                              None, None, None, None) == mc.ERR_INVALID_ARG
    # T == 0 is a no-op
    assert lib.mc_moe_forward(None, None, 0, ctypes.byref(s), b.ctypes.data, None, 0.0, None, None, None, 0,
                              None, None, None, None) == mc.OK
    # NaN / negative / infinite mu
    for mu in (float("nan"), -0.5, float("inf")):
        assert lib.mc_moe_forward(fake, fake, 4, ctypes.byref(s), b.ctypes.data, fake, mu, None, fake, fake,
                                  1 << 30, None, None, None, None) == mc.ERR_INVALID_ARG
        assert "mu" in mc.last_error()
    # null pointers
    assert lib.mc_moe_forward(None, fake, 4, ctypes.byref(s), b.ctypes.data, fake, 0.0, None, fake, fake, 1 << 30,
                              None, None, None, None) == mc.ERR_INVALID_ARG
    # misaligned activations
    assert lib.mc_moe_forward(odd, fake, 4, ctypes.byref(s), b.ctypes.data, fake, 0.0, None, fake, fake, 1 << 30,
                              None, None, None, None) == mc.ERR_INVALID_ARG
    # short workspace
    need = mc.workspace_size(s, 4)
    assert lib.mc_moe_forward(fake, fake, 4, ctypes.byref(s), b.ctypes.data, fake, 0.0, None, fake, fake, need - 256,
                              None, None, None, None) == mc.ERR_INVALID_ARG
    assert "workspace" in mc.last_error()
    # route: same checks
    assert lib.mc_route(fake, fake, 4, ctypes.byref(s), float("nan"), None, fake, fake, fake, fake, fake,
                        None) == mc.ERR_INVALID_ARG


def test_unpack_host_rejects_corrupt_header(mc):
    L = synth.make_layer(2, 128, 128, 2, 64, [1, 2], seed=4)
    shape = mc.Shape(2, 128, 128, 64)
    packed = mc.pack_experts_host(shape, L.bits, _flat(L, "codes"), _flat(L, "scale"), _flat(L, "zero"))
    bad = packed.copy()
    bad[0] ^= 0xFF
    with pytest.raises(mc.MCError) as ei:
        mc.unpack_experts_host(bad, 0, 0, 128, 128, 64)
    assert ei.value.code == mc.ERR_BAD_PACK
    bad = packed.copy()
    bad[32 + 1] = 7  # header bits[1] = 7
    with pytest.raises(mc.MCError) as ei:
        mc.unpack_experts_host(bad, 1, 0, 128, 128, 64)
    assert ei.value.code == mc.ERR_BAD_PACK
    with pytest.raises(mc.MCError):
        mc.unpack_experts_host(packed[:100], 0, 0, 128, 128, 64)


def test_workspace_size_grows_with_tokens(mc):
    s = mc.Shape(8, 4096, 14336, 128)
    a, b = mc.workspace_size(s, 16), mc.workspace_size(s, 4096)
    assert 0 < a < b


def test_odp_threshold_host_matches_oracle():
    """mc_odp_threshold_host (host code, no GPU) against the oracle's quantile of
    w1/w0 over the prunable tokens."""
    import oracle
    import paper_2410_06270_gb300 as mc
    rng = np.random.default_rng(70)
    w0 = rng.uniform(0.5, 1.0, 200).astype(np.float32)
    w = np.stack([w0, (1 - w0)], axis=1).astype(np.float32)
    mask = np.zeros(200, np.uint8)
    mask[::9] = 1
    mask[3::17] = 2
    for q in (0.0, 0.15, 0.5, 1.0):
        assert mc.odp_threshold(w, mask, q) == pytest.approx(oracle.odp_threshold(w, mask, q), rel=1e-6)
    with pytest.raises(mc.MCError):
        mc.odp_threshold(w, np.ones(200, np.uint8), 0.5)


def test_fp16_expert_pack_round_trip_host():
    """16-bit experts: host pack then host unpack returns the fp16 weights; the
    tile bytes follow the documented lane / pair order (pure host code)."""
    import paper_2410_06270_gb300 as mc
    E, H, F = 2, 256, 384
    shape = mc.Shape(E, H, F, 128)
    rng = np.random.default_rng(71)
    mats = [rng.standard_normal((F, H) if m < 2 else (H, F)).astype(np.float16) for e in range(E) for m in range(3)]
    packed = mc.pack_experts_host(shape, [16] * E, mats, [None] * (3 * E), [None] * (3 * E))
    # header, then per expert the W1|W3 region and the W2 region, each 256-byte aligned
    assert packed.nbytes == 4096 + sum(2 * F * H * 2 + H * F * 2 for e in range(E))
    for e in range(E):
        for m in range(3):
            rows, cols = (F, H) if m < 2 else (H, F)
            out = np.empty((rows, cols), np.uint16)
            rc = mc.load().mc_unpack_experts_host(packed.ctypes.data, packed.nbytes, e, m, out.ctypes.data, None, None)
            assert rc == 0
            np.testing.assert_array_equal(out.view(np.float16), mats[3 * e + m])
    # first tile of expert 0's W1: lane 5 (g8 = 1, t = 1), pair j = 6 (k-step 1, rho 2)
    w1 = mats[0]
    tile = packed[4096:4096 + 4096].view(np.uint16)
    row, col = 1, 64 * 0 + 16 * 1 + 4 * 1 + 2 * 1
    assert tile[5 * 64 + 2 * 6] == w1[row, col].view(np.uint16)
    assert tile[5 * 64 + 2 * 6 + 1] == w1[row, col + 1].view(np.uint16)


def test_fp16_experts_cannot_mix_with_quantised():
    import paper_2410_06270_gb300 as mc
    with pytest.raises(mc.MCError) as ei:
        mc.packed_size(mc.Shape(8, 256, 256, 128), [16] * 7 + [3])
    assert "cannot be mixed" in str(ei.value)


def test_pmq_allocation_matches_oracle():
    """mc_expert_significance_host and mc_pmq_allocate (host code) against the
    oracle's counting and brute-force Eq. 4."""
    import oracle
    import paper_2410_06270_gb300 as mc
    rng = np.random.default_rng(72)
    T, E = 300, 8
    idx = np.stack([rng.integers(0, E, T), rng.integers(0, E, T)], axis=1).astype(np.int32)
    idx[:, 1] = (idx[:, 0] + 1 + rng.integers(0, E - 1, T)) % E
    w0 = rng.uniform(0.5, 1.0, T)
    w = np.stack([w0, 1 - w0], axis=1).astype(np.float32)
    pr = (rng.random(T) < 0.15).astype(np.uint8)
    pr[::37] = 2
    phi, wact = mc.expert_significance(idx, w, pr, E)
    ophi, owact = oracle.expert_significance(idx, w, pr, E)
    np.testing.assert_allclose(phi, ophi, rtol=1e-12)
    np.testing.assert_allclose(wact, owact, rtol=1e-6)
    for total, gamma in ((20, 2.0), (16, 2.0), (13, 1.0)):
        eps = np.sort(rng.uniform(0.1, 5.0, (E, 3)), axis=1)[:, ::-1]
        bits, obj = mc.pmq_allocate(phi, wact, eps, total, 1.0, 1.0, gamma)
        obits, oobj = oracle.pmq_allocate(phi, wact, eps, total, 1.0, 1.0, gamma)
        np.testing.assert_array_equal(bits, obits)
        assert obj == pytest.approx(oobj, rel=1e-12)
        assert bits.sum() == total and (bits == 3).any() and (bits == 2).any()
    with pytest.raises(mc.MCError):
        mc.pmq_allocate(phi, wact, eps, 25)


def test_set_path_accepts_only_the_two_paths(mc):
    """mc_set_path: 0 (automatic), 1 (GEMV), 2 (GEMM); any other value is
    rejected and leaves the choice unchanged (host code only)."""
    prev = mc.set_path(mc.PATH_GEMV)
    try:
        for bad in (-1, 3, 7):
            with pytest.raises(mc.MCError) as ei:
                mc.set_path(bad)
            assert ei.value.code == mc.ERR_INVALID_ARG
        assert mc.set_path(mc.PATH_GEMM) == mc.PATH_GEMV
        assert mc.set_path(mc.PATH_AUTO) == mc.PATH_GEMM
    finally:
        mc.set_path(prev)
