"""The tensor-core (tcgen05) building blocks against a plain matrix product."""
import pytest

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
    return m


@pytest.mark.parametrize("a_in_tmem", [False, True])
@pytest.mark.parametrize("N,K", [(16, 64), (16, 128), (32, 256), (64, 128), (128, 64)])
def test_umma_tile_matches_matmul(mc, N, K, a_in_tmem):
    g = torch.Generator().manual_seed(N * 1000 + K)
    A = torch.randn(128, K, generator=g).half().cuda()
    B = torch.randn(N, K, generator=g).half().cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    D = mc.selftest_umma(A, B, st, a_in_tmem=a_in_tmem)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    ref = A.double() @ B.double().T
    err = (D.double() - ref).abs().max().item() / ref.abs().max().item()
    assert err < 1e-5, err


@pytest.mark.parametrize("a_in_tmem", [False, True])
def test_umma_integer_operands_exact(mc, a_in_tmem):
    """Small integers are exact in fp16 and fp32: the product must be exact."""
    g = torch.Generator().manual_seed(7)
    A = torch.randint(0, 8, (128, 128), generator=g).half().cuda()
    B = torch.randint(-4, 5, (16, 128), generator=g).half().cuda()
    D = mc.selftest_umma(A, B, a_in_tmem=a_in_tmem)
    torch.cuda.synchronize()
    assert torch.equal(D.cpu(), (A.float() @ B.float().T).cpu())
