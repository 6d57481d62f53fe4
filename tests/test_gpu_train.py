"""Support maintenance on the GPU (Eq. support, Sec. 3.2; coverage regularizer,
Sec. 3.4) against the CPU oracle, through the C ABI.

TopK is integer work and must match bit for bit (indices and logits, in
deployment order); the coverage loss, the usage u and the gradient match
within a tolerance derived from fp32 exponentials (about 2 ulp each) summed
in double.
"""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")

# (C_in, R, k): the routing matrices of the benchmark layers, and small ones
SHAPES = [(64, 16, 4), (72, 9, 5), (256, 64, 16), (1024, 255, 64), (2048, 511, 128),
          (3072, 767, 32), (3072, 767, 384), (5, 3, 5), (1, 1, 1)]


def _logits(C, R, seed, ties=False):
    rng = np.random.default_rng(seed)
    L = rng.standard_normal((R, C)).astype(np.float32)
    if ties and C >= 8:
        L[:, 1::4] = L[:, 0::4][:, : L[:, 1::4].shape[1]]  # equal pairs
        L[0, :4] = [0.0, -0.0, 0.0, -0.0]                  # signed zeros tie
    return L


@pytest.fixture(scope="module")
def moce():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_23794_gb300 import build, moce as m
    build.build()
    return m


@pytest.mark.parametrize("C,R,k", SHAPES)
@pytest.mark.parametrize("ties", [False, True])
def test_topk_bit_exact(moce, C, R, k, ties):
    L = _logits(C, R, seed=C + R + k, ties=ties)
    idx, lg = moce.moce_topk_supports(torch.from_numpy(L).cuda(), k)
    ridx, rlg = oracle.topk(L, k)
    assert np.array_equal(idx.cpu().numpy(), ridx)
    assert np.array_equal(lg.cpu().numpy().view(np.uint32), rlg.view(np.uint32))


@pytest.mark.parametrize("C,k", [(300, 20), (2048, 128), (96, 96), (33, 1)])
@pytest.mark.parametrize("ties", [False, True])
def test_topk_many_rows_bit_exact(moce, C, k, ties):
    """9000 rows: the per-example row counts of the input-conditioned variant (one warp per
    row for k <= 128) against the oracle."""
    L = _logits(C, 9000, seed=C + k + 1, ties=ties)
    idx, lg = moce.moce_topk_supports(torch.from_numpy(L).cuda(), k)
    ridx, rlg = oracle.topk(L, k)
    assert np.array_equal(idx.cpu().numpy(), ridx)
    assert np.array_equal(lg.cpu().numpy().view(np.uint32), rlg.view(np.uint32))


def test_topk_output_is_already_packed(moce):
    C, R, k = 256, 64, 16
    L = _logits(C, R, seed=3, ties=True)
    idx, lg = moce.moce_topk_supports(torch.from_numpy(L).cuda(), k)
    packed = moce.moce_pack_supports(idx, lg, C)
    assert torch.equal(packed.packed_idx.view(R, k), idx)
    assert torch.equal(packed.packed_logits.view(R, k), lg)
    _, _, resid = oracle.pack(*oracle.topk(L, k), C)
    assert packed.n_resid == len(resid)
    assert np.array_equal(packed.resid_idx[: packed.n_resid].cpu().numpy(), resid)


def test_topk_rejects_non_finite(moce):
    L = _logits(64, 4, seed=1)
    L[2, 17] = np.nan
    with pytest.raises(moce.MoceError) as ei:
        moce.moce_topk_supports(torch.from_numpy(L).cuda(), 4)
    assert ei.value.status == moce.MOCE_ERR_BAD_SUPPORT


@pytest.mark.parametrize("C,R,k", SHAPES)
def test_coverage_matches_oracle(moce, C, R, k):
    L = (1.5 * _logits(C, R, seed=7 * C + R)).astype(np.float32)
    eps = 1e-8
    dL = torch.from_numpy(L).cuda()
    loss, u, g = moce.moce_coverage_loss(dL, eps)
    rloss, ru, rg = oracle.coverage(L, eps)
    assert float(loss.item()) == pytest.approx(rloss, rel=1e-4, abs=1e-7)
    np.testing.assert_allclose(u.cpu().numpy(), ru, rtol=2e-6, atol=1e-12)
    got = g.cpu().numpy().astype(np.float64)
    scale = max(np.abs(rg).max(), 1e-30)
    assert np.abs(got - rg).max() <= 1e-4 * scale + 1e-12
    # two calls give the same bits
    loss2, u2, g2 = moce.moce_coverage_loss(dL, eps)
    assert torch.equal(loss, loss2) and torch.equal(u, u2) and torch.equal(g, g2)


def test_coverage_uniform_rows_are_zero(moce):
    L = torch.full((33, 96), 0.25, dtype=torch.float32, device="cuda")
    loss, u, g = moce.moce_coverage_loss(L, 1e-8)
    assert abs(float(loss.item())) < 1e-9
    assert torch.allclose(u, torch.full_like(u, 1.0 / 96), rtol=1e-6, atol=0)
    assert float(g.abs().max().item()) < 1e-9


def test_coverage_without_gradient(moce):
    L = _logits(128, 12, seed=5)
    loss, u, g = moce.moce_coverage_loss(torch.from_numpy(L).cuda(), 1e-6, grad=False)
    assert g is None
    assert float(loss.item()) == pytest.approx(oracle.coverage(L, 1e-6, grad=False)[0], rel=1e-4)
