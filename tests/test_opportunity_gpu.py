"""asd_opportunity (Eq. 4 counts) against the oracle: integer counts, bit-exact."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu
TAUS = [0.0, 0.25, 0.5, 1.0, 2.0, 4.0, float("inf")]
PS = [0, 1, 2, 3, 4, 8]


def test_opportunity_on_oracle_rows(asd):
    """The kernel on row outputs produced by the oracle (inputs from the oracle only)."""
    counts_orc = np.zeros((len(TAUS), len(PS)), np.int64)
    den_orc = 0
    counts = torch.zeros(len(TAUS) * len(PS) + 1, dtype=torch.int64, device="cuda")
    for blk in range(6):
        b = inputs.gen_block(64, 8, 3000, torch.float32, 70_000 + blk)
        rows = oracle.verify(b.logits, b.draft.numpy(), None, strict=True)
        num, den = oracle.opportunity(rows["row_argmax"], b.draft.numpy(), rows["row_regret"], TAUS, PS)
        counts_orc += num
        den_orc += den
        asd.opportunity(torch.from_numpy(rows["row_argmax"]).cuda(), b.draft.cuda(),
                        torch.from_numpy(rows["row_regret"]).cuda(), TAUS, PS, counts=counts)
    torch.cuda.synchronize()
    got = counts.cpu().numpy()
    assert got[-1] == den_orc
    assert np.array_equal(got[:-1].reshape(len(TAUS), len(PS)), counts_orc)


def test_opportunity_after_gpu_verify_matches_oracle_pipeline(asd):
    """asd_verify's row outputs fed to asd_opportunity, against oracle.verify + oracle.opportunity."""
    B, K, V = 32, 8, 151936
    blk = inputs.gen_block(B, K, V, torch.bfloat16, inputs.seed_for(1, 5, 0), "cuda")
    led = asd.make_ledger(B, 8.0)
    out = asd.verify(blk.logits, blk.draft, led, 1.0, 2)
    counts = asd.opportunity(out["row_argmax"], blk.draft, out["row_regret"], TAUS, PS, status=out["status"])
    torch.cuda.synchronize()
    rows = oracle.verify(blk.logits.cpu(), blk.draft.cpu().numpy(), None, strict=True)
    num, den = oracle.opportunity(rows["row_argmax"], blk.draft.cpu().numpy(), rows["row_regret"], TAUS, PS,
                                  status=rows["status"])
    got = counts.cpu().numpy()
    assert got[-1] == den and np.array_equal(got[:-1].reshape(num.shape), num)
    assert den > 0


@pytest.mark.parametrize("K", [1, 5, 31])
def test_opportunity_edge_k(asd, K):
    rng = np.random.default_rng(K)
    n = 1000
    y = rng.integers(0, 3, size=(n, K + 1)).astype(np.int32)
    x = np.where(rng.random((n, K)) < 0.6, y[:, :K], (y[:, :K] + 1) % 3).astype(np.int32)
    r = rng.choice(np.array([0.0, 0.25, 1.0, 3.0], np.float32), size=(n, K))
    status = (rng.random(n) < 0.05).astype(np.int32)
    num, den = oracle.opportunity(y, x, r, TAUS, PS + [31], status=status)
    counts = asd.opportunity(torch.from_numpy(y).cuda(), torch.from_numpy(x).cuda(), torch.from_numpy(r).cuda(),
                             TAUS, PS + [31], status=torch.from_numpy(status).cuda())
    torch.cuda.synchronize()
    got = counts.cpu().numpy()
    assert got[-1] == den and np.array_equal(got[:-1].reshape(num.shape), num)
