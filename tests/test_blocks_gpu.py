"""asd_verify_blocks: several sequential blocks of the same requests in one launch.

Must equal, bit for bit, the same blocks verified by ordered asd_verify calls
(the ledger of Sec. 3.2 carried from block to block) and the oracle's
sequential run, through both streaming kernels.
"""
import math

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(params=["stream", "tma", "tma-fused"])
def kernel(request, asd):
    """tma-fused: the TMA row stage with the selection inside it (last CTA done)."""
    name = request.param
    asd.set_launch_options(path=name.split("-")[0], fused_select=name.endswith("fused"))
    yield name
    asd.reset_launch_options()


def _blocks(nblk, B, K, V, dtype, seed, mix=inputs.MIX_DEFAULT):
    bl = [inputs.gen_block(B, K, V, dtype, seed + i, "cuda", mix=mix) for i in range(nblk)]
    return torch.stack([b.logits for b in bl]).contiguous(), torch.stack([b.draft for b in bl]).contiguous()


CASES = [
    (16, 4, 8, 1024, torch.float32, 4.0, 1.0, 2),        # the tiny workload's 16 blocks
    (4, 32, 8, 151936, torch.bfloat16, 8.0, 1.0, 2),      # Qwen3-14B shape
    (3, 1, 31, 5000, torch.bfloat16, 2.0, 0.5, 3),
    (5, 7, 0, 33, torch.float32, 1.0, 1.0, 1),
    (6, 5, 4, 1001, torch.bfloat16, 0.5, math.inf, 2**31 - 1),
]


@pytest.mark.parametrize("resident", [False, True])
@pytest.mark.parametrize("case", CASES)
def test_blocks_equal_sequential_calls_and_oracle(asd, kernel, case, resident):
    nblk, B, K, V, dtype, budget, gate, cap = case
    logits, draft = _blocks(nblk, B, K, V, dtype, 31_000 + nblk * 100 + B)
    led_blk = asd.make_ledger(B, budget)
    out = asd.verify_blocks(logits, draft, led_blk, gate, cap, resident=resident)
    led_seq = asd.make_ledger(B, budget)
    ws = asd.Workspace(B, K, V, asd.BF16 if dtype == torch.bfloat16 else asd.F32)
    seq = [asd.verify(logits[i], draft[i], led_seq, gate, cap, workspace=ws, resident=resident) for i in range(nblk)]
    torch.cuda.synchronize()
    for i in range(nblk):
        for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
            assert torch.equal(out[key][i], seq[i][key]), f"block {i}: {key}"
        assert np.array_equal(out["row_regret"][i].cpu().numpy().view(np.uint32),
                              seq[i]["row_regret"].cpu().numpy().view(np.uint32)), f"block {i}: row_regret"
    assert np.array_equal(led_blk.cpu().numpy().view(np.uint32), led_seq.cpu().numpy().view(np.uint32))
    host = [(logits[i].cpu(), draft[i].cpu().numpy()) for i in range(nblk)]
    orc = oracle.verify_blocks(host, np.array([[budget, 0.0]] * B, np.float32), gate, cap)
    for i in range(nblk):
        assert np.array_equal(out["accepted_len"][i].cpu().numpy(), orc[i]["accepted_len"]), f"oracle block {i}"
        assert np.array_equal(out["committed"][i].cpu().numpy(), orc[i]["committed"]), f"oracle block {i}"
    assert np.array_equal(led_blk.cpu().numpy().view(np.uint32), orc[-1]["ledger"].view(np.uint32))


def test_blocks_budget_binds_across_blocks(asd):
    """A small budget is spent in early blocks; later blocks fall back to exact matches only."""
    nblk, B, K, V = 8, 16, 8, 4096
    logits, draft = _blocks(nblk, B, K, V, torch.float32, 555, mix=(0.5, 0.45))
    led = asd.make_ledger(B, 1.0)
    out = asd.verify_blocks(logits, draft, led, 4.0, 8)
    torch.cuda.synchronize()
    spent = led[:, 1].cpu().numpy()
    assert np.all(spent <= 1.0)
    assert np.any(spent > 0.0)


def test_zero_blocks_is_a_noop(asd):
    logits = torch.empty(0, 4, 9, 100, device="cuda")
    draft = torch.empty(0, 4, 8, dtype=torch.int32, device="cuda")
    led = asd.make_ledger(4, 1.0)
    before = led.clone()
    asd.verify_blocks(logits, draft, led, 1.0, 2)
    torch.cuda.synchronize()
    assert torch.equal(led, before)
