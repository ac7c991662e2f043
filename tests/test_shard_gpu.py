"""Vocabulary-sharded verify (asd_shard_partials + asd_shard_combine), emulated on one GPU.

Each shard is a separate tensor holding a slice of the vocabulary, as a
tensor-parallel rank would; the combined result must equal the unsharded
asd_verify and the oracle bit for bit.
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


def run_sharded(asd, logits, draft, bounds, ledger, gate, cap, misalign=0, resident=False):
    V = logits.shape[-1]
    parts = []
    for lo, hi in zip(bounds[:-1], bounds[1:]):
        shard = logits[:, :, lo:hi]
        if misalign:
            flat = torch.empty(shard.numel() + misalign, dtype=shard.dtype, device=shard.device)
            buf = flat[misalign:].view(shard.shape)
            buf.copy_(shard)
            shard = buf
        else:
            shard = shard.contiguous()
        parts.append(asd.shard_partials(shard, draft, lo, V, resident=resident))
    return asd.shard_combine(torch.stack(parts).contiguous(), draft, ledger, gate, cap, V)


CASES = [
    (32, 8, 151936, torch.bfloat16, [0, 50000, 100000, 151936]),
    (4, 8, 1024, torch.float32, [0, 1, 500, 1023, 1024]),
    (6, 5, 1001, torch.bfloat16, [0, 250, 501, 751, 1001]),
    (3, 31, 7000, torch.float32, [0, 7000]),
    (5, 0, 300, torch.bfloat16, [0, 299, 300]),
]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("misalign", [0, 1])
def test_sharded_equals_unsharded_and_oracle(asd, kernel, case, misalign):
    B, K, V, dtype, bounds = case
    blk = inputs.gen_block(B, K, V, dtype, 20_000 + V + B, "cuda")
    draft = blk.draft.clone()
    if K > 1:
        draft[0, 1] = V + 3  # an out-of-range draft id
    led_s = asd.make_ledger(B, 4.0)
    led_u = asd.make_ledger(B, 4.0)
    # the misaligned shards also pass ASD_RESIDENT_INPUTS (their copies were made before the calls)
    sh = run_sharded(asd, blk.logits, draft, bounds, led_s, 1.0, 2, misalign, resident=bool(misalign))
    un = asd.verify(blk.logits, draft, led_u, 1.0, 2)
    torch.cuda.synchronize()
    for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
        assert torch.equal(sh[key], un[key]), key
    a = sh["row_regret"].cpu().numpy()
    b = un["row_regret"].cpu().numpy()
    assert np.array_equal(np.isnan(a), np.isnan(b))
    assert np.array_equal(a[~np.isnan(a)].view(np.uint32), b[~np.isnan(b)].view(np.uint32))
    assert np.array_equal(led_s.cpu().numpy().view(np.uint32), led_u.cpu().numpy().view(np.uint32))
    o = oracle.verify(blk.logits.cpu(), draft.cpu().numpy(), np.array([[4.0, 0.0]] * B, np.float32), 1.0, 2)
    assert np.array_equal(sh["committed"].cpu().numpy(), o["committed"])
    assert np.array_equal(sh["row_argmax"].cpu().numpy(), o["row_argmax"])


def test_sharded_ties_across_shards(asd, kernel):
    """Equal maxima in different shards: the lowest global index wins, as unsharded; zeros of both signs."""
    B, K, V = 4, 3, 600
    z = torch.full((B, K + 1, V), -5.0, device="cuda")
    z[:, :, 100] = 2.0
    z[:, :, 450] = 2.0          # same value in a later shard
    z[1, :, :] = -0.0
    z[1, :, 350] = 0.0          # +0 in shard 2, -0 everywhere else
    draft = torch.tensor([[450, 100, 7]] * B, dtype=torch.int32, device="cuda")
    led_s, led_u = asd.make_ledger(B, 1.0), asd.make_ledger(B, 1.0)
    sh = run_sharded(asd, z, draft, [0, 300, 600], led_s, math.inf, 2**31 - 1)
    un = asd.verify(z, draft, led_u, math.inf, 2**31 - 1)
    torch.cuda.synchronize()
    for key in ("accepted_len", "committed", "recovery", "row_argmax"):
        assert torch.equal(sh[key], un[key]), key
    assert np.array_equal(sh["row_regret"].cpu().numpy().view(np.uint32), un["row_regret"].cpu().numpy().view(np.uint32))
    assert sh["row_argmax"][0, 0].item() == 100


def test_shard_arguments_are_checked(asd):
    blk = inputs.gen_block(2, 2, 100, torch.float32, 3, "cuda")
    with pytest.raises(asd.AsdError):
        asd.shard_partials(blk.logits, blk.draft, 50, 120)  # shard past the end of the vocabulary
