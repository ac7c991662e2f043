"""Seeded random cases for the entry points beyond the single-block verify, each against the oracle:
multi-block verify (random block counts, shapes, controls, with and without resident inputs), the
vocabulary-sharded verify from logits (random shard cuts, combined), and the fused LM head on exactly
representable inputs (random B, K, H, V; unsharded, and per random shard cuts then combined), where every
output must be bit-exact."""
import math

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu
INT32_MAX = 2**31 - 1
KEYS = ("accepted_len", "committed", "recovery", "row_argmax", "status")


def _cuts(rng, V, S):
    """S contiguous shards of [0, V), each at least one entry (fewer if V < S)."""
    S = min(S, V)
    inner = sorted(rng.choice(np.arange(1, V), size=S - 1, replace=False).tolist()) if S > 1 else []
    return [0] + inner + [V]


def _same(a, b, what):
    for key in KEYS:
        assert np.array_equal(a[key], b[key]), f"{what}: {key}"
    assert np.array_equal(a["row_regret"].view(np.uint32), b["row_regret"].view(np.uint32)), f"{what}: row_regret"


@pytest.mark.parametrize("chunk", range(3))
def test_random_multi_block_calls(asd, chunk):
    rng = np.random.default_rng(40_000 + chunk)
    for i in range(12):
        nblk = int(rng.integers(1, 6))
        B = int(rng.choice([1, 3, 8, 33]))
        K = int(rng.choice([0, 1, 4, 8, 16, 31]))
        V = int(rng.choice([1, 9, 100, 1001, 8192, 20001]))
        dtype = torch.bfloat16 if rng.random() < 0.5 else torch.float32
        gate = float(rng.choice([0.0, 0.5, 1.0, math.inf]))
        cap = int(rng.choice([0, 1, 2, INT32_MAX]))
        budget = float(rng.choice([0.0, 1.0, 4.0, math.inf]))
        resident = bool(rng.random() < 0.5)
        bl = [inputs.gen_block(B, K, V, dtype, 41_000 + chunk * 100 + i * 8 + j, "cuda") for j in range(nblk)]
        logits = torch.stack([b.logits for b in bl]).contiguous()
        draft = torch.stack([b.draft for b in bl]).contiguous()
        led = asd.make_ledger(B, budget)
        out = asd.verify_blocks(logits, draft, led, gate, cap, resident=resident)
        torch.cuda.synchronize()
        what = f"blocks {chunk}/{i}: nblk={nblk} B={B} K={K} V={V} {str(dtype)[6:]} g={gate} M={cap} budget={budget}"
        orc = oracle.verify_blocks([(logits[j].cpu(), draft[j].cpu().numpy()) for j in range(nblk)],
                                   np.array([[budget, 0.0]] * B, np.float32), gate, cap)
        for j in range(nblk):
            g = {k: out[k][j].cpu().numpy() for k in KEYS + ("row_regret",)}
            _same(g, orc[j], f"{what} block {j}")
        assert np.array_equal(led.cpu().numpy().view(np.uint32), orc[-1]["ledger"].view(np.uint32)), what


@pytest.mark.parametrize("chunk", range(2))
def test_random_vocabulary_shards_from_logits(asd, chunk):
    rng = np.random.default_rng(42_000 + chunk)
    for i in range(10):
        B = int(rng.choice([1, 4, 17]))
        K = int(rng.choice([0, 3, 8, 31]))
        V = int(rng.choice([2, 50, 1000, 4097, 30001]))
        dtype = torch.bfloat16 if rng.random() < 0.5 else torch.float32
        S = int(rng.integers(1, 6))
        cuts = _cuts(rng, V, S)
        b = inputs.gen_block(B, K, V, dtype, 43_000 + chunk * 100 + i, "cuda")
        parts = torch.empty(len(cuts) - 1, B * (K + 1), asd.PARTIAL_WORDS, dtype=torch.int32, device="cuda")
        for s in range(len(cuts) - 1):
            shard = b.logits[:, :, cuts[s]:cuts[s + 1]].contiguous()
            asd.shard_partials(shard, b.draft, cuts[s], V, out=parts[s], resident=bool(rng.random() < 0.5))
        led = asd.make_ledger(B, 4.0)
        comb = asd.shard_combine(parts, b.draft, led, 1.0, 2, V)
        torch.cuda.synchronize()
        g = {k: v.cpu().numpy() for k, v in comb.items()}
        o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), np.array([[4.0, 0.0]] * B, np.float32), 1.0, 2)
        what = f"shards {chunk}/{i}: B={B} K={K} V={V} {str(dtype)[6:]} cuts={cuts}"
        _same(g, o, what)
        assert np.array_equal(led.cpu().numpy().view(np.uint32), o["ledger"].view(np.uint32)), what


@pytest.mark.parametrize("chunk", range(2))
def test_random_fused_lmhead_exact_inputs(asd, chunk):
    rng = np.random.default_rng(44_000 + chunk)
    for i in range(8):
        B = int(rng.choice([1, 2, 7, 21, 64]))
        K = int(rng.choice([0, 1, 5, 8, 16]))
        H = int(rng.choice([8, 64, 136, 512, 1032]))
        V = int(rng.choice([1, 255, 256, 257, 511, 512, 513, 700, 1025, 3001]))
        inp = inputs.gen_lmhead_exact(B, K, H, V, 45_000 + chunk * 100 + i, "cuda")
        led0 = np.array([[8.0, 0.0]] * B, np.float32)
        led = torch.from_numpy(led0.copy()).cuda()
        out = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, 1.0, 2)
        S = int(rng.integers(1, 5))
        cuts = _cuts(rng, V, S)
        T = B * (K + 1)
        parts = torch.empty(len(cuts) - 1, T, asd.PARTIAL_WORDS, dtype=torch.int32, device="cuda")
        for s in range(len(cuts) - 1):
            asd.lmhead_partials(inp.hidden, inp.weight[cuts[s]:cuts[s + 1]].contiguous(), inp.draft, cuts[s], V,
                                out=parts[s])
        led_s = torch.from_numpy(led0.copy()).cuda()
        comb = asd.shard_combine(parts, inp.draft, led_s, 1.0, 2, V)
        torch.cuda.synchronize()
        z64 = oracle.lmhead_logits_matmul(inp.hidden.cpu(), inp.weight.cpu())
        z32 = z64.astype(np.float32)
        assert np.array_equal(z64, z32.astype(np.float64))
        o = oracle.verify(z32.reshape(B, K + 1, V), inp.draft.cpu().numpy(), led0, 1.0, 2)
        what = f"lmhead {chunk}/{i}: B={B} K={K} H={H} V={V} cuts={cuts}"
        g = {k: v.cpu().numpy() for k, v in out.items()}
        _same(g, o, what)
        assert np.array_equal(g["row_top"].reshape(-1), z32.max(axis=1)), what
        assert np.array_equal(led.cpu().numpy().view(np.uint32), o["ledger"].view(np.uint32)), what
        gs = {k: v.cpu().numpy() for k, v in comb.items()}
        _same(gs, o, what + " sharded")
        assert np.array_equal(led_s.cpu().numpy().view(np.uint32), o["ledger"].view(np.uint32)), what + " sharded"
