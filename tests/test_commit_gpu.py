"""asd_commit (advance along the emitted sequence, Sec. 3.3) against the oracle, over a decode loop."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu


def test_decode_loop_history_and_cache_lengths(asd):
    """12 rounds: verify, then commit; histories and KV lengths equal the oracle's, overflow included."""
    B, K, V, max_tokens = 16, 8, 3000, 40
    led = asd.make_ledger(B, 4.0)
    led_o = np.array([[4.0, 0.0]] * B, np.float32)
    tokens = torch.full((B, max_tokens), -1, dtype=torch.int32, device="cuda")
    token_len = torch.zeros(B, dtype=torch.int32, device="cuda")
    kv_len = torch.arange(B, dtype=torch.int32, device="cuda") * 3
    status = torch.zeros(B, dtype=torch.int32, device="cuda")
    o_tok = tokens.cpu().numpy()
    o_tl = token_len.cpu().numpy()
    o_kv = kv_len.cpu().numpy()
    overflowed = np.zeros(B, bool)
    for rnd in range(12):
        blk = inputs.gen_block(B, K, V, torch.float32, 81_000 + rnd, "cuda")
        out = asd.verify(blk.logits, blk.draft, led, 1.0, 2)
        asd.commit(out["accepted_len"], out["committed"], 1, kv_len, tokens, token_len, status)
        v = oracle.verify(blk.logits.cpu(), blk.draft.cpu().numpy(), led_o, 1.0, 2)
        led_o = v["ledger"]
        c = oracle.commit(v["accepted_len"], v["committed"], 1, o_kv, o_tok, o_tl)
        o_tok, o_tl, o_kv = c["tokens"], c["token_len"], c["kv_len"]
        torch.cuda.synchronize()
        assert np.array_equal(status.cpu().numpy(), c["status"]), f"round {rnd}: status"
        assert np.array_equal(token_len.cpu().numpy(), o_tl), f"round {rnd}: token_len"
        assert np.array_equal(kv_len.cpu().numpy(), o_kv), f"round {rnd}: kv_len"
        assert np.array_equal(tokens.cpu().numpy(), o_tok), f"round {rnd}: history"
        overflowed |= c["status"] == asd.STATUS_OVERFLOW
    assert overflowed.any(), "the loop should reach the history's capacity"


def test_commit_without_history(asd):
    a = torch.tensor([0, 3, 8], dtype=torch.int32, device="cuda")
    committed = torch.zeros(3, 9, dtype=torch.int32, device="cuda")
    kv = torch.tensor([10, 20, 30], dtype=torch.int32, device="cuda")
    asd.commit(a, committed, 0, kv_len=kv)
    torch.cuda.synchronize()
    assert kv.tolist() == [10, 23, 38]
