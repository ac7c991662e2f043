"""Seeded random cases against the oracle: shapes, dtypes, misaligned starts, controls (zero,
infinite, exhausted and invalid ledgers), out-of-range drafts, NaN logits, every row-stage kernel and
launch option, and one to three dependent calls carrying the ledger. Every output is compared bit for
bit as in tests/test_verify_gpu.py (requests flagged for a NaN logit on what is specified for them)."""
import math

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu
INT32_MAX = 2**31 - 1


def _np(out):
    return {k: v.cpu().numpy() for k, v in out.items()}


def _check(g, o, what):
    st = o["status"]
    assert np.array_equal(g["status"], st), f"{what}: status {g['status']} vs {st}"
    ok = (st & oracle.STATUS_NAN_LOGIT) == 0
    for key in ("accepted_len", "recovery", "committed", "row_argmax"):
        assert np.array_equal(g[key][ok], o[key][ok]), f"{what}: {key}"
    gr, orr = g["row_regret"][ok], o["row_regret"][ok]
    same = (gr.view(np.uint32) == orr.view(np.uint32)) | (np.isnan(gr) & np.isnan(orr))
    assert same.all(), f"{what}: row_regret"
    assert np.all(g["accepted_len"][~ok] == 0), f"{what}: flagged request accepted something"
    assert np.array_equal(g["ledger"].view(np.uint32), o["ledger"].view(np.uint32)), f"{what}: ledger"


def _case(rng, i):
    dtype = torch.bfloat16 if rng.random() < 0.6 else torch.float32
    B = int(rng.choice([1, 2, 3, 5, 8, 17, 32, 64]))
    K = int(rng.choice([0, 1, 2, 4, 7, 8, 15, 16, 31]))
    V = int(rng.choice([1, 2, 7, 8, 9, 63, 64, 65, 1000, 1024, 4097, 16384, 30001, 70001]))
    offset = int(rng.integers(0, 8))
    gate = float(rng.choice([0.0, 0.25, 1.0, 2.5, math.inf]))
    cap = int(rng.choice([0, 1, 2, 3, INT32_MAX]))
    budget = float(rng.choice([0.0, 0.5, 4.0, 8.0, math.inf]))
    path = str(rng.choice(["auto", "auto", "stream", "tma", "small"]))
    fused = bool(rng.random() < 0.25)
    pdl = bool(rng.random() < 0.8)
    resident = bool(rng.random() < 0.5)
    ncalls = int(rng.integers(1, 4))
    return dtype, B, K, V, offset, gate, cap, budget, path, fused, pdl, resident, ncalls


@pytest.mark.parametrize("chunk", range(6))
def test_random_cases_match_the_oracle(asd, chunk):
    rng = np.random.default_rng(20_000 + chunk)
    for i in range(50):
        dtype, B, K, V, offset, gate, cap, budget, path, fused, pdl, resident, ncalls = _case(rng, i)
        what = (f"case {chunk}/{i}: B={B} K={K} V={V} {str(dtype)[6:]} off={offset} g={gate} M={cap} "
                f"budget={budget} path={path} fused={fused} pdl={pdl} resident={resident}")
        # ledgers: mostly fresh, some spent, some exhausted, a few invalid
        led0 = np.array([[budget, 0.0]] * B, np.float32)
        for b in range(B):
            u = rng.random()
            if u < 0.15 and math.isfinite(budget):
                led0[b, 1] = budget                      # exhausted
            elif u < 0.25:
                led0[b] = rng.choice([[-1.0, 0.0], [np.nan, 0.0], [2.0, 3.0], [4.0, -0.5]])  # invalid
        ledger = torch.from_numpy(led0.copy()).cuda()
        led_orc = led0.copy()
        try:
            asd.set_launch_options(path=path, fused_select=fused, pdl=pdl)
            for call in range(ncalls):
                b = inputs.gen_block(B, K, V, dtype, 30_000 + chunk * 1000 + i * 10 + call, "cuda")
                draft = b.draft.clone()
                logits = b.logits
                if K > 0 and rng.random() < 0.2:
                    draft[int(rng.integers(0, B)), int(rng.integers(0, K))] = int(rng.choice([-1, V, V + 5]))
                if rng.random() < 0.15:
                    logits = logits.clone()
                    logits[int(rng.integers(0, B)), int(rng.integers(0, K + 1)), int(rng.integers(0, V))] = float("nan")
                flat = torch.empty(B * (K + 1) * V + offset, dtype=dtype, device="cuda")
                view = flat[offset:].view(B, K + 1, V)
                view.copy_(logits)
                out = asd.verify(view, draft, ledger, gate, cap, resident=resident)
                torch.cuda.synchronize()
                g = _np(out)
                g["ledger"] = ledger.cpu().numpy()
                o = oracle.verify(view.cpu(), draft.cpu().numpy(), led_orc, gate, cap)
                _check(g, o, f"{what} call {call}")
                led_orc = o["ledger"]
        finally:
            asd.reset_launch_options()
