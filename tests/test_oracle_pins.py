"""The oracle against the paper's fixed points (CPU only).

Each pin is written independently of the oracle (see oracle_pins.py). The last
test plants plausible mistakes in copies of the oracle's C source and checks
that at least one pin catches every one of them.
"""
import os
import subprocess
import tempfile

import numpy as np
import pytest

import oracle_pins as P
from oracle import oracle


def test_argmax_first_occurrence(oracle_lib):
    P.pin_argmax_vs_numpy(oracle_lib)


def test_regret_is_gather_difference(oracle_lib):
    P.pin_regret_vs_gather(oracle_lib)


def test_selection_equals_bruteforce_exhaustive(oracle_lib):
    P.pin_selection_bruteforce(oracle_lib, Ks=(1, 2, 3, 4, 5, 6, 8, 16, 31), exhaustive_max_k=8)


def test_zero_budget_reduces_to_strict(oracle_lib):
    P.pin_zero_budget_is_strict(oracle_lib)


def test_gate_and_budget_fp32_boundaries(oracle_lib):
    P.pin_gate_and_budget_boundaries(oracle_lib)


def test_fig1_worked_case(oracle_lib):
    P.pin_fig1(oracle_lib)


def test_cap_zero_reduces_to_strict(oracle_lib):
    P.pin_cap_zero_is_strict(oracle_lib)


def test_ledger_carries_over_blocks(oracle_lib):
    P.pin_carry_ledger(oracle_lib)


def test_status_flags(oracle_lib):
    P.pin_status_flags(oracle_lib)


def test_ledger_validity_table(oracle_lib):
    P.pin_ledger_validity(oracle_lib)


def test_lmhead_fp64_matches_numpy(oracle_lib):
    P.pin_lmhead_vs_numpy(oracle_lib)


def test_select_replays_verify(oracle_lib):
    P.pin_select_replays_verify(oracle_lib)


def test_opportunity_statistic_eq4(oracle_lib):
    P.pin_opportunity_eq4(oracle_lib)


def test_commit_advances_along_the_emitted_sequence(oracle_lib):
    P.pin_commit_fig1(oracle_lib)


def test_k_zero_emits_bonus_only(oracle_lib):
    """K = 0 (no draft tokens): a = 0 = K, and the only emitted token is the bonus y*_1."""
    z = np.zeros((3, 1, 5), np.float32)
    z[:, 0, 2] = 1.0
    res = oracle.verify(z, np.zeros((3, 0), np.int32), np.array([[4.0, 0.0]] * 3, np.float32), 1.0, 2)
    assert list(res["accepted_len"]) == [0, 0, 0]
    assert res["committed"].tolist() == [[2], [2], [2]]


def test_invariants_on_generated_blocks(oracle_lib):
    """Sec. 3.2-3.3 invariants on the synthetic generator's blocks (tiny workload, 16 blocks)."""
    import torch
    from paper_2608_03447_gb300 import inputs
    cfg = inputs.CONFIGS[0]
    B, K, V = cfg["B"], cfg["K"], cfg["V"]
    led = np.array([[cfg["budget"], 0.0]] * B, np.float32)
    seen_accept_beyond_strict = False
    for blk in range(cfg["blocks"]):
        block = inputs.gen_block(B, K, V, torch.float32, inputs.seed_for(0, 0, blk))
        z = block.logits.numpy()
        x = block.draft.numpy()
        res = oracle.verify(z, x, led, cfg["gate"], cfg["cap"], lib=oracle_lib)
        st = oracle.verify(z, x, None, strict=True, lib=oracle_lib)
        y = res["row_argmax"]
        r = res["row_regret"]
        for b in range(B):
            a = res["accepted_len"][b]
            d = x[b] != y[b, :K]
            assert res["ledger"][b, 1] <= led[b, 0], "s' <= B (Eq. 13)"
            assert a >= st["accepted_len"][b], "a_ASD >= a_strict when B > 0"
            seen_accept_beyond_strict |= a > st["accepted_len"][b]
            assert d[:a].sum() <= cfg["cap"], "N_a <= M (Eq. 10)"
            for j in range(a):
                if d[j]:
                    assert np.float32(r[b, j]) / np.float32(K - j) <= cfg["gate"], "gate (Eq. 11)"
                else:
                    assert r[b, j].view(np.uint32) == 0, "matched tokens carry no regret (Prop. 1)"
            if a < K:
                assert d[a], "the prefix can only stop at a mismatch"
            C = np.float32(0.0)
            for j in range(a):
                if d[j]:
                    C = np.float32(C + r[b, j])
            assert res["ledger"][b, 1] == np.float32(led[b, 1] + C), "s' = s + C_a (Eq. 13)"
            assert np.all(r[b] >= 0), "r >= 0 (Eq. 3)"
        led = res["ledger"]
    assert seen_accept_beyond_strict, "the workload should exercise accepted mismatches"


def test_monotone_in_controls(oracle_lib):
    """a does not decrease when g, M or the remaining budget grow (Eq. 9-11 only loosen)."""
    import torch
    from paper_2608_03447_gb300 import inputs
    block = inputs.gen_block(16, 8, 512, torch.float32, 4242)
    z, x = block.logits.numpy(), block.draft.numpy()
    prev = None
    for g in (0.0, 0.25, 0.5, 1.0, 2.0, np.inf):
        for M in (0, 1, 2, 4):
            for bud in (0.5, 2.0, 8.0, 32.0):
                led = np.array([[bud, 0.0]] * 16, np.float32)
                a = oracle.verify(z, x, led, g, M, lib=oracle_lib)["accepted_len"]
                for (g2, M2, bud2) in ((g, M, bud * 2), (g, M + 1, bud), (g * 2 if g else 0.25, M, bud)):
                    led2 = np.array([[bud2, 0.0]] * 16, np.float32)
                    a2 = oracle.verify(z, x, led2, g2, M2, lib=oracle_lib)["accepted_len"]
                    assert np.all(a2 >= a)


def test_resume_equals_one_run(oracle_lib):
    """16 blocks in one run == 2 x 8 blocks with the ledger round-tripped through a copy."""
    import torch
    from paper_2608_03447_gb300 import inputs
    blocks = []
    for blk in range(16):
        b = inputs.gen_block(4, 8, 256, torch.float32, inputs.seed_for(0, 3, blk))
        blocks.append((b.logits.numpy(), b.draft.numpy()))
    led0 = np.array([[4.0, 0.0]] * 4, np.float32)
    one = oracle.verify_blocks(blocks, led0, 1.0, 2, lib=oracle_lib)
    first = oracle.verify_blocks(blocks[:8], led0, 1.0, 2, lib=oracle_lib)
    saved = np.array(first[-1]["ledger"], copy=True)
    second = oracle.verify_blocks(blocks[8:], saved, 1.0, 2, lib=oracle_lib)
    for r1, r2 in zip(one, first + second):
        for key in r1:
            assert np.array_equal(r1[key], r2[key]), key


# Plausible mistakes; each must be caught by at least one pin.
MUTANTS = {
    "argmax ties pick the last index": ("if (z > best_value) {", "if (z >= best_value) {"),
    "argmax skips the last vocabulary entry": ("for (int v = 1; v < V; v++) {", "for (int v = 1; v < V - 1; v++) {"),
    "regret sign flipped": ("r[j] = z_top - z_draft;", "r[j] = z_draft - z_top;"),
    "q off by one": ("float q = (float)(K - j);", "float q = (float)(K - j + 1);"),
    "gate strict inequality": ("(r[j] / q) <= gate;", "(r[j] / q) < gate;"),
    "gate as multiplication r <= g q": ("(r[j] / q) <= gate;", "r[j] <= gate * q;"),
    "budget strict inequality": ("(spent + C_next) <= budget;", "(spent + C_next) < budget;"),
    "budget ignores spent": ("(spent + C_next) <= budget;", "C_next <= budget;"),
    "budget as C <= B - s": ("(spent + C_next) <= budget;", "C_next <= budget - spent;"),
    "cap strict inequality": ("int cap_ok = N_next <= cap;", "int cap_ok = N_next < cap;"),
    "cumulative regret not accumulated": ("float C_next = C + r[j];", "float C_next = r[j];"),
    "matches treated as exceptions": ("if (x[j] == y[j]) continue; /* d = 0 */", ""),
    "no zero-budget dispatch": ("} else if (strict || budget == 0.0f) {", "} else if (strict) {"),
    "ledger not updated": ("ledger_b[1] = spent + C; /* Eq. 13 */", ""),
    "recovery from the previous row": ("*recovery_b = y[a];", "*recovery_b = y[a > 0 ? a - 1 : 0];"),
    "committed keeps the mismatched draft": ("if (j < a) token = x[j];", "if (j <= a) token = x[j];"),
    "strict stops one late": ("if (x[j] != y[j]) return j;", "if (x[j] != y[j]) return j + 1;"),
    "lm-head accumulates in fp32": ("double acc = 0.0;", "float acc = 0.0f;"),
    "lm-head ignores the token list": ("h + (int64_t)tokens[t] * H;", "h + (int64_t)t * H;"),
    "opportunity counts the block end": ("int reusable = i + p[u] <= K;", "int reusable = i + p[u] <= K + 1;"),
    "opportunity strict tau": ("if (r[i - 1] <= tau[t]) num[t * np + u] += 1;", "if (r[i - 1] < tau[t]) num[t * np + u] += 1;"),
    "commit drops the recovery token": ("for (int j = 0; j <= a; j++) tokens", "for (int j = 0; j < a; j++) tokens"),
    "commit forgets the pending token": ("if (kv_len) kv_len[b] += pending + a;", "if (kv_len) kv_len[b] += a;"),
    "ledger check misses a NaN budget": ("if (budget != budget || spent != spent) return 1;",
                                          "if (spent != spent) return 1;"),
    "ledger check misses a NaN spent": ("if (budget != budget || spent != spent) return 1;",
                                         "if (budget != budget) return 1;"),
    "ledger check accepts a negative spent": ("if (budget < 0.0f || spent < 0.0f) return 1;",
                                               "if (budget < 0.0f) return 1;"),
    "bad ledger flagged but still selected": ("if (flags) {\n    a = 0;", "if (flags & ~ORC_STATUS_BAD_LEDGER) {\n    a = 0;"),
    "opportunity suffix starts at i": ("for (int l = i + 1; reusable && l <= i + p[u]; l++)", "for (int l = i; reusable && l < i + p[u]; l++)"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistakes(name, tmp_path):
    old, new = MUTANTS[name]
    with open(oracle.SOURCE) as f:
        src = f.read()
    assert src.count(old) == 1, f"mutation anchor not found exactly once: {old!r}"
    mutated = tmp_path / "mutant.c"
    mutated.write_text(src.replace(old, new))
    lib_path = str(tmp_path / "libmutant.so")
    oracle.compile_library(str(mutated), lib_path)
    lib = oracle.load_library(lib_path)
    failed = P.run_all(lib, quick=True)
    assert failed, f"no pin caught the planted mistake: {name}"


def test_lmhead_matmul_path_equals_the_loop(oracle_lib):
    """oracle.lmhead_logits_matmul (numpy float64 matmul over W in blocks of rows) evaluates the same fp64
    logits as the C loop, across block edges and on integer inputs exactly."""
    import torch
    rng = np.random.default_rng(21)
    T, H, V = 7, 200, 50
    h = torch.from_numpy(rng.normal(size=(T, H)).astype(np.float32)).to(torch.bfloat16)
    W = torch.from_numpy(rng.normal(scale=0.02, size=(V, H)).astype(np.float32)).to(torch.bfloat16)
    z64, _ = oracle.lmhead_logits(h, W, lib=oracle_lib)
    for block in (8, 13, 64):
        zm = oracle.lmhead_logits_matmul(h, W, v_block=block)
        assert np.max(np.abs(zm - z64)) <= 1e-12
    hi = torch.from_numpy(rng.integers(-1, 2, size=(T, H)).astype(np.float32)).to(torch.bfloat16)
    Wi = torch.from_numpy(rng.integers(-1, 2, size=(V, H)).astype(np.float32)).to(torch.bfloat16)
    assert np.array_equal(oracle.lmhead_logits_matmul(hi, Wi, v_block=16), oracle.lmhead_logits(hi, Wi, lib=oracle_lib)[0])
