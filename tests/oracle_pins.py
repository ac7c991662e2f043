"""Pins for the CPU oracle: checks against things other than the oracle itself.

Each check takes the oracle library handle, so the same battery runs against the
real oracle and against deliberately broken copies of it (see
test_oracle_pins.py::test_pins_catch_planted_mistakes).

What pins what:
  * argmax (Eq. 1, lowest index on ties): numpy.argmax and torch.argmax, both
    documented to return the first occurrence, on tie-heavy rows with -0/+0
    and -inf;
  * regret (Eq. 3): torch.gather of the fp32 row at the argmax and the draft;
  * selection (Eq. 9-12, Alg. 1): a brute force written from the feasibility
    definition in exact rational arithmetic (fractions.Fraction), over every
    t in 0..K, on exhaustively enumerated mismatch patterns with dyadic regrets
    (exact in fp32, so the fp32 oracle must agree bit for bit);
  * strict rule (Eq. 2) and zero-budget dispatch (Alg. 1): brute force of
    Eq. 2, on tie-heavy blocks where accepting r = 0 mismatches would differ;
  * fp32 gate and budget arithmetic: boundaries built with numpy float32
    division and addition (IEEE, correctly rounded) and one ulp below them;
  * the Fig. 1 worked case: the hand-derived fixture in tests/golden;
  * ledger validity (NaN or negative budget / spent, spent above the budget):
    a hand-written table of ledgers and whether each is valid;
  * fused LM-head logits: numpy float64 matmul.
"""
from __future__ import annotations

import json
import math
import os
from fractions import Fraction

import numpy as np

from oracle import oracle

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
INT32_MAX = 2**31 - 1


# ----------------------------------------------------------------------------- builders

def block_from_targets(y, x, r, V, top=10.0, background=0.0):
    """Logits [B, K+1, V] fp32 whose row argmaxes are y [B, K+1] and whose regrets are r.

    Row j holds `top` at y_j, `top - r_j` at a mismatched draft x_j, `background`
    elsewhere. Callers keep x_j > y_j on mismatches so that r_j = 0 ties resolve
    to y_j, and choose `top` so that top - (top - r_j) == r_j exactly.
    """
    y = np.asarray(y)
    B, K1 = y.shape
    z = np.full((B, K1, V), background, np.float32)
    for b in range(B):
        for j in range(K1):
            z[b, j, y[b, j]] = top
            if j < K1 - 1 and x[b][j] != y[b, j]:
                z[b, j, x[b][j]] = np.float32(top) - np.float32(r[b][j])
    return z


def random_pattern_block(rng, B, K, V, regret_grid):
    y = rng.integers(0, V // 2, size=(B, K + 1))
    x = y[:, :K].copy()
    r = np.zeros((B, K), np.float32)
    mism = rng.random((B, K)) < 0.5
    for b in range(B):
        for j in range(K):
            if mism[b, j]:
                x[b, j] = rng.integers(y[b, j] + 1, V)
                r[b, j] = rng.choice(regret_grid)
    return block_from_targets(y, x, r, V), x.astype(np.int32), y, r


# ----------------------------------------------------------------------------- brute forces

def brute_strict(x, y):
    """Eq. 2: the largest a with x_i = y*_i for every i <= a."""
    K = len(x)
    best = 0
    for a in range(K + 1):
        if all(x[i - 1] == y[i - 1] for i in range(1, a + 1)):
            best = a
    return best


def brute_asd(x, y, r, budget, spent, gate, cap):
    """Eq. 9-12 read literally in exact arithmetic; Alg. 1's zero-budget dispatch first.

    Returns (a, s') with s' a Fraction.
    """
    K = len(x)
    F = Fraction
    if budget == 0:
        return brute_strict(x, y), F(float(spent))
    best_t, best_C = 0, F(0)
    for t in range(K + 1):
        mismatches = [i for i in range(1, t + 1) if x[i - 1] != y[i - 1]]       # d_i = 1
        C_t = sum((F(float(r[i - 1])) for i in mismatches), F(0))                # Eq. 8
        N_t = len(mismatches)                                                    # Eq. 8
        budget_ok = math.isinf(budget) or C_t <= F(float(budget)) - F(float(spent))  # Eq. 9
        cap_ok = N_t <= cap                                                      # Eq. 10
        gate_ok = all(math.isinf(gate) or F(float(r[i - 1])) / (K - i + 1) <= F(float(gate))
                      for i in mismatches)                                       # Eq. 6, 11
        if budget_ok and cap_ok and gate_ok:                                     # Eq. 12: max feasible t
            best_t, best_C = t, C_t
    return best_t, F(float(spent)) + best_C


# ----------------------------------------------------------------------------- pins

def pin_argmax_vs_numpy(lib):
    rng = np.random.default_rng(11)
    palette = np.array([-np.inf, -2.0, -1.0, -0.0, 0.0, 1.0, 3.0], np.float32)
    for V in (1, 2, 7, 64, 1000):
        B, K = 3, 4
        z = rng.choice(palette, size=(B, K + 1, V)).astype(np.float32)
        z[0, 0, :] = -np.inf                       # all -inf: index 0
        if V > 1:
            z[1, 0, :] = 0.0
            z[1, 0, V - 1] = 5.0                   # maximum in the last slot
            z[2, 1, :] = -0.0
            z[2, 1, V // 2] = 0.0                  # -0 == +0: the first index wins
        x = rng.integers(0, V, size=(B, K)).astype(np.int32)
        res = oracle.verify(z, x, strict=True, lib=lib)
        assert np.array_equal(res["row_argmax"], np.argmax(z, axis=2)), "argmax != numpy.argmax"
        import torch
        t = torch.from_numpy(z)
        assert np.array_equal(res["row_argmax"], torch.argmax(t, dim=2).numpy()), "argmax != torch.argmax"
        # bf16: the oracle's widening must agree with torch's bf16 -> fp32 conversion
        tb = (t + torch.from_numpy(rng.normal(size=z.shape).astype(np.float32))).to(torch.bfloat16)
        res_b = oracle.verify(tb, x, strict=True, lib=lib)
        assert np.array_equal(res_b["row_argmax"], torch.argmax(tb.float(), dim=2).numpy())


def pin_regret_vs_gather(lib):
    import torch
    rng = np.random.default_rng(12)
    B, K, V = 5, 6, 300
    z = rng.normal(scale=3.0, size=(B, K + 1, V)).astype(np.float32)
    x = rng.integers(0, V, size=(B, K)).astype(np.int32)
    x[:, 0] = np.argmax(z[:, 0, :], axis=1)        # some matches: r must be +0 exactly
    res = oracle.verify(z, x, strict=True, lib=lib)
    t = torch.from_numpy(z[:, :K, :])
    ystar = torch.from_numpy(res["row_argmax"][:, :K].astype(np.int64))
    top = torch.gather(t, 2, ystar[:, :, None])[:, :, 0]
    drf = torch.gather(t, 2, torch.from_numpy(x.astype(np.int64))[:, :, None])[:, :, 0]
    expect = (top - drf).numpy()
    assert np.array_equal(res["row_regret"].view(np.uint32), expect.view(np.uint32)), "regret != gather difference"
    assert np.all(res["row_regret"][:, 0].view(np.uint32) == 0), "a matching draft must have r = +0"


def pin_selection_bruteforce(lib, Ks=(1, 2, 3, 4, 5, 6), exhaustive_max_k=6):
    """Every mismatch pattern for small K, dyadic regrets, a grid of controls."""
    rng = np.random.default_rng(13)
    V = 16
    regret_grid = np.array([0.0, 0.125, 0.25, 0.5, 0.75, 1.0, 1.5, 2.0, 3.0, 4.0], np.float32)
    controls = [(g, M, Bud, s)
                for g in (0.0, 0.125, 0.25, 1.0, math.inf)
                for M in (0, 1, 2, INT32_MAX)
                for (Bud, s) in ((0.0, 0.0), (0.5, 0.0), (2.0, 0.75), (4.0, 4.0), (8.0, 1.0), (math.inf, 3.0))]
    for K in Ks:
        if K <= exhaustive_max_k:  # every mismatch pattern
            pats = np.array([[(p >> j) & 1 for j in range(K)] for p in range(2 ** K)], bool)
        else:                      # random patterns over all K positions
            pats = rng.random((64, K)) < 0.4
        n_pat = pats.shape[0]
        B = n_pat
        y = rng.integers(0, V // 2, size=(B, K + 1))
        x = y[:, :K].copy()
        r = np.zeros((B, K), np.float32)
        for b in range(B):
            for j in range(K):
                if pats[b, j]:
                    x[b, j] = rng.integers(y[b, j] + 1, V)
                    r[b, j] = rng.choice(regret_grid)
        z = block_from_targets(y, x, r, V)
        x = x.astype(np.int32)
        for (g, M, Bud, s) in controls:
            led = np.tile(np.array([Bud, s], np.float32), (B, 1))
            res = oracle.verify(z, x, led, gate=g, cap=M, lib=lib)
            for b in range(B):
                a, s_new = brute_asd(x[b], y[b], r[b], Bud, s, g, M)
                assert res["accepted_len"][b] == a, (
                    f"K={K} pattern={pats[b].astype(int)} r={r[b]} (g,M,Bud,s)={(g, M, Bud, s)}: "
                    f"oracle a={res['accepted_len'][b]} brute a={a}")
                assert Fraction(float(res["ledger"][b, 1])) == s_new, "ledger != s + C_a (Eq. 13)"
                expect = [int(x[b, j]) if j < a else (int(y[b, a]) if j == a else -1) for j in range(K + 1)]
                assert list(res["committed"][b]) == expect, "committed tokens differ from Alg. 1's output"
                assert res["recovery"][b] == y[b, a]


def pin_zero_budget_is_strict(lib):
    """Alg. 1: at B = 0 the output is the exact greedy output, even with r = 0 ties."""
    rng = np.random.default_rng(14)
    B, K, V = 64, 8, 12
    y = rng.integers(0, V // 2, size=(B, K + 1))
    x = y[:, :K].copy()
    r = np.zeros((B, K), np.float32)            # every mismatch is an exact tie
    mism = rng.random((B, K)) < 0.4
    for b in range(B):
        for j in range(K):
            if mism[b, j]:
                x[b, j] = rng.integers(y[b, j] + 1, V)
    z = block_from_targets(y, x, r, V)
    x = x.astype(np.int32)
    led = np.zeros((B, 2), np.float32)
    res = oracle.verify(z, x, led, gate=math.inf, cap=INT32_MAX, lib=lib)
    strict = oracle.verify(z, x, None, strict=True, lib=lib)
    for b in range(B):
        assert res["accepted_len"][b] == brute_strict(x[b], y[b]), "zero budget must reduce to Eq. 2"
    for key in ("accepted_len", "committed", "recovery", "row_argmax"):
        assert np.array_equal(res[key], strict[key]), key
    assert np.array_equal(res["ledger"].view(np.uint32), led.view(np.uint32)), "zero budget must keep the state"


def pin_gate_and_budget_boundaries(lib):
    """fp32 gate r/q <= g and budget fl(s + C) <= B decided exactly at the boundary."""
    rng = np.random.default_rng(15)
    K, V = 6, 8
    for _ in range(200):
        j = int(rng.integers(0, K))
        r = np.float32(rng.uniform(0.01, 3.0))
        q = np.float32(K - j)                   # Eq. 6 with i = j + 1
        g_exact = np.float32(r / q)             # numpy float32 division: IEEE, correctly rounded
        s = np.float32(rng.uniform(0.0, 2.0))
        bud_exact = np.float32(s + r)
        y = np.zeros((1, K + 1), np.int64)
        x = np.zeros((1, K), np.int64)
        x[0, j] = 3
        rr = np.zeros((1, K), np.float32)
        rr[0, j] = r
        z = block_from_targets(y, x, rr, V, top=0.0, background=-1e30)  # 0 - (0 - r) == r
        xi = x.astype(np.int32)
        def run(g, bud):
            led = np.array([[bud, s]], np.float32)
            return oracle.verify(z, xi, led, gate=float(g), cap=INT32_MAX, lib=lib)
        below = lambda v: np.nextafter(np.float32(v), np.float32(-np.inf))
        assert run(g_exact, np.float32(100.0))["accepted_len"][0] == K
        assert run(below(g_exact), np.float32(100.0))["accepted_len"][0] == j
        ok = run(np.float32(1e9), bud_exact)
        assert ok["accepted_len"][0] == K
        assert ok["ledger"][0, 1] == bud_exact
        assert run(np.float32(1e9), below(bud_exact))["accepted_len"][0] == j


def pin_fig1(lib):
    with open(os.path.join(GOLDEN, "fig1_worked_case.json")) as f:
        golden = json.load(f)
    for case in golden["cases"]:
        K, V = case["K"], case["V"]
        z = np.zeros((1, K + 1, V), np.float32)
        for j, (ytok, xtok, rj) in enumerate(case["target_rows"]):
            z[0, j, ytok] = 10.0
            if xtok >= 0:
                z[0, j, xtok] = 10.0 - rj
        x = np.array([case["draft"]], np.int32)
        st = oracle.verify(z, x, None, strict=True, lib=lib)
        e = case["expect_strict"]
        assert st["accepted_len"][0] == e["accepted_len"], case["name"]
        assert list(st["committed"][0]) == e["committed"], case["name"]
        assert st["recovery"][0] == e["recovery"], case["name"]
        led = np.array([case["ledger"]], np.float32)
        res = oracle.verify(z, x, led, gate=case["gate"], cap=case["cap"], lib=lib)
        e = case["expect_asd"]
        assert res["accepted_len"][0] == e["accepted_len"], case["name"]
        assert list(res["committed"][0]) == e["committed"], case["name"]
        assert res["recovery"][0] == e["recovery"], case["name"]
        assert res["ledger"][0, 1] == np.float32(e["spent"]), case["name"]
        zero = oracle.verify(z, x, np.array([[0.0, 0.0]], np.float32), gate=case["gate"], cap=case["cap"], lib=lib)
        assert list(zero["committed"][0]) == case["expect_strict"]["committed"], case["name"]


def pin_cap_zero_is_strict(lib):
    rng = np.random.default_rng(16)
    B, K, V = 32, 8, 32
    z, x, y, r = random_pattern_block(rng, B, K, V, np.array([0.0, 0.25, 1.0], np.float32))
    led = np.tile(np.array([100.0, 0.0], np.float32), (B, 1))
    res = oracle.verify(z, x, led, gate=math.inf, cap=0, lib=lib)
    for b in range(B):
        assert res["accepted_len"][b] == brute_strict(x[b], y[b]), "M = 0 must reduce to Eq. 2"


def pin_carry_ledger(lib):
    """The ledger persists over blocks (Sec. 3.2, (B, s)): the budget binds across rounds."""
    rng = np.random.default_rng(17)
    B, K, V = 4, 4, 16
    led = np.array([[1.0, 0.0]] * B, np.float32)
    spent_exact = [Fraction(0)] * B
    for blk in range(6):
        z, x, y, r = random_pattern_block(rng, B, K, V, np.array([0.25, 0.5], np.float32))
        res = oracle.verify(z, x, led, gate=math.inf, cap=INT32_MAX, lib=lib)
        for b in range(B):
            a, s_new = brute_asd(x[b], y[b], r[b], 1.0, float(led[b, 1]), math.inf, INT32_MAX)
            assert res["accepted_len"][b] == a
            assert Fraction(float(res["ledger"][b, 1])) == s_new
            assert s_new <= 1
        led = res["ledger"]


def pin_status_flags(lib):
    B, K, V = 4, 3, 8
    z = np.zeros((B, K + 1, V), np.float32)
    z[:, :, 1] = 5.0
    x = np.ones((B, K), np.int32)
    x[1, 2] = V                                  # draft id out of range
    z[2, 1, 4] = np.nan                          # NaN logit
    led = np.array([[4.0, 0.0], [4.0, 0.0], [4.0, 0.0], [1.0, 2.0]], np.float32)  # spent > budget
    res = oracle.verify(z, x, led, gate=1.0, cap=2, lib=lib)
    assert list(res["status"]) == [0, oracle.STATUS_DRAFT_RANGE, oracle.STATUS_NAN_LOGIT, oracle.STATUS_BAD_LEDGER]
    assert list(res["accepted_len"]) == [K, 0, 0, 0]
    assert np.array_equal(res["ledger"][1:], led[1:])


# (budget, spent, valid): the ledger rule read from Sec. 3.2-3.3 (a budget is a
# non-negative amount, the spent regret a non-negative sum of regrets never above
# it, Eq. 13's invariant s <= B), written out case by case. A negative budget
# always comes with a negative spent or a spent above it, so that rule needs no
# test of its own; the table still lists such ledgers.
LEDGER_TABLE = [
    (4.0, 0.0, True),
    (4.0, 4.0, True),           # exhausted: still a valid ledger
    (4.0, -0.0, True),          # -0 is not below zero
    (-0.0, 0.0, True),          # zero budget (strict dispatch)
    (math.inf, 0.0, True),
    (math.inf, math.inf, True),
    (math.nan, 0.0, False),     # NaN budget
    (4.0, math.nan, False),     # NaN spent
    (math.nan, math.nan, False),
    (4.0, -1.0, False),         # negative spent
    (4.0, -math.inf, False),
    (-1.0, -2.0, False),        # negative budget (and spent)
    (-math.inf, -math.inf, False),
    (-1.0, 0.0, False),         # negative budget, spent above it
    (1.0, 2.0, False),          # spent above the budget
    (0.0, 1e-30, False),
]


def pin_ledger_validity(lib):
    """Each ledger of LEDGER_TABLE on a block whose drafts all match: a valid ledger accepts the
    whole block (a = K, bonus y*_K), an invalid one is flagged, accepts nothing, emits y*_0 and
    keeps its ledger bit for bit (NaN payloads included)."""
    B, K, V = len(LEDGER_TABLE), 3, 8
    z = np.zeros((B, K + 1, V), np.float32)
    y = (np.arange(B * (K + 1)).reshape(B, K + 1) % (V - 1)) + 1
    for b in range(B):
        for j in range(K + 1):
            z[b, j, y[b, j]] = 5.0
    x = y[:, :K].astype(np.int32)
    led = np.array([[bud, sp] for bud, sp, _ in LEDGER_TABLE], np.float32)
    res = oracle.verify(z, x, led, gate=1.0, cap=2, lib=lib)
    for b, (bud, sp, valid) in enumerate(LEDGER_TABLE):
        what = f"ledger ({bud}, {sp})"
        if valid:
            assert res["status"][b] == 0, what
            assert res["accepted_len"][b] == K, what
            assert res["recovery"][b] == y[b, K], what
            assert res["ledger"][b, 0] == led[b, 0] and res["ledger"][b, 1] == led[b, 1], what
        else:
            assert res["status"][b] == oracle.STATUS_BAD_LEDGER, what
            assert res["accepted_len"][b] == 0, what
            assert res["recovery"][b] == y[b, 0], what
            assert list(res["committed"][b]) == [y[b, 0]] + [-1] * K, what
            assert np.array_equal(res["ledger"][b].view(np.uint32), led[b].view(np.uint32)), what


def pin_lmhead_vs_numpy(lib):
    import torch
    rng = np.random.default_rng(18)
    T, H, V = 6, 96, 40
    h = torch.from_numpy(rng.normal(size=(T, H)).astype(np.float32)).to(torch.bfloat16)
    W = torch.from_numpy(rng.normal(scale=0.02, size=(V, H)).astype(np.float32)).to(torch.bfloat16)
    tokens = np.array([5, 0, 3], np.int32)
    z64, z32 = oracle.lmhead_logits(h, W, tokens, lib=lib)
    expect = h.double().numpy()[tokens] @ W.double().numpy().T
    assert np.max(np.abs(z64 - expect)) <= 1e-12, "fp64 logits != numpy float64 matmul"
    assert np.array_equal(z32, z64.astype(np.float32))


def pin_select_replays_verify(lib):
    """The selection-only entry on a strict run's row results == the full verify, for every control."""
    import torch
    from paper_2608_03447_gb300 import inputs
    block = inputs.gen_block(8, 6, 700, torch.float32, 777)
    z, x = block.logits.numpy(), block.draft.numpy()
    x[3, 2] = 700                                  # one out-of-range draft
    rows = oracle.verify(z, x, None, strict=True, lib=lib)
    for g, M, bud, s in ((1.0, 2, 4.0, 0.5), (0.25, 1, 8.0, 0.0), (math.inf, INT32_MAX, 0.0, 0.0), (2.0, 4, 1.0, 2.0)):
        led = np.array([[bud, s]] * 8, np.float32)
        full = oracle.verify(z, x, led, g, M, lib=lib)
        sel = oracle.select(x, rows["row_argmax"], rows["row_regret"], rows["status"], led, g, M, lib=lib)
        for key in ("accepted_len", "committed", "recovery", "status", "ledger"):
            assert np.array_equal(full[key], sel[key]), key


def pin_opportunity_eq4(lib):
    """Eq. 4 by explicit enumeration of the mismatch set M, and the Fig. 1 block by hand."""
    rng = np.random.default_rng(19)
    n, K = 200, 9
    y = rng.integers(0, 4, size=(n, K + 1)).astype(np.int32)
    x = y[:, :K].copy()
    flip = rng.random((n, K)) < 0.35
    x[flip] = (x[flip] + 1 + rng.integers(0, 3, size=flip.sum())) % 7
    r = rng.choice(np.array([0.0, 0.25, 0.5, 1.0, 3.0], np.float32), size=(n, K))
    status = (rng.random(n) < 0.1).astype(np.int32)
    taus, ps = [0.0, 0.5, 1.0, float("inf")], [0, 1, 2, 3, 9]
    num, den = oracle.opportunity(y, x, r, taus, ps, status=status, lib=lib)
    M = [(b, i) for b in range(n) if status[b] == 0 for i in range(1, K + 1) if x[b, i - 1] != y[b, i - 1]]
    assert den == len(M), "|M| is the number of mismatch positions"
    for ti, tau in enumerate(taus):
        for pi, pp in enumerate(ps):
            expect = sum(1 for (b, i) in M if r[b, i - 1] <= tau and i + pp <= K
                         and all(x[b, l - 1] == y[b, l - 1] for l in range(i + 1, i + pp + 1)))
            assert num[ti, pi] == expect, f"Eq. 4 count (tau={tau}, p={pp})"
    # Fig. 1 (K=4): one mismatch E (r = 0.5) at i = 1, then F and G match, X mismatches at i = 4
    yf = np.array([[1, 3, 4, 5, 7]], np.int32)
    xf = np.array([[2, 3, 4, 6]], np.int32)
    rf = np.array([[0.5, 0.0, 0.0, 3.0]], np.float32)
    num, den = oracle.opportunity(yf, xf, rf, [0.25, 1.0], [2, 3], lib=lib)
    assert den == 2
    assert num.tolist() == [[0, 0], [1, 0]], "E reuses F, G (p = 2) but not a third token"


def pin_commit_fig1(lib):
    """Sec. 3.3 on the Fig. 1 case: E, F, G accepted, H emitted; the cache keeps the pending token and E, F, G."""
    a = np.array([3, 0], np.int32)
    committed = np.array([[2, 3, 4, 5, -1], [1, -1, -1, -1, -1]], np.int32)   # ASD and strict outputs
    tokens = np.full((2, 8), -9, np.int32)
    tokens[0, :2] = [10, 11]
    res = oracle.commit(a, committed, 1, np.array([2, 5], np.int32), tokens, np.array([2, 0], np.int32), lib=lib)
    assert res["tokens"][0].tolist() == [10, 11, 2, 3, 4, 5, -9, -9], "E F G H appended after the history"
    assert res["tokens"][1].tolist() == [1, -9, -9, -9, -9, -9, -9, -9], "strict: only the recovery E'"
    assert res["token_len"].tolist() == [6, 1]
    assert res["kv_len"].tolist() == [2 + 1 + 3, 5 + 1 + 0]
    full = oracle.commit(a, committed, 0, np.array([0, 0], np.int32), np.zeros((2, 4), np.int32),
                         np.array([1, 4], np.int32), lib=lib)
    assert full["status"].tolist() == [8, 8] and full["token_len"].tolist() == [1, 4], "no room: nothing changes"


ALL_PINS = [pin_argmax_vs_numpy, pin_regret_vs_gather, pin_selection_bruteforce, pin_zero_budget_is_strict,
            pin_gate_and_budget_boundaries, pin_fig1, pin_cap_zero_is_strict, pin_carry_ledger,
            pin_status_flags, pin_ledger_validity, pin_lmhead_vs_numpy, pin_select_replays_verify, pin_opportunity_eq4,
            pin_commit_fig1]


def run_all(lib, quick=False):
    """Run every pin; return the names of those that failed."""
    failed = []
    for pin in ALL_PINS:
        try:
            if quick and pin is pin_selection_bruteforce:
                pin(lib, Ks=(1, 3, 5))
            else:
                pin(lib)
        except AssertionError:
            failed.append(pin.__name__)
    return failed
