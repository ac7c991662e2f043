"""Fused LM-head + verify (asd_lmhead_verify, asd_lmhead_logits) against the fp64 oracle.

The tensor cores accumulate bf16 products in fp32, so the comparison follows
the stated tolerance: logits within 2e-2 (absolute) of the fp64 oracle, and
decisions (argmax, accepted length, committed and recovery tokens) bit-exact
wherever they are decided by a margin larger than the arithmetic can move:
a row's argmax where its top-2 gap exceeds 5e-2; a request's selection where
every row has such a gap, every mismatch has |r/q - g| > 5e-2 and every
budget test has |fl(s + C) - B| > 4e-2 per accumulated mismatch.
"""
import concurrent.futures as cf
import math

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu
LOGIT_TOL = 2e-2
MARGIN = 5e-2


def oracle_logits(hidden, weight, tokens, threads=16):
    """fp64 oracle logits of the given token rows (one thread per token; ctypes releases the GIL)."""
    h = hidden.cpu()
    w = weight.cpu()
    tokens = list(tokens)
    with cf.ThreadPoolExecutor(max_workers=threads) as pool:
        parts = list(pool.map(lambda t: oracle.lmhead_logits(h, w, np.array([t], np.int32)), tokens))
    z64 = np.concatenate([p[0] for p in parts])
    z32 = np.concatenate([p[1] for p in parts])
    return z64, z32


def top2_gap(z64):
    part = np.partition(z64, -2, axis=1)
    return part[:, -1] - part[:, -2]


def eligible(o, z64_req, K, gate, cap, budget, spent):
    """Is this request's selection decided by margins larger than the tolerance?

    Walks the oracle's selection (Alg. 1) position by position. Rows 0..a decide the outcome (their
    argmax fixes d_j and the recovery token), so each needs a top-2 gap above MARGIN; later rows cannot
    change it. At a mismatch, the cap test is exact (integers); the gate test |r/q - g| and the budget
    test |fl(s + C) - B| are robust when they clear MARGIN and 4e-2 per accumulated mismatch. A mismatch
    is decided when every test passes robustly (accepted) or one fails robustly or the cap fails
    (rejected; the other tests then do not matter)."""
    gaps = top2_gap(z64_req)
    y = o["row_argmax"]
    r = o["row_regret"]
    C, N = np.float32(0.0), 0
    for j in range(K + 1):
        if gaps[j] <= MARGIN:
            return False
        if j == K or o["draft"][j] == y[j]:
            if j == K:
                return True
            continue
        gq = float(r[j]) / (K - j)
        C_next = np.float32(C + r[j])
        N_next = N + 1
        s_next = float(np.float32(spent + C_next))
        gate_pass, gate_fail = gq < gate - MARGIN, gq > gate + MARGIN
        bud_pass, bud_fail = s_next < budget - 4e-2 * N_next, s_next > budget + 4e-2 * N_next
        cap_fail = N_next > cap
        if cap_fail or gate_fail or bud_fail:
            return True  # rejected here whatever the rounding: the prefix ends at j, decided
        if not (gate_pass and bud_pass):
            return False
        C, N = C_next, N_next
    return True


def compare(out, z64, z32, draft, tokens, B, K, gate, cap, budget, ledger=None):
    """Check the GPU outputs of the requests whose rows are `tokens` (whole requests) against the oracle;
    with `ledger` (the GPU's updated ledger, started at (budget, 0)) also its spent regret within the
    accumulated tolerance on the margin-decided requests."""
    K1 = K + 1
    reqs = sorted(set(t // K1 for t in tokens))
    g_top = out["row_top"].cpu().numpy().reshape(-1)
    g_arg = out["row_argmax"].cpu().numpy().reshape(-1)
    g_reg = out["row_regret"].cpu().numpy().reshape(B, K)
    g_acc = out["accepted_len"].cpu().numpy()
    g_com = out["committed"].cpu().numpy()
    g_rec = out["recovery"].cpu().numpy()
    x = draft.cpu().numpy()
    pos = {t: i for i, t in enumerate(tokens)}
    n_eligible = 0
    for b in reqs:
        rows = [pos[b * K1 + j] for j in range(K1)]
        zr32 = z32[rows][None]
        o = oracle.verify(zr32, x[b:b + 1], np.array([[budget, 0.0]], np.float32), gate, cap)
        o1 = {k: v[0] for k, v in o.items()}
        o1["draft"] = x[b]
        zmax = z64[rows].max(axis=1)
        assert np.all(np.abs(g_top[b * K1:(b + 1) * K1] - zmax) <= LOGIT_TOL), f"request {b}: top logit"
        gaps = top2_gap(z64[rows])
        decided = gaps > MARGIN
        assert np.array_equal(g_arg[b * K1:(b + 1) * K1][decided], o1["row_argmax"][decided]), f"request {b}: argmax"
        for j in range(K):
            if 0 <= x[b, j]:
                zx = z64[rows[j], x[b, j]]
                assert abs(g_reg[b, j] - (zmax[j] - zx)) <= 2 * LOGIT_TOL, f"request {b} row {j}: regret"
        if eligible(o1, z64[rows], K, gate, cap, budget, 0.0):
            n_eligible += 1
            assert g_acc[b] == o1["accepted_len"], f"request {b}: accepted length"
            assert np.array_equal(g_com[b], o1["committed"]), f"request {b}: committed"
            assert g_rec[b] == o1["recovery"], f"request {b}: recovery"
            if ledger is not None:
                spent = float(ledger[b, 1].item())
                assert abs(spent - float(o1["ledger"][1])) <= 2 * LOGIT_TOL * max(1, o1["accepted_len"]), \
                    f"request {b}: spent"
    return n_eligible, len(reqs)


@pytest.mark.parametrize("T,H,V", [(36, 512, 1000), (300, 136, 777), (130, 64, 256), (129, 5120, 2100),
                                   (5, 64, 1), (200, 72, 257), (15000, 64, 300)])
def test_lmhead_logits_match_fp64(asd, T, H, V):
    """Includes V = 1, a last 256-row vocabulary tile holding one row, and more token tiles (79) than
    SM pairs, so the grid runs in two waves."""
    g = torch.Generator(device="cuda").manual_seed(T * 7 + H + V)
    h = torch.randn(T, H, generator=g, device="cuda").to(torch.bfloat16)
    w = (0.02 * torch.randn(V, H, generator=g, device="cuda")).to(torch.bfloat16)
    z = asd.lmhead_logits(h, w)
    torch.cuda.synchronize()
    z64, _ = oracle_logits(h, w, range(T))
    err = np.abs(z.cpu().numpy().astype(np.float64) - z64)
    assert err.max() <= LOGIT_TOL, f"max |logit - fp64| = {err.max()}"
    assert err.max() <= 1e-3, f"fp32 accumulation should be far inside the tolerance: {err.max()}"


@pytest.mark.parametrize("B,K,H,V", [(4, 8, 512, 4096), (16, 7, 1024, 3000), (3, 0, 256, 999), (24, 8, 5120, 3000)])
def test_lmhead_verify_small(asd, B, K, H, V):
    inp = inputs.gen_lmhead(B, K, H, V, 4000 + B + K + H, "cuda")
    led = asd.make_ledger(B, 8.0)
    out = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, 1.0, 2)
    torch.cuda.synchronize()
    T = B * (K + 1)
    z64, z32 = oracle_logits(inp.hidden, inp.weight, range(T))
    n_ok, n = compare(out, z64, z32, inp.draft, list(range(T)), B, K, 1.0, 2, 8.0, ledger=led)
    print(f"\nmargin-decided requests {n_ok}/{n}")
    # small hidden sizes shrink the logit spread (0.02 sqrt(H)), so more rows sit within the margins than
    # at the workload's H = 5120, where the floor is 80 %
    floor = 0.8 if H >= 4096 else 0.6
    assert n_ok >= floor * n, f"too few requests decided by margin ({n_ok}/{n}); the workload is too tie-heavy"


def test_lmhead_strict_budget_zero_matches_argmax(asd):
    """Budget 0: the fused verify is exact greedy verification on its own argmaxes."""
    B, K, H, V = 8, 8, 512, 2048
    inp = inputs.gen_lmhead(B, K, H, V, 77, "cuda")
    led = asd.make_ledger(B, 0.0)
    out = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, 1.0, 2)
    torch.cuda.synchronize()
    y = out["row_argmax"].cpu().numpy()
    x = inp.draft.cpu().numpy()
    for b in range(B):
        a = next((j for j in range(K) if x[b, j] != y[b, j]), K)
        assert out["accepted_len"][b].item() == a
        assert out["recovery"][b].item() == y[b, a]
    assert torch.equal(led.cpu(), torch.zeros(B, 2))


def test_lmhead_full_size_every_row(asd):
    """B=64, K=8, H=5120, V=151936 (Qwen3-14B LM head shape), every one of the 576 rows against the fp64
    oracle: all 87.5 M logits within 2e-2 (asd_lmhead_logits, same main loop), every argmax-decided row
    (top-2 gap > 5e-2) equal, and every request whose selection is decided by margins equal bit for bit
    in accepted length, committed and recovery tokens; the decided fraction is reported and floored."""
    cfg = inputs.CONFIGS[4]
    B, K, H, V = cfg["B"], cfg["K"], cfg["H"], cfg["V"]
    gate, cap, budget = cfg["gate"], cfg["cap"], cfg["budget"]
    inp = inputs.gen_lmhead(B, K, H, V, inputs.seed_for(4), "cuda")
    led = asd.make_ledger(B, budget)
    ws = asd.lmhead_workspace(B, K, V, H)
    for _ in range(2):  # the second call reuses the workspace
        led.copy_(asd.make_ledger(B, budget))
        out = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, gate, cap, workspace=ws)
    z_gpu = asd.lmhead_logits(inp.hidden, inp.weight)
    torch.cuda.synchronize()
    assert ws.error() == 0
    T = B * (K + 1)
    z64 = oracle.lmhead_logits_matmul(inp.hidden.cpu(), inp.weight.cpu())
    err = np.abs(z_gpu.cpu().numpy().astype(np.float64) - z64).max()
    print(f"\nfull-size LM head: max |logit - fp64| = {err:.3e} over {T * V} logits")
    assert err <= LOGIT_TOL
    gaps = top2_gap(z64)
    decided_rows = gaps > MARGIN
    g_arg = out["row_argmax"].cpu().numpy().reshape(-1)
    assert np.array_equal(g_arg[decided_rows], z64.argmax(axis=1)[decided_rows])
    n_ok, n = compare(out, z64, z64.astype(np.float32), inp.draft, list(range(T)), B, K, gate, cap, budget,
                      ledger=led)
    print(f"argmax-decided rows {decided_rows.mean():.3f}; margin-decided requests {n_ok}/{n} = {n_ok / n:.3f}")
    assert decided_rows.mean() >= 0.95
    assert n_ok >= 0.8 * n, f"too few margin-decided requests: {n_ok}/{n}"


def test_lmhead_full_size_exact_inputs_bit_exact(asd):
    """B=64, K=8, H=5120, V=151936 on integer h and W (sums of at most 5120 unit products are exact in
    fp32, whatever the order): every output of the fused verify equals the oracle's bit for bit, ties
    across warps, SMs and SM pairs included."""
    cfg = inputs.CONFIGS[4]
    B, K, H, V = cfg["B"], cfg["K"], cfg["H"], cfg["V"]
    inp = inputs.gen_lmhead_exact(B, K, H, V, inputs.seed_for(4, 1), "cuda")
    ledger0 = torch.tensor([[cfg["budget"], 0.0]] * B, dtype=torch.float32)
    led = ledger0.cuda()
    out = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, cfg["gate"], cfg["cap"])
    torch.cuda.synchronize()
    z64 = oracle.lmhead_logits_matmul(inp.hidden.cpu(), inp.weight.cpu())
    z32 = z64.astype(np.float32)
    assert np.array_equal(z64, z32.astype(np.float64)), "integer inputs must give exact logits"
    o = oracle.verify(z32.reshape(B, K + 1, V), inp.draft.cpu().numpy(), ledger0.numpy(), cfg["gate"], cfg["cap"])
    for key in ("row_argmax", "accepted_len", "committed", "recovery", "status"):
        assert np.array_equal(out[key].cpu().numpy(), o[key]), key
    assert np.array_equal(out["row_top"].cpu().numpy().reshape(-1), z32.max(axis=1))
    assert np.array_equal(out["row_regret"].cpu().numpy().view(np.int32), o["row_regret"].view(np.int32))
    assert np.array_equal(led.cpu().numpy().view(np.int32), o["ledger"].view(np.int32))
    ties = int(((z32 == z32.max(axis=1, keepdims=True)).sum(axis=1) > 1).sum())
    assert ties > 0
    assert int((o["accepted_len"] > 0).sum()) > 0


@pytest.mark.parametrize("B,K,H,V", [(8, 8, 512, 1000), (40, 8, 256, 2100), (5, 0, 64, 777), (3, 16, 320, 1300),
                                     (1500, 9, 64, 300), (6, 8, 8, 1000), (7, 3, 40, 513)])
def test_lmhead_verify_exact_inputs_bit_exact(asd, B, K, H, V):
    """Integer h and W: the fp32 logits are exact, so every output equals the oracle's bit for bit,
    ties across warps, SMs and SM pairs included (lowest index wins)."""
    inp = inputs.gen_lmhead_exact(B, K, H, V, 7000 + B + K + H, "cuda")
    ledger0 = torch.tensor([[8.0, 0.0]] * B, dtype=torch.float32)
    led = ledger0.cuda()
    out = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, 1.0, 2)
    torch.cuda.synchronize()
    T = B * (K + 1)
    z64, z32 = oracle_logits(inp.hidden, inp.weight, range(T))
    assert np.array_equal(z64, z32.astype(np.float64)), "integer inputs must give exact logits"
    o = oracle.verify(z32.reshape(B, K + 1, V), inp.draft.cpu().numpy(), ledger0.numpy(), 1.0, 2)
    assert np.array_equal(out["row_argmax"].cpu().numpy(), o["row_argmax"])
    assert np.array_equal(out["row_top"].cpu().numpy(), z32.reshape(B, K + 1, V).max(axis=2))
    assert np.array_equal(out["row_regret"].cpu().numpy().view(np.int32), o["row_regret"].view(np.int32))
    assert np.array_equal(out["accepted_len"].cpu().numpy(), o["accepted_len"])
    assert np.array_equal(out["committed"].cpu().numpy(), o["committed"])
    assert np.array_equal(out["recovery"].cpu().numpy(), o["recovery"])
    assert np.array_equal(led.cpu().numpy().view(np.int32), o["ledger"].view(np.int32))
    assert np.array_equal(out["status"].cpu().numpy(), o["status"])
    # the planted copies do produce ties that the lowest index has to win
    zr = z32.reshape(T, V)
    ties = int(((zr == zr.max(axis=1, keepdims=True)).sum(axis=1) > 1).sum())
    assert ties > 0


def test_lmhead_verify_nan_row_flags_its_request(asd):
    """A NaN hidden state makes every logit of its row NaN: that request is flagged and left alone
    (a = 0, ledger unchanged); every other request matches the oracle exactly."""
    B, K, H, V = 6, 4, 128, 900
    inp = inputs.gen_lmhead_exact(B, K, H, V, 7100, "cuda")
    bad_row = 2 * (K + 1) + 3  # request 2, row 3
    hidden = inp.hidden.clone()
    hidden[bad_row, 5] = float("nan")
    ledger0 = torch.tensor([[8.0, 0.5]] * B, dtype=torch.float32)
    led = ledger0.cuda()
    out = asd.lmhead_verify(hidden, inp.weight, inp.draft, led, 1.0, 2)
    torch.cuda.synchronize()
    z64, z32 = oracle_logits(hidden, inp.weight, range(B * (K + 1)))
    assert np.isnan(z32[bad_row]).all()
    o = oracle.verify(z32.reshape(B, K + 1, V), inp.draft.cpu().numpy(), ledger0.numpy(), 1.0, 2)
    st = out["status"].cpu().numpy()
    assert st[2] & oracle.STATUS_NAN_LOGIT and o["status"][2] & oracle.STATUS_NAN_LOGIT
    assert out["accepted_len"][2].item() == 0
    assert np.array_equal(led.cpu().numpy()[2], ledger0.numpy()[2])
    for b in [0, 1, 3, 4, 5]:
        assert st[b] == o["status"][b] == 0
        assert out["accepted_len"][b].item() == o["accepted_len"][b]
        assert np.array_equal(out["committed"][b].cpu().numpy(), o["committed"][b])
        assert np.array_equal(led.cpu().numpy()[b].view(np.int32), o["ledger"][b].view(np.int32))


@pytest.mark.parametrize("B,K,H,V,bounds", [(8, 8, 256, 1000, (0, 300, 650, 1000)),
                                            (40, 8, 128, 2100, (0, 512, 1000, 1601, 2100)),
                                            (5, 0, 64, 777, (0, 129, 777)),
                                            (3, 16, 320, 1300, (0, 1, 1300))])
def test_lmhead_sharded_partials_combine_to_the_unsharded_verify(asd, B, K, H, V, bounds):
    """The fused LM-head per vocabulary shard (a tensor-parallel rank's share of W), its partials
    combined: every output equals the unsharded fused verify and the oracle, bit for bit (exact
    inputs), with shard edges inside 256-row tiles, a one-row shard, and ties across shards."""
    inp = inputs.gen_lmhead_exact(B, K, H, V, 7300 + B + K + H, "cuda")
    T = B * (K + 1)
    S = len(bounds) - 1
    parts = torch.empty(S, T, asd.PARTIAL_WORDS, dtype=torch.int32, device="cuda")
    for i in range(S):
        shard = inp.weight[bounds[i]:bounds[i + 1]].contiguous()
        asd.lmhead_partials(inp.hidden, shard, inp.draft, bounds[i], V, out=parts[i])
    led_s = asd.make_ledger(B, 8.0)
    sharded = asd.shard_combine(parts, inp.draft, led_s, 1.0, 2, V)
    led_u = asd.make_ledger(B, 8.0)
    whole = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led_u, 1.0, 2)
    torch.cuda.synchronize()
    for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
        assert np.array_equal(sharded[key].cpu().numpy(), whole[key].cpu().numpy()), key
    assert np.array_equal(sharded["row_regret"].cpu().numpy().view(np.int32),
                          whole["row_regret"].cpu().numpy().view(np.int32))
    assert np.array_equal(led_s.cpu().numpy().view(np.int32), led_u.cpu().numpy().view(np.int32))
    z64, z32 = oracle_logits(inp.hidden, inp.weight, range(T))
    o = oracle.verify(z32.reshape(B, K + 1, V), inp.draft.cpu().numpy(), np.array([[8.0, 0.0]] * B, np.float32),
                      1.0, 2)
    for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
        assert np.array_equal(sharded[key].cpu().numpy(), o[key]), f"oracle: {key}"
    assert np.array_equal(led_s.cpu().numpy().view(np.int32), o["ledger"].view(np.int32))


def test_lmhead_full_size_four_shards_equal_the_unsharded_verify(asd):
    """B=64, K=8, H=5120, V=151936 on integer h and W, the vocabulary cut into the four 37984-row shards
    of four tensor-parallel ranks (each shard ends inside a 512-row unit): the combined partials equal
    the unsharded fused verify bit for bit (that one equals the oracle on these inputs, above)."""
    cfg = inputs.CONFIGS[4]
    B, K, H, V = cfg["B"], cfg["K"], cfg["H"], cfg["V"]
    inp = inputs.gen_lmhead_exact(B, K, H, V, inputs.seed_for(4, 1), "cuda")
    T = B * (K + 1)
    S = 4
    bounds = [i * V // S for i in range(S + 1)]
    parts = torch.empty(S, T, asd.PARTIAL_WORDS, dtype=torch.int32, device="cuda")
    for i in range(S):
        shard = inp.weight[bounds[i]:bounds[i + 1]].contiguous()
        asd.lmhead_partials(inp.hidden, shard, inp.draft, bounds[i], V, out=parts[i])
        del shard
    led_s = asd.make_ledger(B, cfg["budget"])
    sharded = asd.shard_combine(parts, inp.draft, led_s, cfg["gate"], cfg["cap"], V)
    led_u = asd.make_ledger(B, cfg["budget"])
    whole = asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led_u, cfg["gate"], cfg["cap"])
    torch.cuda.synchronize()
    for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
        assert np.array_equal(sharded[key].cpu().numpy(), whole[key].cpu().numpy()), key
    assert np.array_equal(sharded["row_regret"].cpu().numpy().view(np.int32),
                          whole["row_regret"].cpu().numpy().view(np.int32))
    assert np.array_equal(led_s.cpu().numpy().view(np.int32), led_u.cpu().numpy().view(np.int32))
    # the winners are spread over the shards, so the combine had real work to do
    owner = np.searchsorted(np.array(bounds[1:]), whole["row_argmax"].cpu().numpy().reshape(-1), side="right")
    assert len(set(owner.tolist())) == S


def test_lmhead_verify_infinities_through_the_tensor_cores(asd):
    """A +inf weight: where h is +1 the row's logit is +inf (it wins), where h is -1 it is -inf, and
    0 x inf = NaN flags the request; every other output equals the fp64 oracle (IEEE on both sides)."""
    B, K, H, V = 6, 4, 64, 700
    inp = inputs.gen_lmhead_exact(B, K, H, V, 7500, "cuda")
    K1 = K + 1
    weight = inp.weight.clone()
    weight[5, 0] = float("inf")
    hidden = inp.hidden.clone()
    sign = torch.tensor([1.0, 1.0, -1.0, -1.0, -1.0, 1.0], device="cuda").repeat_interleave(K1)
    hidden[:, 0] = sign.to(torch.bfloat16)
    hidden[4 * K1 + 2, 0] = 0.0            # request 4, row 2: 0 x inf = NaN
    draft = inp.draft.clone()
    draft[0, 0] = 5                        # matches an +inf argmax (its regret is inf - inf = NaN, unused)
    ledger0 = np.array([[8.0, 0.0]] * B, np.float32)
    led = torch.from_numpy(ledger0).cuda()
    out = asd.lmhead_verify(hidden, weight, draft, led, 1.0, 2)
    torch.cuda.synchronize()
    T = B * K1
    z64, z32 = oracle_logits(hidden, weight, range(T))
    assert np.isposinf(z32[0, 5]) and np.isneginf(z32[2 * K1, 5]) and np.isnan(z32[4 * K1 + 2, 5])
    o = oracle.verify(z32.reshape(B, K1, V), draft.cpu().numpy(), ledger0, 1.0, 2)
    g = {k: v.cpu().numpy() for k, v in out.items()}
    assert np.array_equal(g["status"], o["status"])
    assert g["status"][4] & oracle.STATUS_NAN_LOGIT and g["accepted_len"][4] == 0
    ok = g["status"] == 0
    for key in ("accepted_len", "committed", "recovery", "row_argmax"):
        assert np.array_equal(g[key][ok], o[key][ok]), key
    assert np.all(g["row_argmax"][:2] == 5)
    a, b = g["row_regret"][ok], o["row_regret"][ok]
    assert np.array_equal(np.isnan(a), np.isnan(b))
    assert np.array_equal(a[~np.isnan(a)].view(np.int32), b[~np.isnan(b)].view(np.int32))
    assert np.array_equal(led.cpu().numpy().view(np.int32), o["ledger"].view(np.int32))
