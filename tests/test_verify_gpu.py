"""Parity of the CUDA verifier (asd_verify / asd_verify_strict) with the CPU oracle.

Bit-exact on every output: argmax indices, accepted lengths, committed and
recovery tokens, status words, and the fp32 regrets and ledgers (same fp32
operation order on both sides). Requests flagged for a NaN logit are compared
on what is specified for them (status, a = 0, ledger kept).
"""
import concurrent.futures as cf
import math

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu
INT32_MAX = 2**31 - 1


@pytest.fixture(params=["stream", "tma", "tma-fused", "small"])
def kernel(request, asd):
    """Runs the test through the register-streaming kernel, the TMA pipeline kernel (with its selection
    kernel, and with the selection inside the row stage) and the one-CTA-per-request kernel (shapes it
    does not take fall back to the default choice)."""
    name = request.param
    asd.set_launch_options(path=name.split("-")[0], fused_select=name.endswith("fused"))
    yield name
    asd.reset_launch_options()


def _np(out: dict) -> dict:
    return {k: v.cpu().numpy() for k, v in out.items()}


def gpu_verify(asd, logits, draft, ledger, gate, cap, strict=False, resident=False):
    if strict:
        out = asd.verify_strict(logits, draft, resident=resident)
    else:
        out = asd.verify(logits, draft, ledger, gate, cap, resident=resident)
    torch.cuda.synchronize()
    res = _np(out)
    if ledger is not None:
        res["ledger"] = ledger.cpu().numpy()
    return res


def assert_parity(gpu: dict, orc: dict, what: str = "", ledger: bool = True):
    st = orc["status"]
    assert np.array_equal(gpu["status"], st), f"{what}: status"
    ok = (st & oracle.STATUS_NAN_LOGIT) == 0   # NaN rows: the argmax is unspecified
    for key in ("accepted_len", "recovery"):
        assert np.array_equal(gpu[key][ok], orc[key][ok]), f"{what}: {key}"
    for key in ("committed", "row_argmax"):
        if key in gpu:
            diff = np.argwhere(gpu[key][ok] != orc[key][ok])
            assert diff.size == 0, f"{what}: {key} differs at {diff[:5].tolist()}"
    if "row_regret" in gpu:
        g, o = gpu["row_regret"][ok], orc["row_regret"][ok]
        same = (g.view(np.uint32) == o.view(np.uint32)) | (np.isnan(g) & np.isnan(o))
        assert same.all(), f"{what}: row_regret differs at {np.argwhere(~same)[:5].tolist()}"
    assert np.array_equal(gpu["accepted_len"][~ok], np.zeros((~ok).sum(), np.int32))
    if ledger:
        assert np.array_equal(gpu["ledger"].view(np.uint32), orc["ledger"].view(np.uint32)), f"{what}: ledger"


def run_sequence(asd, B, K, V, dtype, blocks, gate, cap, budget, config, mix=inputs.MIX_DEFAULT, point=0,
                 resident=False):
    """Sequential blocks on the same requests; the GPU carries its ledger on the device."""
    led_gpu = asd.make_ledger(B, budget)
    led_orc = np.array([[budget, 0.0]] * B, np.float32)
    for blk in blocks:
        b = inputs.gen_block(B, K, V, dtype, inputs.seed_for(config, point, blk), "cuda", mix=mix)
        g = gpu_verify(asd, b.logits, b.draft, led_gpu, gate, cap, resident=resident)
        o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), led_orc, gate, cap)
        assert_parity(g, o, f"config {config} block {blk}")
        led_orc = o["ledger"]
        # strict entry on the same block
        gs = gpu_verify(asd, b.logits, b.draft, None, 0, 0, strict=True, resident=resident)
        os_ = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), None, strict=True)
        assert_parity(gs, os_, f"config {config} block {blk} strict", ledger=False)
    return led_orc


@pytest.mark.parametrize("resident", [False, True])
def test_tiny_fp32_sixteen_blocks(asd, kernel, resident):
    """Sixteen dependent calls (each reads the ledger the previous one wrote), with and without
    ASD_RESIDENT_INPUTS: the early start of a call never reads the ledger early."""
    cfg = inputs.CONFIGS[0]
    led = run_sequence(asd, cfg["B"], cfg["K"], cfg["V"], cfg["dtype"], range(cfg["blocks"]),
                       cfg["gate"], cfg["cap"], cfg["budget"], 0, resident=resident)
    assert np.all(led[:, 1] <= cfg["budget"])


def test_tiny_zero_budget_is_strict(asd, kernel):
    cfg = inputs.CONFIGS[0]
    B, K, V = cfg["B"], cfg["K"], cfg["V"]
    for blk in range(cfg["blocks"]):
        b = inputs.gen_block(B, K, V, cfg["dtype"], inputs.seed_for(0, 1, blk), "cuda")
        led = asd.make_ledger(B, 0.0)
        g = gpu_verify(asd, b.logits, b.draft, led, cfg["gate"], cfg["cap"])
        s = gpu_verify(asd, b.logits, b.draft, None, 0, 0, strict=True)
        for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
            assert np.array_equal(g[key], s[key]), key
        assert np.array_equal(g["ledger"], np.zeros((B, 2), np.float32))


@pytest.mark.parametrize("resident", [False, True])
def test_qwen3_shape_bf16_blocks(asd, kernel, resident):
    cfg = inputs.CONFIGS[1]
    run_sequence(asd, cfg["B"], cfg["K"], cfg["V"], cfg["dtype"], range(8), cfg["gate"], cfg["cap"],
                 cfg["budget"], 1, resident=resident)


def test_budget_cap_sweep(asd):
    """B=128, K=16, V=151936 bf16: 64 control points x 16 sequential blocks, ledger reset per point."""
    cfg = inputs.CONFIGS[2]
    B, K, V = cfg["B"], cfg["K"], cfg["V"]
    nblocks = cfg["blocks"]
    blocks, rows = [], []
    for blk in range(nblocks):
        b = inputs.gen_block(B, K, V, cfg["dtype"], inputs.seed_for(2, 0, blk), "cuda")
        blocks.append(b)
        rows.append(oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), None, strict=True))
    for g in cfg["gates"]:
        for M in cfg["caps"]:
            for bud in cfg["budgets"]:
                led_gpu = asd.make_ledger(B, bud)
                led_orc = np.array([[bud, 0.0]] * B, np.float32)
                for blk in range(nblocks):
                    b, r = blocks[blk], rows[blk]
                    out = gpu_verify(asd, b.logits, b.draft, led_gpu, g, M)
                    o = oracle.select(b.draft.cpu().numpy(), r["row_argmax"], r["row_regret"], r["status"],
                                      led_orc, g, M)
                    o["row_argmax"], o["row_regret"] = r["row_argmax"], r["row_regret"]
                    assert_parity(out, o, f"g={g} M={M} B={bud} block {blk}")
                    led_orc = o["ledger"]
                    if bud == 0.0:
                        assert np.array_equal(out["committed"], r["committed"]), "budget 0 != strict"


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_ragged_shapes(asd, kernel, dtype):
    rng = np.random.default_rng(5)
    for V in (1, 2, 3, 7, 8, 9, 33, 1000, 1001, 4097, 70001):
        for K in (0, 1, 5, 31):
            for B in (1, 3):
                b = inputs.gen_block(B, K, V, dtype, 10_000 + V * 64 + K * 4 + B, "cuda")
                budget = float(rng.choice([0.0, 0.5, 4.0, math.inf]))
                led = asd.make_ledger(B, budget)
                g = gpu_verify(asd, b.logits, b.draft, led, 1.0, 2)
                o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), np.array([[budget, 0.0]] * B, np.float32),
                                  1.0, 2)
                assert_parity(g, o, f"B={B} K={K} V={V}")


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_misaligned_logits(asd, kernel, dtype):
    B, K, V = 3, 4, 1003
    for offset in range(1, 9):
        flat = torch.empty(B * (K + 1) * V + offset, dtype=dtype, device="cuda")
        b = inputs.gen_block(B, K, V, dtype, 777 + offset, "cuda")
        view = flat[offset:].view(B, K + 1, V)
        view.copy_(b.logits)
        led = asd.make_ledger(B, 4.0)
        g = gpu_verify(asd, view, b.draft, led, 1.0, 2)
        o = oracle.verify(view.cpu(), b.draft.cpu().numpy(), np.array([[4.0, 0.0]] * B, np.float32), 1.0, 2)
        assert_parity(g, o, f"offset {offset}")


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_ties_zeros_and_infinities(asd, kernel, dtype):
    rng = np.random.default_rng(6)
    palette = np.array([-np.inf, -2.0, -0.0, 0.0, 1.5], np.float32)
    B, K = 6, 7
    for V in (5, 64, 999, 20000):
        z = rng.choice(palette, size=(B, K + 1, V)).astype(np.float32)
        z[0, :, :] = -np.inf                 # whole request at -inf: y* = 0 everywhere
        z[1, :, :] = -0.0
        z[1, :, V // 2:] = 0.0               # zeros of both signs: the first index wins
        z[2, :, :] = 1.5                     # all equal
        x = rng.integers(0, V, size=(B, K)).astype(np.int32)
        x[3, :] = 0
        t = torch.from_numpy(z).to(dtype).cuda()
        xt = torch.from_numpy(x).cuda()
        for budget in (0.0, 3.0):
            led = asd.make_ledger(B, budget)
            g = gpu_verify(asd, t, xt, led, math.inf, INT32_MAX)
            o = oracle.verify(t.cpu(), x, np.array([[budget, 0.0]] * B, np.float32), math.inf, INT32_MAX)
            assert_parity(g, o, f"V={V} budget={budget}")


def test_status_flags(asd, kernel):
    B, K, V = 6, 5, 3000
    b = inputs.gen_block(B, K, V, torch.bfloat16, 99, "cuda")
    logits, draft = b.logits.clone(), b.draft.clone()
    draft[1, 3] = V            # out of range
    draft[2, 0] = -4           # out of range
    logits[3, 2, 1234] = float("nan")
    led = asd.make_ledger(B, 4.0)
    led[4] = torch.tensor([1.0, 2.0])          # spent > budget
    led[5] = torch.tensor([float("nan"), 0.0])
    led_before = led.cpu().numpy()
    g = gpu_verify(asd, logits, draft, led, 1.0, 2)
    o = oracle.verify(logits.cpu(), draft.cpu().numpy(), led_before, 1.0, 2)
    assert list(g["status"]) == [0, 1, 1, 2, 4, 4]
    assert_parity(g, o, "flags")
    assert np.array_equal(g["ledger"][1:].view(np.uint32), led_before[1:].view(np.uint32))


def test_ledger_validity_table(asd, kernel):
    """Every ledger of the oracle pin's hand-written validity table (NaN and negative budgets and
    spent values, spent above the budget, -0, infinities), on real blocks: status, outputs and the
    ledger (bit for bit) equal the oracle's, and invalid ledgers are left untouched."""
    from oracle_pins import LEDGER_TABLE
    B, K, V = len(LEDGER_TABLE), 6, 4000
    b = inputs.gen_block(B, K, V, torch.bfloat16, 4322, "cuda")
    led0 = np.array([[bud, sp] for bud, sp, _ in LEDGER_TABLE], np.float32)
    led = torch.from_numpy(led0.copy()).cuda()
    g = gpu_verify(asd, b.logits, b.draft, led, 1.0, 2)
    o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), led0, 1.0, 2)
    assert_parity(g, o, "ledger table")
    bad = np.array([not v for _, _, v in LEDGER_TABLE])
    assert np.all(g["status"][bad] == oracle.STATUS_BAD_LEDGER)
    assert np.all(g["status"][~bad] == 0)
    assert np.array_equal(g["ledger"][bad].view(np.uint32), led0[bad].view(np.uint32))


def test_infinite_controls_and_exhausted_ledger(asd, kernel):
    B, K, V = 16, 8, 5000
    b = inputs.gen_block(B, K, V, torch.float32, 4321, "cuda")
    for (gate, cap, budget, spent) in ((math.inf, INT32_MAX, math.inf, 0.0), (0.0, 2, 4.0, 4.0),
                                       (1.0, 0, 8.0, 0.0), (math.inf, INT32_MAX, 1e-30, 0.0)):
        led = asd.make_ledger(B, budget, spent)
        g = gpu_verify(asd, b.logits, b.draft, led, gate, cap)
        o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), np.array([[budget, spent]] * B, np.float32),
                          gate, cap)
        assert_parity(g, o, f"controls {(gate, cap, budget, spent)}")


def test_many_small_requests(asd, kernel):
    """Many short rows per warp: each warp finishes and selects several requests."""
    for (B, K, V) in ((3000, 31, 40), (5000, 3, 7), (700, 16, 130)):
        b = inputs.gen_block(B, K, V, torch.bfloat16, B + K + V, "cuda")
        led = asd.make_ledger(B, 2.0)
        g = gpu_verify(asd, b.logits, b.draft, led, 0.5, 3)
        o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), np.array([[2.0, 0.0]] * B, np.float32), 0.5, 3)
        assert_parity(g, o, f"B={B} K={K} V={V}")


def test_empty_batch_is_a_noop(asd):
    logits = torch.empty(0, 9, 100, device="cuda")
    draft = torch.empty(0, 8, dtype=torch.int32, device="cuda")
    led = asd.make_ledger(0, 1.0)
    out = asd.verify(logits, draft, led, 1.0, 2)
    torch.cuda.synchronize()
    assert out["accepted_len"].numel() == 0


def test_one_workspace_serves_many_shapes(asd, kernel):
    """The workspace resets itself: one buffer reused across shapes and entry points."""
    ws = asd.Workspace(64, 31, 1, asd.F32)
    rng = np.random.default_rng(8)
    for i in range(20):
        B, K, V = int(rng.integers(1, 64)), int(rng.integers(0, 32)), int(rng.integers(1, 3000))
        dtype = torch.bfloat16 if i % 2 else torch.float32
        b = inputs.gen_block(B, K, V, dtype, 555 + i, "cuda")
        led = asd.make_ledger(B, 3.0)
        out = asd.verify(b.logits, b.draft, led, 1.0, 2, workspace=ws) if i % 3 else \
            asd.verify_strict(b.logits, b.draft, workspace=ws)
        torch.cuda.synchronize()
        g = _np(out)
        g["ledger"] = led.cpu().numpy()
        o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), np.array([[3.0, 0.0]] * B, np.float32), 1.0, 2,
                          strict=(i % 3 == 0))
        assert_parity(g, o, f"call {i}", ledger=bool(i % 3))
    assert ws.error() == 0


def test_verify_reads_pinned_host_memory_in_place(asd, kernel):
    """verify_from_host: kernels read pinned host logits through their device alias; same results."""
    import ctypes

    B, K, V = 8, 8, 70001
    b = inputs.gen_block(B, K, V, torch.bfloat16, 5151, "cuda")
    hl, hd = b.logits.cpu().pin_memory(), b.draft.cpu().pin_memory()
    led_h, led_d = asd.make_ledger(B, 4.0), asd.make_ledger(B, 4.0)
    ws = asd.Workspace(B, K, V, asd.BF16)
    out = asd.alloc_outputs(B, K)
    host_out = {k: torch.empty(out[k].shape, dtype=out[k].dtype, pin_memory=True)
                for k in ("accepted_len", "committed", "recovery")}
    for _ in range(2):  # two rounds: the ledger carries over
        asd.verify_from_host(hl, hd, led_h, 1.0, 2, ws, out, host_out)
        ref = asd.verify(b.logits, b.draft, led_d, 1.0, 2)
        torch.cuda.synchronize()
        for k in ("accepted_len", "committed", "recovery"):
            assert torch.equal(host_out[k], ref[k].cpu()), k
        assert torch.equal(out["row_argmax"], ref["row_argmax"])
        assert torch.equal(led_h, led_d)
    with pytest.raises(ValueError):
        asd.host_alias(torch.zeros(4))  # the binding insists on pinned tensors
    alias = ctypes.c_void_p(0)
    assert asd.load().asd_host_alias(hl.data_ptr(), ctypes.byref(alias)) == 0 and alias.value


ERR_TIMEOUT = 9  # ASD_ERR_TIMEOUT


def test_bounded_wait_reports_timeout_and_context_survives(asd):
    """Failure detection without a fault: a bounded wait on a barrier that nothing signals gives up
    after about a second, the workspace's error word reads ASD_ERR_TIMEOUT, and the same context and
    workspace then verify a block correctly once the workspace is re-initialised."""
    import time
    B, K, V = 4, 8, 1024
    ws = asd.Workspace(B, K, V, 0)
    assert ws.error() == 0
    t0 = time.perf_counter()
    asd.selftest_wait_timeout(ws)
    assert ws.error() == ERR_TIMEOUT
    elapsed = time.perf_counter() - t0
    assert 0.5 < elapsed < 30.0, f"the wait should give up after about a second, took {elapsed:.2f} s"
    # until the workspace is re-initialised, every request of a call that uses it is flagged incomplete:
    # it accepts nothing and keeps its ledger (the small-request kernel here, the TMA row stage below)
    for shape, wsp in (((B, K, V), ws), ((4, 8, 151936), asd.Workspace(4, 8, 151936, 0))):
        if wsp is not ws:
            asd.selftest_wait_timeout(wsp)
            assert wsp.error() == ERR_TIMEOUT
        blk = inputs.gen_block(*shape, torch.float32, 4320, "cuda")
        led = asd.make_ledger(shape[0], 4.0)
        out = asd.verify(blk.logits, blk.draft, led, 1.0, 2, workspace=wsp)
        torch.cuda.synchronize()
        assert np.all(out["status"].cpu().numpy() == asd.STATUS_INCOMPLETE), shape
        assert np.all(out["accepted_len"].cpu().numpy() == 0), shape
        assert torch.equal(led, asd.make_ledger(shape[0], 4.0)), shape
    ws.reset()
    assert ws.error() == 0
    block = inputs.gen_block(B, K, V, torch.float32, 4321, "cuda")
    led = asd.make_ledger(B, 4.0)
    led0 = led.cpu().numpy()
    out = asd.verify(block.logits, block.draft, led, 1.0, 2, workspace=ws)
    torch.cuda.synchronize()
    o = oracle.verify(block.logits.cpu().numpy(), block.draft.cpu().numpy(), led0, 1.0, 2)
    assert ws.error() == 0
    assert np.array_equal(out["accepted_len"].cpu().numpy(), o["accepted_len"])
    assert np.array_equal(out["committed"].cpu().numpy(), o["committed"])
    assert np.array_equal(led.cpu().numpy().view(np.int32), o["ledger"].view(np.int32))


@pytest.mark.parametrize("shape", [(32, 8, 151936), (4, 8, 1024)])
def test_logits_written_by_the_previous_kernel(asd, shape):
    """Without ASD_RESIDENT_INPUTS the logits may come from the kernel right before the call on the same
    stream (as from the model's LM head): every call sees that kernel's output, eagerly and in a CUDA graph."""
    B, K, V = shape
    blocks = [inputs.gen_block(B, K, V, torch.bfloat16, 8800 + i, "cuda") for i in range(4)]
    expect = [oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), np.array([[8.0, 0.0]] * B, np.float32), 1.0, 2)
              for b in blocks]
    buf = torch.empty_like(blocks[0].logits)
    ledgers = [asd.make_ledger(B, 8.0) for _ in range(8)]
    outs = [asd.alloc_outputs(B, K) for _ in range(8)]
    ws = asd.Workspace(B, K, V, asd.BF16)

    def sequence():
        for n in range(8):
            b = blocks[n % 4]
            torch.mul(b.logits, 1, out=buf)  # a kernel writes the logits; the verify follows it directly
            asd.verify(buf, b.draft, ledgers[n], 1.0, 2, workspace=ws, out=outs[n])

    def check(what):
        torch.cuda.synchronize()
        for n in range(8):
            o, g = expect[n % 4], _np(outs[n])
            for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
                assert np.array_equal(g[key], o[key]), f"{what} call {n}: {key}"
            assert np.array_equal(ledgers[n].cpu().numpy().view(np.int32), o["ledger"].view(np.int32))

    for _ in range(3):
        for led in ledgers:
            led.copy_(asd.make_ledger(B, 8.0))
        sequence()
        check("eager")
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        sequence()
    for _ in range(3):
        for led in ledgers:
            led.copy_(asd.make_ledger(B, 8.0))
        graph.replay()
        check("graph")


@pytest.mark.parametrize("resident", [False, True])
@pytest.mark.parametrize("shape", [(4, 8, 1024, torch.float32, 16), (32, 8, 151936, torch.bfloat16, 6)])
def test_back_to_back_calls_carry_the_ledger(asd, shape, resident):
    """Dependent calls issued back to back with no synchronisation in between (eagerly and as one
    CUDA graph): each reads the ledger the previous one wrote, which a call that starts early
    (programmatic dependent launch) must not read before that call has completed."""
    B, K, V, dtype, n = shape
    blocks = [inputs.gen_block(B, K, V, dtype, 9100 + i, "cuda") for i in range(n)]
    led0 = np.array([[4.0, 0.0]] * B, np.float32)
    expect, led = [], led0
    for b in blocks:
        o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), led, 1.0, 2)
        expect.append(o)
        led = o["ledger"]
    ledger = torch.from_numpy(led0).cuda()
    outs = [asd.alloc_outputs(B, K) for _ in range(n)]
    ws = asd.Workspace(B, K, V, asd.BF16 if dtype == torch.bfloat16 else asd.F32)

    def sequence():
        for i, b in enumerate(blocks):
            asd.verify(b.logits, b.draft, ledger, 1.0, 2, workspace=ws, out=outs[i], resident=resident)

    def check(what):
        torch.cuda.synchronize()
        for i in range(n):
            g = _np(outs[i])
            for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
                assert np.array_equal(g[key], expect[i][key]), f"{what} call {i}: {key}"
            assert np.array_equal(g["row_regret"].view(np.int32), expect[i]["row_regret"].view(np.int32))
        assert np.array_equal(ledger.cpu().numpy().view(np.int32), expect[-1]["ledger"].view(np.int32))

    sequence()
    check("eager")
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    ledger.copy_(torch.from_numpy(led0))
    torch.cuda.synchronize()
    with torch.cuda.graph(graph, stream=side):
        sequence()
    for _ in range(2):
        ledger.copy_(torch.from_numpy(led0).cuda())
        graph.replay()
        check("graph")


@pytest.mark.parametrize("cfg_id,dtype", [(1, torch.bfloat16), (3, torch.float32), (3, torch.bfloat16)])
def test_zero_budget_is_strict_on_the_large_configs(asd, cfg_id, dtype):
    """Budget 0 (Alg. 1's dispatch) equals asd_verify_strict and the oracle's strict mode bit for bit,
    and leaves the ledger untouched, on the Qwen3-14B and the large-batch 129k workloads."""
    cfg = inputs.CONFIGS[cfg_id]
    B, K, V = cfg["B"], cfg["K"], cfg["V"]
    for blk in range(2):
        b = inputs.gen_block(B, K, V, dtype, inputs.seed_for(cfg_id, 40, blk), "cuda")
        led = asd.make_ledger(B, 0.0, 0.0)
        g = gpu_verify(asd, b.logits, b.draft, led, 1.0, 2)
        s = gpu_verify(asd, b.logits, b.draft, None, 0, 0, strict=True)
        o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), None, strict=True)
        for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
            assert np.array_equal(g[key], s[key]), f"strict entry: {key}"
            assert np.array_equal(g[key], o[key]), f"oracle strict: {key}"
        assert np.array_equal(g["ledger"], np.zeros((B, 2), np.float32))


@pytest.mark.parametrize("shape", [(4, 8, 1024, torch.float32), (32, 8, 151936, torch.bfloat16),
                                   (64, 31, 3000, torch.bfloat16)])
def test_launches_without_programmatic_dependent_launch(asd, shape):
    """The no_pdl launch option (plain stream order, no early start) gives the same results bit for bit
    as the default launches, on each row-stage kernel the shape reaches, over four carried blocks."""
    B, K, V, dtype = shape
    blocks = [inputs.gen_block(B, K, V, dtype, 9300 + i, "cuda") for i in range(4)]
    results = {}
    try:
        for pdl in (True, False):
            for path in ("auto", "stream", "tma"):
                asd.set_launch_options(path=path, pdl=pdl)
                led = asd.make_ledger(B, 4.0)
                outs = [gpu_verify(asd, b.logits, b.draft, led, 1.0, 2) for b in blocks]
                results[(pdl, path)] = outs
    finally:
        asd.reset_launch_options()
    ref = results[(True, "auto")]
    for key, outs in results.items():
        for i, (g, r) in enumerate(zip(outs, ref)):
            for k in ("accepted_len", "committed", "recovery", "row_argmax", "status", "ledger"):
                assert np.array_equal(g[k].view(np.uint32) if g[k].dtype == np.float32 else g[k],
                                      r[k].view(np.uint32) if r[k].dtype == np.float32 else r[k]), \
                    f"{key} block {i}: {k}"
    led0 = np.array([[4.0, 0.0]] * B, np.float32)
    o = oracle.verify(blocks[0].logits.cpu(), blocks[0].draft.cpu().numpy(), led0, 1.0, 2)
    assert_parity(results[(False, "auto")][0], o, "no pdl, block 0")


def test_concurrent_streams_keep_their_own_state(asd):
    """Three streams issue dependent sequences at the same time, interleaved call by call and never
    synchronised with each other: the TMA row stage with its selection kernel (Qwen3-14B shape), the
    one-CTA-per-request kernel (the tiny shape), and the fused LM-head verify (exact inputs). Each
    stream has its own workspace and ledger; every call equals the oracle, so no call sees another
    stream's state."""
    n = 5
    specs = [(32, 8, 151936, torch.bfloat16), (4, 8, 1024, torch.float32)]
    seqs = []
    for s, (B, K, V, dtype) in enumerate(specs):
        blocks = [inputs.gen_block(B, K, V, dtype, 9400 + 10 * s + i, "cuda") for i in range(n)]
        led = np.array([[4.0, 0.0]] * B, np.float32)
        expect = []
        for b in blocks:
            o = oracle.verify(b.logits.cpu(), b.draft.cpu().numpy(), led, 1.0, 2)
            expect.append(o)
            led = o["ledger"]
        seqs.append(dict(blocks=blocks, expect=expect, ledger=asd.make_ledger(B, 4.0),
                         ws=asd.Workspace(B, K, V, asd.BF16 if dtype == torch.bfloat16 else asd.F32),
                         outs=[asd.alloc_outputs(B, K) for _ in range(n)], stream=torch.cuda.Stream()))
    Bl, Kl, Hl, Vl = 8, 8, 256, 1300
    lm = [inputs.gen_lmhead_exact(Bl, Kl, Hl, Vl, 9500 + i, "cuda") for i in range(n)]
    lm_expect, led = [], np.array([[8.0, 0.0]] * Bl, np.float32)
    for inp in lm:
        z64 = oracle.lmhead_logits_matmul(inp.hidden.cpu(), inp.weight.cpu())
        o = oracle.verify(z64.astype(np.float32).reshape(Bl, Kl + 1, Vl), inp.draft.cpu().numpy(), led, 1.0, 2)
        lm_expect.append(o)
        led = o["ledger"]
    lm_led = asd.make_ledger(Bl, 8.0)
    lm_ws = asd.lmhead_workspace(Bl, Kl, Vl, Hl, torch.device("cuda"))
    lm_outs = [asd.alloc_outputs(Bl, Kl) for _ in range(n)]
    lm_stream = torch.cuda.Stream()
    for st in [q["stream"] for q in seqs] + [lm_stream]:
        st.wait_stream(torch.cuda.current_stream())
    for i in range(n):
        for q in seqs:
            with torch.cuda.stream(q["stream"]):
                b = q["blocks"][i]
                asd.verify(b.logits, b.draft, q["ledger"], 1.0, 2, workspace=q["ws"], out=q["outs"][i])
        with torch.cuda.stream(lm_stream):
            asd.lmhead_verify(lm[i].hidden, lm[i].weight, lm[i].draft, lm_led, 1.0, 2, workspace=lm_ws,
                              out=lm_outs[i])
    torch.cuda.synchronize()
    for s, q in enumerate(seqs):
        for i in range(n):
            g = _np(q["outs"][i])
            for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
                assert np.array_equal(g[key], q["expect"][i][key]), f"stream {s} call {i}: {key}"
        assert np.array_equal(q["ledger"].cpu().numpy().view(np.int32), q["expect"][-1]["ledger"].view(np.int32))
    for i in range(n):
        g = _np(lm_outs[i])
        for key in ("accepted_len", "committed", "recovery", "row_argmax", "status"):
            assert np.array_equal(g[key], lm_expect[i][key]), f"LM-head stream call {i}: {key}"
    assert np.array_equal(lm_led.cpu().numpy().view(np.int32), lm_expect[-1]["ledger"].view(np.int32))
