"""Parity over the run lengths the workloads state: the ledger (B, s) of Sec. 3.2 carried across every
block of a request, every block checked against the oracle bit for bit (Alg. 1's outputs, Eq. 13's
ledger, the row argmaxes and fp32 regrets).

  * Qwen3-14B-shaped verify (B=32, K=8, V=151936 bf16, g=1, M=2, budget 8): 256 sequential blocks, through
    the default launch (the row stage waits for the previous kernel), with resident inputs (overlapping
    launches), with the selection inside the row stage, and through the register-streaming kernel;
  * large-batch serving shape (B=256, K=4, V=129280, g=1, M=1, budget 4): 64 blocks at each of the four
    acceptance points, fp32 and bf16, with and without resident inputs;
  * the benchmark's launch configuration: 256 steps over its rotating buffers captured in one CUDA graph,
    every step writing its own outputs, with and without resident inputs.

The oracle's row stage (argmax, regret) runs per block in a thread pool (the C oracle releases the GIL);
its selection is then replayed block after block with the carried ledger (oracle.select, which the pins
show equal to oracle.verify).
"""
import concurrent.futures as cf
import threading

import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2608_03447_gb300 import inputs

pytestmark = pytest.mark.gpu

KEYS = ("accepted_len", "committed", "recovery", "row_argmax", "status")
HOST_BYTES_IN_FLIGHT = 6 << 30  # logits copied to the host and waiting for the oracle


class RowStage:
    """Oracle row stage of many blocks, in parallel, with a bound on the host bytes held."""

    def __init__(self, threads=16):
        self.pool = cf.ThreadPoolExecutor(max_workers=threads)
        self.cond = threading.Condition()
        self.held = 0
        self.futures = []

    def _run(self, z, x, nbytes):
        try:
            return oracle.verify(z, x, None, strict=True)
        finally:
            with self.cond:
                self.held -= nbytes
                self.cond.notify_all()

    def submit(self, logits: torch.Tensor, draft: torch.Tensor) -> None:
        nbytes = logits.numel() * logits.element_size()
        with self.cond:
            self.cond.wait_for(lambda: self.held == 0 or self.held + nbytes <= HOST_BYTES_IN_FLIGHT)
            self.held += nbytes
        z, x = logits.cpu(), draft.cpu().numpy()
        self.futures.append(self.pool.submit(self._run, z, x, nbytes))

    def results(self):
        out = [f.result() for f in self.futures]
        self.pool.shutdown()
        return out


def _np(out):
    return {k: v.cpu().numpy() for k, v in out.items()}


def check_block(g, o, what, ledger_gpu=None):
    for key in KEYS:
        if key in g:
            diff = np.argwhere(g[key] != o[key])
            assert diff.size == 0, f"{what}: {key} differs at {diff[:5].tolist()}"
    if "row_regret" in g:
        gr, orr = g["row_regret"], o["row_regret"]
        same = (gr.view(np.uint32) == orr.view(np.uint32)) | (np.isnan(gr) & np.isnan(orr))
        assert same.all(), f"{what}: row_regret differs at {np.argwhere(~same)[:5].tolist()}"
    if ledger_gpu is not None:
        assert np.array_equal(ledger_gpu.view(np.uint32), o["ledger"].view(np.uint32)), f"{what}: ledger"


def replay(rows, drafts, budget, B, gate, cap):
    """The oracle's selection over the blocks in order, ledger carried (Sec. 3.2)."""
    led = np.array([[budget, 0.0]] * B, np.float32)
    expect = []
    for r, x in zip(rows, drafts):
        o = oracle.select(x, r["row_argmax"], r["row_regret"], r["status"], led, gate, cap)
        o["row_argmax"], o["row_regret"] = r["row_argmax"], r["row_regret"]
        expect.append(o)
        led = o["ledger"]
    return expect


def long_run(asd, B, K, V, dtype, nblocks, gate, cap, budget, config, variants, mix=inputs.MIX_DEFAULT,
             point=0, strict_check=True):
    """nblocks sequential blocks; each variant (launch options + resident flag) carries its own ledger
    on the device; every block of every variant is checked against the oracle."""
    ledgers = {name: asd.make_ledger(B, budget) for name in variants}
    got = {name: [] for name in variants}
    strict_got = []
    drafts = []
    stage = RowStage()
    try:
        for blk in range(nblocks):
            b = inputs.gen_block(B, K, V, dtype, inputs.seed_for(config, point, blk), "cuda", mix=mix)
            for name, (opts, resident) in variants.items():
                asd.set_launch_options(**opts)
                out = asd.verify(b.logits, b.draft, ledgers[name], gate, cap, resident=resident)
                g = _np(out)
                g["ledger"] = ledgers[name].cpu().numpy()
                got[name].append(g)
            asd.reset_launch_options()
            if strict_check:
                strict_got.append(_np(asd.verify_strict(b.logits, b.draft)))
            drafts.append(b.draft.cpu().numpy())
            stage.submit(b.logits, b.draft)
    finally:
        asd.reset_launch_options()
    rows = stage.results()
    expect = replay(rows, drafts, budget, B, gate, cap)
    for blk in range(nblocks):
        for name in variants:
            g = got[name][blk]
            check_block(g, expect[blk], f"{name} block {blk}", g["ledger"])
        if strict_check:
            check_block(strict_got[blk], rows[blk], f"strict block {blk}")
    return expect


DEFAULT = ({}, False)
RESIDENT = ({}, True)
FUSED = ({"path": "tma", "fused_select": True}, False)
STREAM = ({"path": "stream"}, False)


def test_qwen3_shape_256_carried_blocks(asd):
    """B=32, K=8, V=151936 bf16, g=1, M=2, budget 8 carried over all 256 blocks of every request."""
    cfg = inputs.CONFIGS[1]
    expect = long_run(asd, cfg["B"], cfg["K"], cfg["V"], cfg["dtype"], 256, cfg["gate"], cfg["cap"],
                      cfg["budget"], 1, {"default": DEFAULT, "resident": RESIDENT, "fused": FUSED,
                                         "stream": STREAM})
    spent = expect[-1]["ledger"][:, 1]
    assert np.all(spent <= cfg["budget"])
    assert np.all(spent > 0), "every request should have spent some of its budget over 256 blocks"
    accepted_mismatch = sum(int(((o["accepted_len"][:, None] > np.arange(cfg["K"]))
                                 & (o["row_argmax"][:, :cfg["K"]] != o["committed"][:, :cfg["K"]])).sum())
                            for o in expect)
    assert accepted_mismatch > 0, "the run must exercise accepted mismatches"


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_large_batch_129k_64_blocks_per_hit_point(asd, dtype):
    """B=256, K=4, V=129280, g=1, M=1, budget 4 over 64 blocks at p_hit in {0.3, 0.5, 0.7, 0.9}."""
    cfg = inputs.CONFIGS[3]
    for pi, hit in enumerate(cfg["hits"]):
        long_run(asd, cfg["B"], cfg["K"], cfg["V"], dtype, 64, cfg["gate"], cfg["cap"], cfg["budget"], 3,
                 {"default": DEFAULT, "resident": RESIDENT}, mix=inputs.mix_for_hit(hit), point=pi,
                 strict_check=(pi == 0))


@pytest.mark.parametrize("resident", [True, False])
def test_bench_graph_every_step_matches_oracle(asd, resident):
    """The benchmark's launch configuration (rotating buffers larger than L2, one CUDA graph of steps,
    ledger carried): 256 steps, each writing its own outputs, every step compared with the oracle."""
    from paper_2608_03447_gb300.workload import VerifyWorkload
    cfg = inputs.CONFIGS[1]
    B, K = cfg["B"], cfg["K"]
    wl = VerifyWorkload(B, K, cfg["V"], cfg["dtype"], cfg["gate"], cfg["cap"], cfg["budget"], config=1,
                        with_rows=True, resident=resident)
    nsteps = 256
    outs = [asd.alloc_outputs(B, K) for _ in range(nsteps)]
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        wl.step(0, stream)  # set-up outside capture
    torch.cuda.current_stream().wait_stream(stream)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for i in range(nsteps):
            k = i % wl.nbuf
            asd.verify(wl.logits[k], wl.drafts[k], wl.ledger, wl.gate, wl.cap, wl.workspace, outs[i],
                       torch.cuda.current_stream(), resident=resident)
    # the same steps with the ledger copied out after each one (extra copy kernels between the calls)
    hist = torch.empty(nsteps, B, 2, device="cuda")
    graph_hist = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph_hist, stream=stream):
        for i in range(nsteps):
            k = i % wl.nbuf
            asd.verify(wl.logits[k], wl.drafts[k], wl.ledger, wl.gate, wl.cap, wl.workspace, outs[i],
                       torch.cuda.current_stream(), resident=resident)
            hist[i].copy_(wl.ledger)
    stage = RowStage()
    for k in range(wl.nbuf):
        stage.submit(wl.logits[k], wl.drafts[k])
    rows = stage.results()
    drafts = [wl.drafts[k].cpu().numpy() for k in range(wl.nbuf)]
    expect = replay([rows[i % wl.nbuf] for i in range(nsteps)], [drafts[i % wl.nbuf] for i in range(nsteps)],
                    cfg["budget"], B, cfg["gate"], cfg["cap"])
    for rep in range(2):
        wl.reset_ledger()
        for o in outs:
            for t in o.values():
                t.fill_(-7)
        graph.replay()
        torch.cuda.synchronize()
        for i in range(nsteps):
            check_block(_np(outs[i]), expect[i], f"replay {rep} step {i}")
        assert np.array_equal(wl.ledger.cpu().numpy().view(np.uint32), expect[-1]["ledger"].view(np.uint32))
    wl.reset_ledger()
    graph_hist.replay()
    torch.cuda.synchronize()
    h = hist.cpu().numpy()
    for i in range(nsteps):
        check_block(_np(outs[i]), expect[i], f"ledger-history replay step {i}", h[i])
    assert wl.workspace.error() == 0


@pytest.mark.parametrize("path", ["auto", "stream"])
def test_more_than_2_31_logits(asd, path):
    """B=1600, K=8, V=151936 bf16: 2.19e9 logits (4.4 GB), past every 32-bit element offset. The TMA row
    stage (with and without resident inputs) and the register-streaming kernel match the oracle, which
    runs request slices in parallel (requests are independent; each slice carries its own ledgers)."""
    B, K, V = 1600, 8, 151936
    assert B * (K + 1) * V > 2**31
    b = inputs.gen_block(B, K, V, torch.bfloat16, 7_777, "cuda")
    led0 = np.array([[4.0, 0.0]] * B, np.float32)
    outs = []
    try:
        asd.set_launch_options(path=path)
        for resident in (False, True):
            led = torch.from_numpy(led0.copy()).cuda()
            out = _np(asd.verify(b.logits, b.draft, led, 1.0, 2, resident=resident))
            out["ledger"] = led.cpu().numpy()
            outs.append(out)
    finally:
        asd.reset_launch_options()
    z, x = b.logits.cpu(), b.draft.cpu().numpy()
    del b
    step = 100
    with cf.ThreadPoolExecutor(max_workers=16) as pool:
        parts = list(pool.map(lambda s: oracle.verify(z[s:s + step], x[s:s + step], led0[s:s + step], 1.0, 2),
                              range(0, B, step)))
    o = {k: np.concatenate([p[k] for p in parts]) for k in parts[0]}
    for g in outs:
        check_block(g, o, f"{path} > 2^31 logits", g["ledger"])
