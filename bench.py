"""Throughput of the ASD verifier step on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Workload (one step = one asd_verify call, the whole hot path): the
Qwen3-14B-shaped verify, B=32 requests x (K=8)+1 rows x V=151936 bf16 logits,
gate 1.0, cap 2, budget 8.0 carried across steps. Inputs are resident in HBM,
rotating over distinct logit buffers whose total exceeds 4x the L2 size, and the
K timed steps replay CUDA graphs (two kernel nodes per step: the row stage and
the selection, chained by programmatic dependent launch). Prints one JSON
line (rank 0). Under torchrun each rank verifies its own batch (weak scaling, no
collective on the data path; the barrier and the max over ranks time the job).

--impl reference times the CPU oracle as it stands on the host cores (rank 0
only), one full block of the same workload per step.

--case NAME --launches N runs only a few launches of one workload (the
profiler captures in profiles/ use it).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "verify rows/s & HBM GB/s (% of ~8 TB/s), V=151936 bf16 B=32 K=8"
NOMINAL_HBM_GBS = 8000.0
B, K, V = 32, 8, 151936
GATE, CAP, BUDGET = 1.0, 2, 8.0
WORKLOAD = "qwen3-14b-verify: B=32 requests, K=8 draft tokens (288 target rows), V=151936, bf16 logits, " \
           "gate=1.0, cap=2, budget=8.0 carried across steps"


def bench_config(world: int) -> dict:
    """The workload, as both arms report it (the same dict, so the two lines compare like for like)."""
    return {"workload": WORKLOAD, "B": B, "K": K, "V": V, "gate": GATE, "cap": CAP, "budget": BUDGET,
            "parallelism": f"dp{world} (independent requests per rank)",
            "l2": "inputs larger than L2: steps rotate over logit buffers totalling more than 4x the L2 size"}
CSRC = os.path.join(ROOT, "paper_2608_03447_gb300", "csrc")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
# the sources each profiled kernel is built from (a recorded traffic figure is
# reported only while these are unchanged)
KERNEL_SOURCES = {
    "verify_tma_kernel": ["asd_verify.cu", "asd_device.cuh"],
    "lmhead_verify_kernel": ["asd_lmhead.cu", "asd_device.cuh"],
}
LM_B, LM_K, LM_H, LM_V = 64, 8, 5120, 151936
LM_WORKLOAD = "fused-lmhead: B=64 requests, K=8 (576 target rows), H=5120, V=151936, bf16 h and W, fp32 " \
              "accumulation on tcgen05, gate=1.0, cap=2, budget=8.0"


def peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "source": "fallback"}


def source_digest(kernel: str) -> str:
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[kernel]:
        with open(os.path.join(CSRC, name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def recorded_traffic(kernel: str, workload: str | None = None) -> float | None:
    """DRAM bytes per launch from the committed ncu summary (the headline workload's, or the named
    workload's entry), if it is for the current kernel sources."""
    try:
        with open(TRAFFIC_FILE) as f:
            rec = json.load(f)[kernel]
        if rec.get("sources_sha256") != source_digest(kernel):
            return None
        return float(rec["dram_bytes_per_launch"] if workload is None else rec["workloads"][workload])
    except (OSError, ValueError, KeyError, TypeError, AttributeError):
        return None


def bf16_peaks() -> dict:
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"burst": float(p["bf16_tflops"]), "sustained": float(p["bf16_tflops_sustained"]),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"burst": 1900.0, "sustained": 1700.0, "source": "fallback"}


def run_lmhead(dev, clocks=None, iters: int = 20, sustain_s: float = 1.2) -> dict:
    """The fused LM-head + verify timed alone: CUDA events around `iters` launches (burst peak), then a
    sustained loop of about `sustain_s` seconds with the SM clock sampled, so that each time can be read
    with the clock it ran at (time x median SM GHz separates a tiling change from clock drift)."""
    from paper_2608_03447_gb300 import asd, inputs
    inp = inputs.gen_lmhead(LM_B, LM_K, LM_H, LM_V, inputs.seed_for(4), dev)
    led = asd.make_ledger(LM_B, 8.0, 0.0, dev)
    ws = asd.lmhead_workspace(LM_B, LM_K, LM_V, LM_H, dev)
    out = asd.alloc_outputs(LM_B, LM_K, dev)
    out["row_top"] = torch.empty(LM_B, LM_K + 1, device=dev)
    stream = torch.cuda.current_stream(dev)

    def launch():
        asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, 1.0, 2, workspace=ws, out=out)

    def timed(n):
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0 = time.time()
        start.record(stream)
        for _ in range(n):
            launch()
        end.record(stream)
        end.synchronize()
        return start.elapsed_time(end) / n, t0, time.time()

    for _ in range(3):
        launch()
    torch.cuda.synchronize(dev)
    ms, tb0, tb1 = timed(iters)
    flop = 2.0 * LM_B * (LM_K + 1) * LM_H * LM_V
    # the library GEMM of the same shape alone (bf16 logits out, no reduction), timed the same way
    logits = torch.empty(LM_B * (LM_K + 1), LM_V, dtype=torch.bfloat16, device=dev)
    for _ in range(3):
        torch.matmul(inp.hidden, inp.weight.t(), out=logits)
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0.record(stream)
    for _ in range(iters):
        torch.matmul(inp.hidden, inp.weight.t(), out=logits)
    c1.record(stream)
    c1.synchronize()
    ms_gemm = c0.elapsed_time(c1) / iters
    del logits
    tflops = flop / (ms * 1e-3) / 1e12
    pk = bf16_peaks()
    # one of four tensor-parallel ranks: its quarter of W, the partials (the all-gather and the
    # combine follow; the combine is timed with the sharded verify row); a burst too, so it runs
    # before the sustained loop pulls the clock down to the power cap
    S = 4
    vs = LM_V // S
    shard = inp.weight[:vs].contiguous()
    parts = torch.empty(LM_B * (LM_K + 1), asd.PARTIAL_WORDS, dtype=torch.int32, device=dev)
    sws = asd.lmhead_workspace(LM_B, LM_K, vs, LM_H, dev)
    for _ in range(3):
        asd.lmhead_partials(inp.hidden, shard, inp.draft, 0, LM_V, workspace=sws, out=parts)
    torch.cuda.synchronize(dev)
    s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s2.record(stream)
    for _ in range(iters):
        asd.lmhead_partials(inp.hidden, shard, inp.draft, 0, LM_V, workspace=sws, out=parts)
    e2.record(stream)
    e2.synchronize()
    ms_rank = s2.elapsed_time(e2) / iters
    del shard
    rank_tflops = flop / S / (ms_rank * 1e-3) / 1e12
    n_sus = max(iters, int(sustain_s / (ms * 1e-3)))
    ms_sus, ts0, ts1 = timed(n_sus)
    tflops_sus = flop / (ms_sus * 1e-3) / 1e12
    clk_b = clocks.window(tb0, tb1) if clocks is not None else {"sm_mhz": None}
    clk_s = clocks.window(ts0, ts1) if clocks is not None else {"sm_mhz": None}

    def ghz_ms(t, c):
        return None if c.get("sm_mhz") is None else t * c["sm_mhz"] / 1e3

    summary = {"bound": "tensor", "achieved": tflops, "peak": pk["burst"], "unit": "TFLOP/s",
               "frac": tflops / pk["burst"], "ms": ms, "library_gemm_ms": ms_gemm, "sm_mhz": clk_b.get("sm_mhz"),
               "ms_x_ghz": ghz_ms(ms, clk_b),
               "sustained": {"ms": ms_sus, "achieved": tflops_sus, "peak": pk["sustained"],
                             "frac": tflops_sus / pk["sustained"], "sm_mhz": clk_s.get("sm_mhz"),
                             "ms_x_ghz": ghz_ms(ms_sus, clk_s), "launches": n_sus,
                             "reasons": clk_s.get("reasons")},
               "traffic": recorded_traffic("lmhead_verify_kernel"), "kernel": "lmhead_verify_kernel",
               "algorithmic_flop_per_launch": flop, "peak_source": pk["source"]}
    detail = {"workload": LM_WORKLOAD, "ms_per_step": ms, "rows_per_s": LM_B * (LM_K + 1) / (ms * 1e-3),
              "launches": iters,
              "per_rank_of_4": {"ms": ms_rank, "tflops": rank_tflops, "frac": rank_tflops / pk["burst"],
                                "workload": f"asd_lmhead_partials on a {vs} x {LM_H} shard of W (one of {S} "
                                            "tensor-parallel ranks), 576 rows"}}
    return {"summary": summary, "detail": detail}


class ClockSampler:
    """nvidia-smi clock / throttle sampling in the background (200 ms period)."""

    QUERY = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    def _rows(self):
        """(unix time, sm MHz, max MHz, reason names) per sample."""
        self.file.flush()
        self.file.seek(0)
        out = []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.file.read().strip().splitlines():
            r = [x.strip() for x in line.split(",")]
            try:
                t = time.mktime(time.strptime(r[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                t += float("0." + r[0].split(".")[1]) if "." in r[0] else 0.0
                out.append((t, float(r[1]), float(r[2]),
                            {n for n, v in zip(names, r[5:9]) if v.lower() in ("active", "1")}))
            except (ValueError, IndexError):
                continue
        return out

    def window(self, t0: float, t1: float, min_samples: int = 1) -> dict:
        """Median SM clock and throttle reasons of the samples taken in [t0, t1]."""
        rows = [r for r in self._rows() if t0 - 0.25 <= r[0] <= t1 + 0.25]
        if len(rows) < min_samples:
            return {"sm_mhz": None, "samples": len(rows)}
        return {"sm_mhz": statistics.median(r[1] for r in rows), "sm_max_mhz": max(r[2] for r in rows),
                "reasons": sorted(set().union(*(r[3] for r in rows))), "samples": len(rows)}

    def stop(self) -> None:
        if self.proc is None:
            return
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()

    def close(self) -> None:
        try:
            os.unlink(self.file.name)
        except OSError:
            pass


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_config(rank: int) -> int:
    """Seed family of a rank's own batch: ranks verify disjoint requests (weak scaling)."""
    return 1 + 100 * rank


def max_over_ranks(value: float, device, world: int) -> float:
    """The job's time is its slowest rank's (all_reduce MAX over the process group)."""
    t = torch.tensor([value], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rows_per_s(world: int, rows_per_step: int, steps: int, seconds: float) -> float:
    """Whole-job throughput: the rows every rank verified over the slowest rank's time."""
    return world * rows_per_step * steps / seconds


def run_reference(args) -> None:
    """The CPU oracle as it stands, on the host cores: one full block of the workload per step."""
    import concurrent.futures as cf
    from oracle import oracle
    from paper_2608_03447_gb300 import inputs
    rank, world, _ = dist_env()
    if rank != 0:
        return
    cores = os.cpu_count() or 1
    lib = oracle.load_library()
    nblk = 2
    blocks = [inputs.gen_block(B, K, V, torch.bfloat16, inputs.seed_for(1, 0, i), "cpu") for i in range(nblk)]
    host = [(oracle.bf16_bits(b.logits), b.draft.numpy()) for b in blocks]
    led = np.array([[BUDGET, 0.0]] * B, np.float32)

    def one_request(args_):
        z, x, b, led_b = args_
        return oracle.verify(z[b:b + 1], x[b:b + 1], led_b, GATE, CAP, dtype=oracle.DTYPE_BF16, lib=lib)

    pool = cf.ThreadPoolExecutor(max_workers=cores)

    def step(i):
        nonlocal led
        z, x = host[i % nblk]
        res = list(pool.map(one_request, [(z, x, b, led[b:b + 1]) for b in range(B)]))
        led = np.concatenate([r["ledger"] for r in res])

    for i in range(args.warmup):
        step(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(i)
    dt = time.perf_counter() - t0
    pool.shutdown()
    rows_per_s = args.steps * B * (K + 1) / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": rows_per_s, "unit": "rows/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": bench_config(world),
        "cpu_baseline": {"value": rows_per_s, "unit": "rows/s", "cores": cores, "kind": "oracle",
                         "sample": f"{args.steps} full blocks of {B}x{K + 1}x{V} bf16, one request per thread"},
        "e2e": {"value": rows_per_s, "unit": "rows/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def cpu_baseline(wl, seconds: float = 12.0) -> dict:
    """The oracle as it stands on the host cores, on a bounded sample of the same workload."""
    import concurrent.futures as cf
    from oracle import oracle
    lib = oracle.load_library()
    cores = os.cpu_count() or 1
    nblk = min(2, wl.nbuf)
    host = [(oracle.bf16_bits(wl.logits[i].cpu()), wl.drafts[i].cpu().numpy()) for i in range(nblk)]
    led = np.array([[BUDGET, 0.0]] * B, np.float32)

    def one_request(a):
        z, x, b = a
        return oracle.verify(z[b:b + 1], x[b:b + 1], led[b:b + 1], GATE, CAP, dtype=oracle.DTYPE_BF16, lib=lib)

    rows = 0
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(max_workers=cores) as pool:
        i = 0
        while True:
            z, x = host[i % nblk]
            list(pool.map(one_request, [(z, x, b) for b in range(B)]))
            rows += B * (K + 1)
            i += 1
            if time.perf_counter() - t0 >= seconds:
                break
    dt = time.perf_counter() - t0
    # one thread, and the two stages apart: the row stage (the strict oracle: argmax, draft logits,
    # regrets, plus Eq. 2's trivial selection) and Alg. 1 alone (oracle_select on those rows)
    z, x = host[0]
    n1, t1 = 0, time.perf_counter()
    while time.perf_counter() - t1 < 2.0:
        rows_out = oracle.verify(z, x, None, strict=True, dtype=oracle.DTYPE_BF16, lib=lib)
        n1 += 1
    row_ms = (time.perf_counter() - t1) / n1 * 1e3
    n2, t2 = 0, time.perf_counter()
    while time.perf_counter() - t2 < 0.5:
        oracle.select(x, rows_out["row_argmax"], rows_out["row_regret"], rows_out["status"], led, GATE, CAP, lib=lib)
        n2 += 1
    sel_ms = (time.perf_counter() - t2) / n2 * 1e3
    return {"value": rows / dt, "unit": "rows/s", "cores": cores, "kind": "oracle",
            "sample": f"{i} full blocks ({B}x{K + 1}x{V} bf16 from the GPU buffers), one request per thread, "
                      f"{dt:.1f} s",
            "single_thread": {"rows_per_s": B * (K + 1) / ((row_ms + sel_ms) / 1e3),
                              "row_stage_ms_per_block": row_ms, "selection_ms_per_block": sel_ms,
                              "sample": f"{n1} row-stage and {n2} selection passes over one block"}}


def run_gpu(args) -> None:
    import torch.distributed as dist
    from paper_2608_03447_gb300 import asd, inputs
    from paper_2608_03447_gb300.workload import VerifyWorkload, l2_bytes

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    asd.load()

    # the logit buffers are written once, before any step: ASD_RESIDENT_INPUTS lets consecutive steps overlap
    wl = VerifyWorkload(B, K, V, torch.bfloat16, GATE, CAP, BUDGET, config=rank_config(rank), device=dev,
                        resident=True)
    steps, warmup = args.steps, args.warmup
    G = min(steps, 512)
    graph_full = wl.capture(G, first=0)
    graph_rem = wl.capture(steps % G, first=(steps // G) * G) if steps % G else None
    wl.reset_ledger()
    torch.cuda.synchronize(dev)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    clocks = ClockSampler(local)
    clocks.start()
    # warm-up: W graph replays, then untimed steps until ~1 s of load (clocks settle, sampler sees load)
    stream = torch.cuda.current_stream(dev)
    for _ in range(max(3, warmup)):
        graph_full.replay()
    t_soak = time.time()
    while time.time() - t_soak < 1.0:
        graph_full.replay()
        torch.cuda.synchronize(dev)
    barrier()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks.mark_start()
    start.record(stream)
    for _ in range(steps // G):
        graph_full.replay()
    if graph_rem is not None:
        graph_rem.replay()
    end.record(stream)
    end.synchronize()
    barrier()
    clocks.mark_end()
    ms_max = max_over_ranks(start.elapsed_time(end), dev, world)
    sec_per_step = ms_max / 1e3 / steps
    rows_per_step = B * (K + 1)
    value = job_rows_per_s(world, rows_per_step, steps, ms_max / 1e3)
    bytes_per_launch = wl.bytes_per_step
    achieved_gbs = bytes_per_launch / sec_per_step / 1e9

    # ASD and strict steps interleaved, graph by graph (median and best of 5 each)
    wl.strict = True
    graph_strict = wl.capture(G, first=0)
    wl.strict = False
    per = {"asd": [], "strict": []}
    for _ in range(5):
        for name, gr in (("asd", graph_full), ("strict", graph_strict)):
            if name == "asd":
                wl.reset_ledger()
            s_i, e_i = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            s_i.record(stream)
            gr.replay()
            e_i.record(stream)
            e_i.synchronize()
            per[name].append(s_i.elapsed_time(e_i) * 1e3 / G)
    interleaved = {k: {"median_us": float(np.median(v)), "best_us": float(min(v))} for k, v in per.items()}
    del graph_strict

    # the lone call: the same steps without the flag, each row stage reading nothing before the previous
    # kernel completes (what a call right behind a producer kernel of its logits gets); graphs of 512
    wl.resident = False
    G_lone = 512
    graph_lone = wl.capture(G_lone, first=0)
    wl.reset_ledger()
    graph_lone.replay()
    torch.cuda.synchronize(dev)
    lone = []
    for _ in range(3):
        s_d, e_d = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s_d.record(stream)
        graph_lone.replay()
        e_d.record(stream)
        e_d.synchronize()
        lone.append(s_d.elapsed_time(e_d) * 1e3 / G_lone)
    lone_us = float(np.median(lone))
    del graph_lone
    wl.resident = True
    wl.reset_ledger()

    # the allocation-free entry point on the same steps, eager (it clears its scratch before each call)
    noalloc = run_noalloc(wl, dev) if rank == 0 else None

    # end to end through the public API from pinned host buffers (copies inside the timed region)
    e2e = run_e2e(wl, dev, steps=max(10, min(steps, 200)), world=world)

    nxt = run_next_rows(wl, dev) if rank == 0 else None
    other = run_other_configs(dev) if rank == 0 and args.configs else None
    # last: its sustained loop runs at the power cap, and the clock takes a while to come back
    lm = run_lmhead(dev, clocks) if rank == 0 else None
    clocks.stop()
    timed = clocks.window(clocks.t0, clocks.t1)
    if timed["sm_mhz"] is not None:
        clk = dict(timed, window="the timed region and 0.25 s either side of it (one sample every 200 ms; the "
                                 "step graph ran back to back over the 1 s before it)")
    else:
        clk = dict(clocks.window(t_soak, clocks.t1),
                   window="1 s of the same step graph ending at the timed region (which is shorter than "
                          "the 200 ms sampling period)")
    clocks.close()
    if rank == 0:
        pk = peaks()
        cpu = cpu_baseline(wl) if world == 1 else None
        lone_gbs = bytes_per_launch / (lone_us * 1e-6) / 1e9
        roofline = {
            "bound": "hbm", "achieved": achieved_gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
            "frac": achieved_gbs / pk["hbm_gbs"], "traffic": recorded_traffic("verify_tma_kernel"),
            "peak_source": pk["source"], "kernel": "verify_tma_kernel<bf16> + select_kernel, resident inputs",
            "algorithmic_bytes_per_launch": bytes_per_launch, "pct_of_8tbs": achieved_gbs / NOMINAL_HBM_GBS,
            "launch": f"CUDA graphs of {G} steps, {asd.verify_launches(B, K, V, asd.BF16)} kernels per step; "
                      "ASD_RESIDENT_INPUTS (buffers written before the timed region; consecutive steps overlap)",
            "lone_call": {"us_per_step": lone_us, "achieved": lone_gbs, "frac": lone_gbs / pk["hbm_gbs"],
                          "launch": f"graphs of {G_lone} steps without ASD_RESIDENT_INPUTS: each step waits "
                                    "for the previous kernel before its first read"},
        }
        if lm is not None:
            roofline["fused_lmhead"] = lm["summary"]
        if other is not None:
            roofline["other_configs"] = {k: {"us": round(v["us_per_step"], 2),
                                             "frac": round(v["roofline"]["frac"], 3),
                                             "traffic": v["roofline"]["traffic"]}
                                         for k, v in other.items() if "roofline" in v}
        line = {
            "metric": METRIC, "value": value, "unit": "rows/s", "n_gpus": world, "steps": steps,
            "warmup": warmup, "ms_per_step": sec_per_step * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": bench_config(world),
            "roofline": roofline,
            "clocks": clk,
            "e2e": e2e,
            "gpu_launches": steps * asd.verify_launches(B, K, V, asd.BF16),
            "cpu_baseline": cpu,
            "interleaved_graphs_us_per_step": interleaved,
            "noalloc": noalloc,
            "fused_lmhead": lm["detail"] if lm is not None else None,
            "next_rows": nxt,
            "other_configs": other,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_noalloc(wl, dev, calls: int = 200) -> dict:
    """asd_verify_noalloc against asd_verify on the same steps, both eager on one stream."""
    from paper_2608_03447_gb300 import asd
    stream = torch.cuda.current_stream(dev)
    out = asd.alloc_outputs(B, K, dev)

    def run(fn):
        for i in range(3):
            fn(i)
        torch.cuda.synchronize(dev)
        s_, e_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s_.record(stream)
        for i in range(calls):
            fn(i)
        e_.record(stream)
        e_.synchronize()
        return s_.elapsed_time(e_) * 1e3 / calls

    def with_ws(i):
        k = i % wl.nbuf
        asd.verify(wl.logits[k], wl.drafts[k], wl.ledger, GATE, CAP, wl.workspace, out, resident=True)

    def without(i):
        k = i % wl.nbuf
        asd.verify_noalloc(wl.logits[k], wl.drafts[k], wl.ledger, GATE, CAP, out, resident=True)

    us_ws = run(with_ws)
    us_na = run(without)
    wl.reset_ledger()
    return {"verify_us_per_call": us_ws, "noalloc_us_per_call": us_na,
            "note": f"{calls} eager calls each (host launch overhead included), resident inputs; the "
                    "allocation-free call clears its scratch with a memset before its kernels"}


def run_e2e(wl, dev, steps: int, world: int) -> dict:
    """The same step through asd.verify_from_host: pinned host logits and drafts read in place by the
    kernels over the host link, the per-request results copied back to pinned host memory."""
    from paper_2608_03447_gb300 import asd
    import torch.distributed as dist
    host_logits = [wl.logits[i].cpu().pin_memory() for i in range(2)]
    host_draft = [wl.drafts[i].cpu().pin_memory() for i in range(2)]
    host_out = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True)
                for k, v in wl.out.items() if k in ("accepted_len", "committed", "recovery")}
    stream = torch.cuda.current_stream(dev)
    for i in range(3):
        asd.verify_from_host(host_logits[i % 2], host_draft[i % 2], wl.ledger, GATE, CAP, wl.workspace, wl.out,
                             host_out, resident=True)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for i in range(steps):
        asd.verify_from_host(host_logits[i % 2], host_draft[i % 2], wl.ledger, GATE, CAP, wl.workspace, wl.out,
                             host_out, resident=True)
    end.record(stream)
    end.synchronize()
    sec = max_over_ranks(start.elapsed_time(end), dev, world) / 1e3
    h2d = host_logits[0].numel() * host_logits[0].element_size() + host_draft[0].numel() * 4
    d2h = sum(v.numel() * v.element_size() for v in host_out.values())
    return {"value": job_rows_per_s(world, B * (K + 1), steps, sec), "unit": "rows/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps, "host_link_gbs": h2d * steps / sec / 1e9,
            "transfer": "kernels read the pinned host logits and drafts in place over the host link"}


def _time(fn, dev, iters: int) -> float:
    """Mean ms per call of fn over `iters` calls after 3 warm-up calls (CUDA events)."""
    for _ in range(3):
        fn()
    torch.cuda.synchronize(dev)
    stream = torch.cuda.current_stream(dev)
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record(stream)
    for _ in range(iters):
        fn()
    e.record(stream)
    e.synchronize()
    return s.elapsed_time(e) / iters


def _time_graph(fn, dev, per_graph: int, replays: int = 5) -> float:
    """Mean ms per call of fn, with `per_graph` calls captured in one CUDA graph (launch cost off the host)."""
    fn()
    torch.cuda.synchronize(dev)
    side = torch.cuda.Stream(dev)
    side.wait_stream(torch.cuda.current_stream(dev))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        for _ in range(per_graph):
            fn()
    for _ in range(2):
        graph.replay()
    torch.cuda.synchronize(dev)
    stream = torch.cuda.current_stream(dev)
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record(stream)
    for _ in range(replays):
        graph.replay()
    e.record(stream)
    e.synchronize()
    return s.elapsed_time(e) / (replays * per_graph)


def run_other_configs(dev) -> dict:
    """The verify step on the other workloads of the scope table (parity cases elsewhere), timed like
    the headline: CUDA graphs of steps over rotating buffers larger than 4x L2."""
    from paper_2608_03447_gb300 import asd, inputs
    from paper_2608_03447_gb300.workload import VerifyWorkload
    pk = peaks()
    cases = [
        ("tiny-fp32", 0, 4, 8, 1024, torch.float32, 1.0, 2, 4.0, inputs.MIX_DEFAULT, None),
        ("budget-cap-sweep bf16 (g=1, M=2, budget=8)", 2, 128, 16, 151936, torch.bfloat16, 1.0, 2, 8.0,
         inputs.MIX_DEFAULT, "budget-cap-sweep"),
        ("large-batch-129k fp32 (p_hit=0.7)", 3, 256, 4, 129280, torch.float32, 1.0, 1, 4.0, inputs.mix_for_hit(0.7),
         "large-batch-129k-f32"),
        ("large-batch-129k bf16 (p_hit=0.7)", 3, 256, 4, 129280, torch.bfloat16, 1.0, 1, 4.0, inputs.mix_for_hit(0.7),
         "large-batch-129k-bf16"),
    ]
    out = {}
    for name, cfg, b, k, v, dtype, gate, cap, budget, mix, traffic_key in cases:
        wl = VerifyWorkload(b, k, v, dtype, gate, cap, budget, config=cfg, mix=mix, device=dev, resident=True)
        steps = 200 if wl.bytes_per_step > (1 << 26) else 2000
        graph = wl.capture(steps)
        for _ in range(3):
            graph.replay()
        torch.cuda.synchronize(dev)
        stream = torch.cuda.current_stream(dev)
        s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s.record(stream)
        graph.replay()
        e.record(stream)
        e.synchronize()
        sec = s.elapsed_time(e) / 1e3 / steps
        gbs = wl.bytes_per_step / sec / 1e9
        code = asd.BF16 if dtype == torch.bfloat16 else asd.F32
        rec = {"config": cfg, "B": b, "K": k, "V": v, "dtype": "bf16" if dtype == torch.bfloat16 else "f32",
               "us_per_step": sec * 1e6, "rows_per_s": b * (k + 1) / sec, "hbm_gbs": gbs,
               "kernels_per_step": asd.verify_launches(b, k, v, code), "buffers": wl.nbuf, "steps": steps}
        if wl.bytes_per_step > (1 << 26):
            rec["roofline"] = {"bound": "hbm", "achieved": gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
                               "frac": gbs / pk["hbm_gbs"],
                               "traffic": recorded_traffic("verify_tma_kernel", traffic_key),
                               "algorithmic_bytes_per_launch": wl.bytes_per_step}
        else:
            rec["bound"] = "launch latency (147 KB per call)"
        out[name] = rec
        del graph, wl
        torch.cuda.empty_cache()
    return out


def run_next_rows(wl, dev) -> dict:
    """Throughput of the rows beyond the single-block step, on the same workload's buffers."""
    from paper_2608_03447_gb300 import asd
    from paper_2608_03447_gb300.workload import l2_bytes
    pk = peaks()
    out = {}
    # multi-block: all rotating buffers as one call of nblk sequential blocks (> 4x L2 per call)
    nblk = wl.nbuf
    logits = torch.stack(wl.logits).contiguous()
    drafts = torch.stack(wl.drafts).contiguous()
    led = asd.make_ledger(B, BUDGET, 0.0, dev)
    ws = asd.blocks_workspace(nblk, B, K, V, asd.BF16, dev)
    flat = asd.alloc_outputs(nblk * B, K, dev)
    res = {k: v.view(nblk, B, *v.shape[1:]) for k, v in flat.items()}
    ms = _time(lambda: asd.verify_blocks(logits, drafts, led, GATE, CAP, ws, res, resident=True), dev, 30)
    gbs = logits.numel() * 2 / (ms * 1e-3) / 1e9
    out["multi_block"] = {"workload": f"{nblk} sequential blocks of the step's batch per call", "ms_per_call": ms,
                          "rows_per_s": nblk * B * (K + 1) / (ms * 1e-3), "hbm_gbs": gbs,
                          "roofline": {"bound": "hbm", "achieved": gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
                                       "frac": gbs / pk["hbm_gbs"]}}
    del logits, drafts, flat, res
    # vocabulary-sharded verify: 4 shards per block, partials then combine
    S = 4
    bounds = [round(V * i / S) for i in range(S + 1)]
    shards = [[wl.logits[k][:, :, bounds[i]:bounds[i + 1]].contiguous() for i in range(S)] for k in range(wl.nbuf)]
    parts = torch.empty(S, B * (K + 1), asd.PARTIAL_WORDS, dtype=torch.int32, device=dev)
    sws = [asd.Workspace(B, K, bounds[i + 1] - bounds[i], asd.BF16, dev) for i in range(S)]
    sled = asd.make_ledger(B, BUDGET, 0.0, dev)
    sout = asd.alloc_outputs(B, K, dev)
    step = [0]
    # each shard on its own stream (graph branches that run side by side, as the ranks would),
    # joined before the combine
    rank_streams = [torch.cuda.Stream(dev) for _ in range(S)]

    def sharded():
        k = step[0] % wl.nbuf
        step[0] += 1
        main = torch.cuda.current_stream(dev)
        for i in range(S):
            rank_streams[i].wait_stream(main)
            with torch.cuda.stream(rank_streams[i]):
                asd.shard_partials(shards[k][i], wl.drafts[k], bounds[i], V, sws[i], parts[i], resident=True)
        for i in range(S):
            main.wait_stream(rank_streams[i])
        asd.shard_combine(parts, wl.drafts[k], sled, GATE, CAP, V, sout)

    ms = _time_graph(sharded, dev, 4 * wl.nbuf)
    gbs = B * (K + 1) * V * 2 / (ms * 1e-3) / 1e9
    shard_launches = sum(asd.verify_launches(B, K, bounds[i + 1] - bounds[i], asd.BF16) for i in range(S))
    # what one tensor-parallel rank runs: its shard's partials (over rotating shard buffers > 4x L2),
    # then, after the all-gather of partials, the combine and selection
    vs = bounds[1] - bounds[0]
    shard_bytes = B * (K + 1) * vs * 2
    nrot = max(2, -(-4 * l2_bytes(dev) // shard_bytes))
    rank_logits = [wl.logits[k % wl.nbuf][:, :, bounds[(k // wl.nbuf) % S]:bounds[(k // wl.nbuf) % S] + vs]
                   .contiguous() for k in range(nrot)]
    rstep = [0]

    def one_rank():
        k = rstep[0] % nrot
        rstep[0] += 1
        asd.shard_partials(rank_logits[k], wl.drafts[k % wl.nbuf], 0, V, sws[0], parts[0], resident=True)

    ms_rank = _time_graph(one_rank, dev, 4 * nrot)
    ms_combine = _time_graph(lambda: asd.shard_combine(parts, wl.drafts[0], sled, GATE, CAP, V, sout), dev, 100)
    rank_gbs = shard_bytes / (ms_rank * 1e-3) / 1e9
    del rank_logits
    out["vocab_sharded"] = {
        "workload": f"{S} vocabulary shards of the step's logits (tensor-parallel ranks), partials + all-gather "
                    "of 24-byte partials + combine",
        "per_rank": {"partials_us": ms_rank * 1e3, "combine_us": ms_combine * 1e3, "shard_bytes": shard_bytes,
                     "hbm_gbs": rank_gbs,
                     "roofline": {"bound": "hbm", "achieved": rank_gbs, "peak": pk["hbm_gbs"], "unit": "GB/s",
                                  "frac": rank_gbs / pk["hbm_gbs"]},
                     "note": "the all-gather between the two needs several GPUs and is not timed here"},
        "all_shards_on_one_gpu": {"ms_per_step": ms, "rows_per_s": B * (K + 1) / (ms * 1e-3), "hbm_gbs": gbs,
                                  "launches_per_step": shard_launches + 1,
                                  "note": "emulation: the four shards share one GPU's SMs and HBM"}}
    del shards
    # opportunity counts and history advance on the step's outputs (latency-bound, one launch each)
    rows = asd.alloc_outputs(B, K, dev)
    asd.verify(wl.logits[0], wl.drafts[0], asd.make_ledger(B, BUDGET, 0.0, dev), GATE, CAP, wl.workspace, rows)
    counts = torch.zeros(4 * 4 + 1, dtype=torch.int64, device=dev)
    ms = _time_graph(lambda: asd.opportunity(rows["row_argmax"], wl.drafts[0], rows["row_regret"],
                                             [0.25, 0.5, 1.0, 2.0], [1, 2, 3, 4], counts=counts), dev, 100)
    out["opportunity"] = {"workload": "Eq. 4 counts over the step's 32 x 8 positions, 4 taus x 4 ps",
                          "us_per_call": ms * 1e3, "bound": "launch latency (graph of 100 calls)"}
    tokens = torch.zeros(B, 4096, dtype=torch.int32, device=dev)
    tlen = torch.zeros(B, dtype=torch.int32, device=dev)
    kv = torch.zeros(B, dtype=torch.int32, device=dev)

    def commit():
        tlen.zero_()
        asd.commit(rows["accepted_len"], rows["committed"], 1, kv, tokens, tlen)

    ms = _time_graph(commit, dev, 100)
    out["commit"] = {"workload": "append the step's emitted tokens and advance 32 KV lengths (with a zeroing of "
                                 "the history length per call)", "us_per_call": ms * 1e3,
                     "bound": "launch latency (graph of 100 calls)"}
    return out


CASES = {
    # name: (config, B, K, V, dtype, resident, forced path)
    "verify-qwen3": (1, 32, 8, 151936, "bf16", True, "auto"),
    "verify-qwen3-lone": (1, 32, 8, 151936, "bf16", False, "auto"),
    "verify-qwen3-stream": (1, 32, 8, 151936, "bf16", True, "stream"),
    "verify-sweep": (2, 128, 16, 151936, "bf16", True, "auto"),
    "verify-129k-f32": (3, 256, 4, 129280, "f32", True, "auto"),
    "verify-129k-bf16": (3, 256, 4, 129280, "bf16", True, "auto"),
    "verify-tiny": (0, 4, 8, 1024, "f32", True, "auto"),
}


def run_case(name: str, launches: int) -> None:
    """A few launches of one workload and nothing else, for a profiler to capture (one GPU, small)."""
    from paper_2608_03447_gb300 import asd, inputs
    from paper_2608_03447_gb300.workload import VerifyWorkload
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    asd.load()
    if name in ("lmhead", "cublas-lmhead"):
        inp = inputs.gen_lmhead(LM_B, LM_K, LM_H, LM_V, inputs.seed_for(4), dev)
        led = asd.make_ledger(LM_B, 8.0, 0.0, dev)
        logits = torch.empty(LM_B * (LM_K + 1), LM_V, dtype=torch.bfloat16, device=dev)
        for _ in range(2 + launches):
            if name == "lmhead":
                asd.lmhead_verify(inp.hidden, inp.weight, inp.draft, led, 1.0, 2)
            else:  # the library GEMM of the same shape (bf16 logits out, no reduction), for comparison
                torch.matmul(inp.hidden, inp.weight.t(), out=logits)
        torch.cuda.synchronize(dev)
        print(json.dumps({"case": name, "launches": 2 + launches}))
        return
    control = name.startswith("torch-amax:")
    cfg, b, k, v, dt, resident, path = CASES[name.split(":", 1)[1] if control else name]
    dtype = torch.bfloat16 if dt == "bf16" else torch.float32
    mix = inputs.mix_for_hit(0.7) if cfg == 3 else inputs.MIX_DEFAULT
    wl = VerifyWorkload(b, k, v, dtype, GATE, CAP, BUDGET, config=cfg, mix=mix, device=dev, resident=resident)
    asd.set_launch_options(path=path)
    for i in range(2 + launches):
        if control:  # the same bytes through a library row reduction, for comparison
            torch.amax(wl.logits[i % wl.nbuf], dim=-1)
        else:
            wl.step(i)
    torch.cuda.synchronize(dev)
    asd.reset_launch_options()
    print(json.dumps({"case": name, "launches": 2 + launches, "bytes_per_launch": wl.bytes_per_step,
                      "buffers": wl.nbuf}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="asd", choices=["asd", "reference"])
    ap.add_argument("--case", default=None,
                    help="run only a few launches of one workload (for ncu): " + ", ".join(
                        list(CASES) + ["lmhead", "cublas-lmhead"] + [f"torch-amax:{c}" for c in CASES]))
    ap.add_argument("--launches", type=int, default=3)
    ap.add_argument("--no-configs", dest="configs", action="store_false",
                    help="skip timing the other workloads (configs 0, 2, 3)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.case is not None:
        run_case(args.case, args.launches)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
