"""Device-resident verify workloads: rotating logit buffers, a persistent ledger, captured steps.

A "step" is one asd_verify call over one batch of draft blocks. Consecutive
steps read different logit buffers (``nbuf`` of them, together several times
the L2 size), so every step streams its logits from HBM, and they carry the
ledger from step to step as a serving loop would.
"""
from __future__ import annotations

import torch

from . import asd, inputs


def l2_bytes(device=None) -> int:
    props = torch.cuda.get_device_properties(device or torch.cuda.current_device())
    return int(getattr(props, "L2_cache_size", 0) or 0)


class VerifyWorkload:
    def __init__(self, B: int, K: int, V: int, dtype: torch.dtype, gate: float, cap: int, budget: float,
                 config: int = 1, nbuf: int | None = None, min_total_bytes: int | None = None,
                 mix=inputs.MIX_DEFAULT, device="cuda", with_rows: bool = False, strict: bool = False,
                 resident: bool = False):
        self.B, self.K, self.V, self.dtype = B, K, V, dtype
        self.resident = resident  # pass ASD_RESIDENT_INPUTS: the buffers are written once, before any step
        self.gate, self.cap, self.budget, self.strict = gate, cap, budget, strict
        self.device = torch.device(device)
        elem = torch.tensor([], dtype=dtype).element_size()
        self.bytes_per_step = B * (K + 1) * V * elem
        if nbuf is None:
            need = min_total_bytes if min_total_bytes is not None else 4 * max(l2_bytes(self.device), 1)
            nbuf = max(2, -(-need // self.bytes_per_step))
        self.nbuf = nbuf
        self.logits, self.drafts = [], []
        for i in range(nbuf):
            blk = inputs.gen_block(B, K, V, dtype, inputs.seed_for(config, 0, i), self.device, mix=mix)
            self.logits.append(blk.logits)
            self.drafts.append(blk.draft)
        self.ledger0 = asd.make_ledger(B, budget, 0.0, self.device)
        self.ledger = self.ledger0.clone()
        code = asd.BF16 if dtype == torch.bfloat16 else asd.F32
        self.workspace = asd.Workspace(B, K, V, code, self.device)
        self.out = asd.alloc_outputs(B, K, self.device, with_rows=with_rows)

    def reset_ledger(self) -> None:
        self.ledger.copy_(self.ledger0)

    def step(self, i: int, stream=None) -> dict:
        k = i % self.nbuf
        if self.strict:
            return asd.verify_strict(self.logits[k], self.drafts[k], self.workspace, self.out, stream,
                                     resident=self.resident)
        return asd.verify(self.logits[k], self.drafts[k], self.ledger, self.gate, self.cap,
                          self.workspace, self.out, stream, resident=self.resident)

    def capture(self, nsteps: int, first: int = 0) -> torch.cuda.CUDAGraph:
        """Capture steps first .. first+nsteps-1 into one CUDA graph (one kernel node per step)."""
        stream = torch.cuda.Stream(self.device)
        stream.wait_stream(torch.cuda.current_stream(self.device))
        with torch.cuda.stream(stream):
            self.step(first, stream)  # the library queries the device once, outside capture
        torch.cuda.current_stream(self.device).wait_stream(stream)
        torch.cuda.synchronize(self.device)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for i in range(first, first + nsteps):
                self.step(i, torch.cuda.current_stream(self.device))
        return graph
