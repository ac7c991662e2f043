"""Seeded synthetic inputs for the ASD verifier (shared by the tests, the oracle runs and the bench).

This module holds none of the verifier's arithmetic: it never takes a maximum,
an argmax or a regret. It plants structure instead, so that the drafts hit the
target's top token, a near miss, or a random token with the stated mix.

Verify-path logits (one block of B requests, K+1 rows each, vocabulary V):
  * background  z ~ N(0, sigma^2), sigma = 3;
  * five planted slots per row, indices drawn uniformly from [0, V)
    (slot 0 "top", slots 1-4 "near misses"; slots may coincide, rarely);
  * top value   = sigma * sqrt(2 ln V) + U(0, 8)   (the expected background
    maximum plus the boost, so slot 0 is the row argmax in nearly all rows);
  * near misses = top - gap, gaps sorted U(0.5, 6); in 20 % of rows the first
    gap is U(0, 0.5) instead (near ties, some of which collapse to exact ties
    after the bf16 cast);
  * values are written slot 4 first and slot 0 last, then cast to the dtype
    (round to nearest even for bf16).
Drafts for positions j < K: slot 0 of row j with probability p_hit, one of
slots 1-4 (uniform) with probability p_near, a uniform token id otherwise.

Fused LM-head inputs: W ~ N(0, 0.02^2) [V, H] bf16; hidden states
h = n + beta * W[p]/|W[p]| + beta' * W[p']/|W[p']| with n ~ N(0, 1) [T, H],
p, p' planted token ids, beta ~ 5 + U(0, 4) (so z(p) sits about 7-13 above 0
against a background logit spread of 0.02 * sqrt(H) = 1.43) and
beta' = beta - U(0, 0.7) in 20 % of rows, beta - U(1, 4) otherwise; cast to
bf16. Drafts use the same p_hit / p_near / uniform mix over (p, p', uniform).

Exactly representable fused LM-head inputs (parity without tolerances): W and
h hold integers in {-1, 0, 1}, so every product and every partial sum is an
integer far below 2^24 and the fp32 logits are exact whatever the summation
order. Sixteen source rows of W are copied to rows at distances 1, 40, 130
and 600 (the same warp, another warp, the other SM of a pair, another pair of
the 2-SM kernel's tiling), so exact ties cross every level of the reduction.
Token t copies W[p_t] on a random 75 % of its coordinates (zeros elsewhere),
p_t a source row with probability 1/2, else uniform; drafts are p_t with
probability 0.6, else uniform. Where p_t has a lower-indexed copy the draft
differs from the target's token with zero regret.

Seeds: seed = 1000 * config + 17 * point + block.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import torch

MIX_DEFAULT = (0.6, 0.25)  # (p_hit, p_near); p_uniform = 1 - p_hit - p_near


def seed_for(config: int, point: int = 0, block: int = 0) -> int:
    return 1000 * config + 17 * point + block


def mix_for_hit(p_hit: float) -> tuple[float, float]:
    """The draft mix at acceptance p_hit: the rest splits 0.625 : 0.375 between near misses and uniform."""
    return (p_hit, 0.625 * (1.0 - p_hit))


@dataclass
class Block:
    logits: torch.Tensor   # [B, K+1, V] fp32 or bf16
    draft: torch.Tensor    # [B, K] int32


def _generator(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def gen_block(B: int, K: int, V: int, dtype: torch.dtype, seed: int, device="cpu",
              mix: tuple[float, float] = MIX_DEFAULT, sigma: float = 3.0,
              out: torch.Tensor | None = None) -> Block:
    """One block of verify inputs (see the module docstring for the recipe)."""
    dev = torch.device(device)
    g = _generator(dev, seed)
    R = B * (K + 1)
    z = torch.randn(R, V, generator=g, device=dev, dtype=torch.float32)
    z.mul_(sigma)
    slots = torch.randint(0, V, (R, 5), generator=g, device=dev)
    top = sigma * math.sqrt(2.0 * math.log(max(V, 2))) + 8.0 * torch.rand(R, generator=g, device=dev)
    gaps = 0.5 + 5.5 * torch.rand(R, 4, generator=g, device=dev)
    gaps, _ = torch.sort(gaps, dim=1)
    near_tie = torch.rand(R, generator=g, device=dev) < 0.2
    tie_gap = 0.5 * torch.rand(R, generator=g, device=dev)
    gaps[:, 0] = torch.where(near_tie, tie_gap, gaps[:, 0])
    values = torch.cat([top[:, None], top[:, None] - gaps], dim=1)
    rows = torch.arange(R, device=dev)
    for k in (4, 3, 2, 1, 0):  # slot 0 written last: it wins if slots coincide
        z[rows, slots[:, k]] = values[:, k]
    if out is not None:
        out.view(R, V).copy_(z)
        logits = out
    else:
        logits = z.to(dtype).view(B, K + 1, V)
    del z

    p_hit, p_near = mix
    pos_rows = (torch.arange(B, device=dev)[:, None] * (K + 1) + torch.arange(K, device=dev)[None, :])
    u = torch.rand(B, K, generator=g, device=dev)
    near_slot = torch.randint(1, 5, (B, K), generator=g, device=dev)
    uniform = torch.randint(0, V, (B, K), generator=g, device=dev)
    s = slots[pos_rows]  # [B, K, 5]
    hit_tok = s[:, :, 0]
    near_tok = torch.gather(s, 2, near_slot[:, :, None])[:, :, 0]
    draft = torch.where(u < p_hit, hit_tok, torch.where(u < p_hit + p_near, near_tok, uniform))
    return Block(logits=logits, draft=draft.to(torch.int32).contiguous())


@dataclass
class LMHeadInputs:
    hidden: torch.Tensor   # [B*(K+1), H] bf16
    weight: torch.Tensor   # [V, H] bf16
    draft: torch.Tensor    # [B, K] int32


def gen_weight(V: int, H: int, seed: int, device="cpu", chunk_rows: int = 16384) -> torch.Tensor:
    """LM-head weight W ~ N(0, 0.02^2), bf16, generated in row chunks to bound fp32 scratch."""
    dev = torch.device(device)
    g = _generator(dev, seed)
    W = torch.empty(V, H, dtype=torch.bfloat16, device=dev)
    for r0 in range(0, V, chunk_rows):
        r1 = min(V, r0 + chunk_rows)
        W[r0:r1] = (0.02 * torch.randn(r1 - r0, H, generator=g, device=dev)).to(torch.bfloat16)
    return W


def gen_lmhead(B: int, K: int, H: int, V: int, seed: int, device="cpu",
               mix: tuple[float, float] = MIX_DEFAULT, weight: torch.Tensor | None = None) -> LMHeadInputs:
    """Inputs of the fused LM-head verify (see the module docstring)."""
    dev = torch.device(device)
    W = weight if weight is not None else gen_weight(V, H, seed + 500_000, dev)
    g = _generator(dev, seed)
    T = B * (K + 1)
    n = torch.randn(T, H, generator=g, device=dev)
    planted = torch.randint(0, V, (T, 2), generator=g, device=dev)
    beta = 5.0 + 4.0 * torch.rand(T, generator=g, device=dev)
    near_tie = torch.rand(T, generator=g, device=dev) < 0.2
    drop = torch.where(near_tie, 0.7 * torch.rand(T, generator=g, device=dev),
                       1.0 + 3.0 * torch.rand(T, generator=g, device=dev))
    beta2 = beta - drop
    w = W[planted].float()                         # [T, 2, H]
    w = w / w.norm(dim=-1, keepdim=True)
    h = n + beta[:, None] * w[:, 0] + beta2[:, None] * w[:, 1]
    hidden = h.to(torch.bfloat16).contiguous()

    p_hit, p_near = mix
    pos_rows = (torch.arange(B, device=dev)[:, None] * (K + 1) + torch.arange(K, device=dev)[None, :])
    u = torch.rand(B, K, generator=g, device=dev)
    uniform = torch.randint(0, V, (B, K), generator=g, device=dev)
    p = planted[pos_rows]
    draft = torch.where(u < p_hit, p[:, :, 0], torch.where(u < p_hit + p_near, p[:, :, 1], uniform))
    return LMHeadInputs(hidden=hidden, weight=W, draft=draft.to(torch.int32).contiguous())


TIE_OFFSETS = (1, 40, 130, 600)


def gen_lmhead_exact(B: int, K: int, H: int, V: int, seed: int, device="cpu") -> LMHeadInputs:
    """Integer-valued fused LM-head inputs with planted exact ties (see the module docstring)."""
    dev = torch.device(device)
    g = _generator(torch.device("cpu"), seed)
    T = B * (K + 1)
    W = torch.randint(-1, 2, (V, H), generator=g).float()
    sources = torch.randint(0, V, (16,), generator=g)
    for src in sources.tolist():
        for off in TIE_OFFSETS:
            if src + off < V:
                W[src + off] = W[src]
    pick_src = torch.rand(T, generator=g) < 0.5
    p = torch.where(pick_src, sources[torch.randint(0, 16, (T,), generator=g)], torch.randint(0, V, (T,), generator=g))
    keep = torch.rand(T, H, generator=g) < 0.75
    h = torch.where(keep, W[p], torch.zeros(()))
    pos_rows = (torch.arange(B)[:, None] * (K + 1) + torch.arange(K)[None, :])
    u = torch.rand(B, K, generator=g)
    draft = torch.where(u < 0.6, p[pos_rows], torch.randint(0, V, (B, K), generator=g))
    return LMHeadInputs(hidden=h.to(torch.bfloat16).contiguous().to(dev),
                        weight=W.to(torch.bfloat16).contiguous().to(dev),
                        draft=draft.to(torch.int32).contiguous().to(dev))


# The five workloads (sizes from the paper's settings: Qwen3 vocabulary 151936,
# a DeepSeek-class vocabulary 129280, draft horizons K in {4, 8, 16}).
CONFIGS = {
    0: dict(name="tiny-fp32", B=4, K=8, V=1024, dtype=torch.float32, gate=1.0, cap=2, budget=4.0, blocks=16),
    1: dict(name="qwen3-14b-verify", B=32, K=8, V=151936, dtype=torch.bfloat16, gate=1.0, cap=2, budget=8.0, blocks=256),
    2: dict(name="budget-cap-sweep", B=128, K=16, V=151936, dtype=torch.bfloat16,
            gates=(0.0, 0.5, 1.0, 2.0), caps=(0, 1, 2, 4), budgets=(0.0, 2.0, 8.0, 32.0), blocks=16),
    3: dict(name="large-batch-129k", B=256, K=4, V=129280, dtypes=(torch.float32, torch.bfloat16),
            hits=(0.3, 0.5, 0.7, 0.9), gate=1.0, cap=1, budget=4.0, blocks=64),
    4: dict(name="fused-lmhead", B=64, K=8, H=5120, V=151936, gate=1.0, cap=2, budget=8.0),
}
