"""Seeded synthetic workloads for one structured-suffix denoising step.

This module only draws inputs: it holds the five workload shapes and the
seeded generators that both the CUDA path and the CPU oracle consume.  It
contains none of the method's arithmetic (no selection, mixing, attention
or unmasking), so the two implementations share nothing but their inputs.

The shapes follow the paper's experimental settings (Sec. 4.1: block 32,
confidence threshold 0.9, generation lengths 256/512/1024; Table 4: 1024-token
long-sequence runs with a prefix cache) on LLaDA-8B / Dream-7B-shaped layers.
The benchmark datasets and trained weights are not available, so every tensor
is drawn from a fixed distribution (recipe in ``draw_*`` below).
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import torch

LLADA_VOCAB = 126464


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    seed: int
    h_q: int
    h_kv: int
    head_dim: int
    prompt: int
    gen: int
    block: int
    local: int
    middle: int
    tail: int
    batch: int
    vocab: int
    logits_dtype: str          # "f32" or "bf16"
    logits_sigma: float
    rope_theta: float
    prefix_cached: bool        # True: prompt K/V come from a cache; False: prompt rows are recomputed
    block_indices: tuple = (0,)
    threshold: float = 0.9
    topk: int = 5              # previous-step candidates per retained suffix position (Eq. 6)
    alpha: float = 0.4         # mixing ratio of Eq. 8

    @property
    def hidden(self) -> int:
        return self.h_q * self.head_dim

    @property
    def n_blocks(self) -> int:
        return self.gen // self.block


WORKLOADS = {
    "tiny": Workload("tiny", 0, 4, 4, 64, 64, 256, 32, 32, 8, 4, 1, 4096, "f32", 3.0,
                     10000.0, True),
    "llada": Workload("llada", 1, 32, 32, 128, 512, 256, 32, 32, 16, 8, 1, LLADA_VOCAB, "bf16",
                      4.0, 500000.0, False),
    "dream": Workload("dream", 2, 28, 4, 128, 512, 1024, 32, 64, 32, 8, 4, LLADA_VOCAB, "bf16",
                      4.0, 1.0e6, True),
    "long": Workload("long", 3, 32, 32, 128, 1024, 2048, 32, 64, 64, 16, 1, LLADA_VOCAB, "bf16",
                     4.0, 500000.0, True, block_indices=tuple(range(64))),
    "serve": Workload("serve", 4, 32, 32, 128, 512, 1024, 32, 32, 32, 8, 8, LLADA_VOCAB, "bf16",
                      4.0, 500000.0, True),
}


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def draw_normal_bf16(shape, sigma: float, seed: int, device="cpu") -> torch.Tensor:
    """N(0, sigma^2) draws (std sigma, torch convention), rounded to bf16."""
    g = _gen(seed, device)
    return (torch.randn(shape, generator=g, device=device, dtype=torch.float32) * sigma).to(torch.bfloat16)


def draw_normal_f32(shape, sigma: float, seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed, device)
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32) * sigma


def draw_block_tokens(batch: int, block: int, vocab: int, mask_id: int, masked_frac: float,
                      seed: int, device="cpu") -> torch.Tensor:
    """Current-block token ids: a seeded fraction is [MASK], the rest random committed ids.

    masked_frac = 1.0 is the first step of a block (every position masked).
    """
    g = _gen(seed, device)
    ids = torch.randint(0, vocab - 1, (batch, block), generator=g, device=device, dtype=torch.int64)
    u = torch.rand((batch, block), generator=g, device=device)
    ids = torch.where(u < masked_frac, torch.full_like(ids, mask_id), ids)
    return ids.to(torch.int32)


def draw_prev_topk(rows: int, k: int, vocab: int, seed: int, device="cpu",
                   no_pred_frac: float = 0.0):
    """Stand-in for the previous step's top-k prediction at each retained suffix position.

    ids: k distinct uniform ids per row (id -1 marks "no prediction");
    probs: a sorted softmax of N(0, 3^2) draws, scaled by a mass u ~ U(0.2, 1] so
    that the k values look like full-vocabulary probabilities (sum <= 1).
    """
    g = _gen(seed, device)
    scores = torch.rand((rows, vocab), generator=g, device="cpu") if vocab <= 8192 else None
    if scores is not None:
        ids = torch.topk(scores, k, dim=1).indices
    else:
        # distinct ids without a rows x vocab matrix: sample with rejection of duplicates
        ids = torch.randint(0, vocab, (rows, k), generator=g, device="cpu")
        for _ in range(8):
            s, _ = torch.sort(ids, dim=1)
            dup = (s[:, 1:] == s[:, :-1]).any(dim=1)
            if not bool(dup.any()):
                break
            ids[dup] = torch.randint(0, vocab, (int(dup.sum()), k), generator=g, device="cpu")
    z = torch.randn((rows, k), generator=g) * 3.0
    p = torch.softmax(z, dim=1)
    p, _ = torch.sort(p, dim=1, descending=True)
    mass = 0.2 + 0.8 * torch.rand((rows, 1), generator=g)
    probs = (p * mass).to(torch.float32)
    if no_pred_frac > 0:
        none = torch.rand((rows,), generator=g) < no_pred_frac
        ids[none] = -1
    return ids.to(torch.int32).to(device), probs.to(device)


def draw_logits(shape, dtype: str, sigma: float, seed: int, device="cpu",
                planted_frac: float = 0.0, planted_boost: float = 20.0) -> torch.Tensor:
    """Per-position vocabulary logits ~ N(0, sigma^2); a planted fraction of rows gets
    +planted_boost on one random id so that its max probability clears the threshold."""
    g = _gen(seed, device)
    x = torch.randn(shape, generator=g, device=device, dtype=torch.float32) * sigma
    if planted_frac > 0:
        rows = x.reshape(-1, shape[-1])
        gc = _gen(seed + 7919, "cpu")
        sel = torch.rand((rows.shape[0],), generator=gc) < planted_frac
        ids = torch.randint(0, shape[-1], (rows.shape[0],), generator=gc)
        r = torch.nonzero(sel).flatten()
        rows[r.to(device), ids[r].to(device)] += planted_boost
    if dtype == "bf16":
        return x.to(torch.bfloat16)
    return x


def block_start(w: Workload, b: int) -> int:
    """Absolute position of the first token of block b (the prompt occupies [0, prompt))."""
    return w.prompt + b * w.block
