"""Seeded synthetic inputs for the mixed prefill+decode attention step.

This module only draws random numbers and lays out shapes.  It holds none of
the method's arithmetic (no attention, no budget rule, no chunking), so both
the CUDA path and the CPU oracle can take their inputs from it.

Recipe (the paper's workloads have no public dataset; only lengths and
arrival processes are given):

* Q, K, V activations: float32 N(0, 1) rounded to bf16 (round-to-nearest-even
  by ``Tensor.to(torch.bfloat16)``), drawn from a ``torch.Generator`` seeded
  per tensor.
* Pages: a 16-token block pool whose free order is a seeded permutation
  (``numpy.random.default_rng(seed).permutation``); literal-shape workloads
  give each sequence consecutive runs of that order.
* Requests: Poisson arrivals (cumulative exponential gaps in integer
  microseconds from t = 0), prompt and output lengths uniform over inclusive
  integer ranges (Section 4.2 lengths: prompts 20k-30k, outputs 16-64).
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import List, Tuple

import numpy as np
import torch

PAGE_TOKENS = 16


@dataclass(frozen=True)
class Geometry:
    name: str
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    n_layers: int

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.head_dim)


QWEN25_3B = Geometry("Qwen2.5-3B", 16, 2, 128, 36)
LLAMA31_8B = Geometry("Llama-3.1-8B", 32, 8, 128, 32)


@dataclass
class StepShape:
    """One attention step: rows listed decodes first, then prefill chunks."""
    q_lens: List[int]
    ctx_lens: List[int]

    @property
    def n_seqs(self) -> int:
        return len(self.q_lens)

    @property
    def total_q(self) -> int:
        return int(sum(self.q_lens))


def bf16_normal(shape, seed: int, device="cpu") -> torch.Tensor:
    """N(0, 1) float32 draws rounded to bf16 (the activations of every workload)."""
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return torch.randn(*shape, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)


def page_permutation(num_blocks: int, seed: int) -> np.ndarray:
    return np.random.default_rng(int(seed)).permutation(num_blocks).astype(np.int32)


def blocks_for(ctx: int) -> int:
    return -(-int(ctx) // PAGE_TOKENS)


def literal_tables(shape: StepShape, free_order: np.ndarray, width: int | None = None):
    """Block tables for a literal step shape: sequence ``s`` takes the next
    ``ceil(ctx_s / 16)`` blocks of the seeded free order.  Padding is -1."""
    need = [blocks_for(c) for c in shape.ctx_lens]
    width = max(need + [1]) if width is None else width
    tables = np.full((shape.n_seqs, width), -1, dtype=np.int32)
    pos = 0
    for s, n in enumerate(need):
        if pos + n > len(free_order):
            raise ValueError("block pool too small for this step")
        tables[s, :n] = free_order[pos:pos + n]
        pos += n
    return tables


# --------------------------------------------------------------------------
# the five workloads (shapes only)
# --------------------------------------------------------------------------

def tiny_steps() -> List[StepShape]:
    """2048-token prompt prefilled as 4 chunks of 512 at MBT 512; the last
    chunk is batched with 2 decode rows of context 2048."""
    steps = [StepShape([512], [512 * (i + 1)]) for i in range(3)]
    steps.append(StepShape([1, 1, 512], [2048, 2048, 2048]))
    return steps


def low_pressure_steps() -> List[StepShape]:
    """25,000-token prompt at MBT 16384: chunks (16384, prefix 0), (8616, prefix 16384)."""
    return [StepShape([16384], [16384]), StepShape([8616], [25000])]


def high_pressure_step(seed: int = 0) -> StepShape:
    """4 prefill chunks of 512 sharing a 2048 budget, prefixes ~ U[0, 24576);
    8 decode rows with contexts ~ U[25000, 25032)."""
    rng = np.random.default_rng(int(seed))
    prefixes = rng.integers(0, 24576, size=4)
    dec = rng.integers(25000, 25032, size=8)
    return StepShape([1] * 8 + [512] * 4, [int(c) for c in dec] + [int(p) + 512 for p in prefixes])


def llama_hi_step(seed: int = 0) -> StepShape:
    """Llama-3.1-8B geometry at MBT 16384: one 16384 chunk (prefix 0) and 4
    decode rows with contexts ~ U[30000, 30064)."""
    rng = np.random.default_rng(int(seed) + 1000)
    dec = rng.integers(30000, 30064, size=4)
    return StepShape([1] * 4 + [16384], [int(c) for c in dec] + [16384])


def llama_lo_step(seed: int = 0) -> StepShape:
    """Llama-3.1-8B geometry at MBT 2048: chunks 683, 683, 682 with prefixes
    ~ U[0, 30000 - q) and 16 decode rows with contexts ~ U[30000, 30064)."""
    rng = np.random.default_rng(int(seed) + 2000)
    qs = [683, 683, 682]
    prefixes = [int(rng.integers(0, 30000 - q)) for q in qs]
    dec = rng.integers(30000, 30064, size=16)
    return StepShape([1] * 16 + qs, [int(c) for c in dec] + [p + q for p, q in zip(prefixes, qs)])


@dataclass
class RequestSpec:
    arrival_us: int
    prompt_len: int
    output_len: int


def poisson_burst(n: int, rate_per_s: float, seed: int, prompt=(20000, 30000),
                  output=(16, 64)) -> List[RequestSpec]:
    """``n`` requests with exponential inter-arrival gaps of mean ``1/rate``
    seconds, accumulated from t = 0 and floored to integer microseconds."""
    rng = np.random.default_rng(int(seed))
    gaps = rng.exponential(1.0 / float(rate_per_s), size=n)
    arrivals = np.floor(np.cumsum(gaps) * 1e6).astype(np.int64)
    prompts = rng.integers(prompt[0], prompt[1] + 1, size=n)
    outputs = rng.integers(output[0], output[1] + 1, size=n)
    return [RequestSpec(int(a), int(p), int(o)) for a, p, o in zip(arrivals, prompts, outputs)]


def bursty_trace(seed: int, burst_rate: float, steady_rate: float = 0.2, phase_s: float = 10.0,
                 duration_s: float = 50.0, prompt=(25000, 25000), output=(32, 32)) -> List[RequestSpec]:
    """Alternating steady/burst Poisson phases (Section 4.1): 10 s phases over a
    50 s trace, steady rate 0.2 req/s, burst phases at ``burst_rate``."""
    rng = np.random.default_rng(int(seed))
    out, t = [], 0.0
    n_phases = int(round(duration_s / phase_s))
    for k in range(n_phases):
        rate = steady_rate if k % 2 == 0 else burst_rate
        t0, t1 = k * phase_s, (k + 1) * phase_s
        t = t0
        while True:
            t += rng.exponential(1.0 / rate)
            if t >= t1:
                break
            out.append(t)
    prompts = rng.integers(prompt[0], prompt[1] + 1, size=len(out))
    outputs = rng.integers(output[0], output[1] + 1, size=len(out))
    return [RequestSpec(int(math.floor(a * 1e6)), int(p), int(o))
            for a, p, o in zip(out, prompts, outputs)]


def step_pairs(shape: StepShape) -> int:
    """Causal (query, key) pairs per q-head of a step: sum over rows of the
    number of keys each query sees."""
    total = 0
    for q, c in zip(shape.q_lens, shape.ctx_lens):
        p = c - q
        total += q * p + q * (q + 1) // 2
    return total


def step_flops(shape: StepShape, geo: Geometry) -> int:
    """Algorithmic FLOPs: 2 * D for the score and 2 * D for the weighted sum,
    per causal pair and q-head."""
    return 4 * geo.head_dim * geo.n_q_heads * step_pairs(shape)


def step_bytes(shape: StepShape, geo: Geometry, out_bytes: int = 2) -> int:
    """Algorithmic bytes: Q read, K and V read once per (sequence, kv-head,
    context token), O written."""
    tq = shape.total_q
    kv = sum(shape.ctx_lens) * geo.n_kv_heads * geo.head_dim * 2 * 2
    return tq * geo.n_q_heads * geo.head_dim * (2 + out_bytes) + kv
