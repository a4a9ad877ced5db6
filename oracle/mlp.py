"""float64 oracle for the gate-up projection of the decoder MLP.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): the product path never
imports this module.

What is computed
----------------
Section 6.1 profiles the "fused gate-up projection" of a decoder block next to
attention, for the same prompt processed as 2k and as 16k chunks.  The paper
does not write the operation out; Qwen2.5 models use a SwiGLU MLP whose first
half is that projection: one matrix product of the chunk's hidden states
``X`` [T, H] with the stacked gate and up weights ``W`` [2 I, H] (rows
``0 .. I-1`` gate, ``I .. 2I-1`` up), followed by the gated activation

    Y = silu(X W_gate^T) * (X W_up^T),   silu(a) = a / (1 + exp(-a)),

giving ``Y`` [T, I].  Every token row is independent, so a chunked prompt
gives the same rows as the whole prompt.  Arithmetic is float64 on the
widened bf16 inputs: one matrix product per half, an elementwise silu and
product, nothing fused or reordered.
"""
from __future__ import annotations

import numpy as np


def silu(a: np.ndarray) -> np.ndarray:
    """silu(a) = a * sigmoid(a), written as a / (1 + exp(-a))."""
    a = np.asarray(a, dtype=np.float64)
    return a / (1.0 + np.exp(-a))


def gate_up(x: np.ndarray, w: np.ndarray) -> np.ndarray:
    """Y = silu(X W_gate^T) * (X W_up^T) for X [T, H] and W = [W_gate; W_up] [2I, H]."""
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    inter = w.shape[0] // 2
    gate = x @ w[:inter].T
    up = x @ w[inter:].T
    return silu(gate) * up


def gate_up_rows(x: np.ndarray, w: np.ndarray, rows) -> np.ndarray:
    """The same for a subset of token rows (each row is independent)."""
    rows = np.asarray(rows, dtype=np.int64)
    return gate_up(np.asarray(x)[rows], w)
