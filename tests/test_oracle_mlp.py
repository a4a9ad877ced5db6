"""Pins of the gate-up projection oracle (CPU): hand-worked values, silu's
closed forms and symmetries, brute-force dot products, row independence
(chunk invariance) and the gate/up split of the stacked weight."""
import math

import numpy as np
import pytest

from oracle import mlp


def test_silu_closed_forms():
    assert mlp.silu(np.array([0.0]))[0] == 0.0
    # silu(a) - silu(-a) = a   (sigmoid(a) + sigmoid(-a) = 1)
    a = np.linspace(-20, 20, 81)
    np.testing.assert_allclose(mlp.silu(a) - mlp.silu(-a), a, rtol=0, atol=1e-12)
    # limits: ~a for large a, ~0 for very negative a
    assert abs(mlp.silu(np.array([40.0]))[0] - 40.0) < 1e-12
    assert abs(mlp.silu(np.array([-40.0]))[0]) < 1e-15
    # a worked value: silu(1) = 1 / (1 + e^-1)
    assert mlp.silu(np.array([1.0]))[0] == pytest.approx(1.0 / (1.0 + math.exp(-1.0)), abs=1e-15)


def test_gate_up_brute_force_small():
    rng = np.random.default_rng(0)
    T, H, I = 3, 5, 4
    x = rng.standard_normal((T, H))
    w = rng.standard_normal((2 * I, H))
    y = mlp.gate_up(x, w)
    for t in range(T):
        for i in range(I):
            g = sum(x[t, k] * w[i, k] for k in range(H))
            u = sum(x[t, k] * w[I + i, k] for k in range(H))
            assert y[t, i] == pytest.approx(g / (1 + math.exp(-g)) * u, rel=1e-12, abs=1e-12)


def test_gate_and_up_halves_are_not_swapped():
    # with X = e_0, W_gate row i = (i, ...) and W_up row i = (1, ...):
    # Y[0, i] = silu(i) * 1
    H, I = 3, 4
    x = np.zeros((1, H)); x[0, 0] = 1.0
    w = np.zeros((2 * I, H))
    w[:I, 0] = np.arange(I)
    w[I:, 0] = 1.0
    np.testing.assert_allclose(mlp.gate_up(x, w)[0], mlp.silu(np.arange(I, dtype=float)), rtol=0, atol=1e-15)
    # swapping the halves gives silu(1) * i instead
    w2 = np.concatenate([w[I:], w[:I]])
    np.testing.assert_allclose(mlp.gate_up(x, w2)[0], mlp.silu(np.ones(I)) * np.arange(I), rtol=0, atol=1e-15)


def test_rows_are_independent_chunk_invariance():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((64, 16))
    w = rng.standard_normal((24, 16))
    whole = mlp.gate_up(x, w)
    chunks = np.concatenate([mlp.gate_up(x[i:i + 16], w) for i in range(0, 64, 16)])
    np.testing.assert_array_equal(whole, chunks)
    np.testing.assert_array_equal(mlp.gate_up_rows(x, w, [5, 40]), whole[[5, 40]])
