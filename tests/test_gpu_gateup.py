"""Gate-up projection with the fused gated activation (Section 6.1's second
profiled kernel) against the float64 oracle: every element of small and
ragged shapes, sampled rows of the Qwen2.5-3B size (hidden 2048, intermediate
11008) at 16,384 tokens, chunk invariance (8 x 2k = one 16k pass, bitwise:
rows are independent), and the weight packing."""
import numpy as np
import pytest
import torch

from oracle import mlp
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


def _inputs(T, H, I, seed):
    x = wl.bf16_normal((T, H), seed, "cuda")
    # weights scaled to unit-variance products, rounded to bf16
    w = (wl.bf16_normal((2 * I, H), seed + 1, "cuda").float() / np.sqrt(H)).to(torch.bfloat16)
    return x, w


def _run(ppas, x, w, T, H, I):
    wp = torch.empty_like(w)
    ppas.ppas_gateup_pack(w, wp, H, I)
    y = torch.empty((T, I), dtype=torch.bfloat16, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ppas.ppas_gateup_swiglu(x, wp, y, T, H, I, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    return y, wp


def _check(got, want, what):
    got = np.asarray(got, dtype=np.float64)
    assert np.all(np.isfinite(got)), what
    # bf16 output: relative rounding 2^-8 at most
    tol = 8e-3 * np.abs(want) + 2e-3
    bad = np.abs(got - want) > tol
    assert not bad.any(), f"{what}: {int(bad.sum())} elements off, max err {np.abs(got - want).max():.3e}"


@pytest.mark.parametrize("T,H,I", [(1, 64, 128), (130, 256, 128), (300, 256, 384), (257, 512, 256)])
def test_small_shapes_every_element(ppas, T, H, I):
    x, w = _inputs(T, H, I, seed=T + H + I)
    y, _ = _run(ppas, x, w, T, H, I)
    want = mlp.gate_up(x.float().cpu().numpy(), w.float().cpu().numpy())
    _check(y.float().cpu().numpy(), want, f"T={T} H={H} I={I}")


def test_packing_layout(ppas):
    H, I = 64, 384
    # row id in two columns (id // 32, id % 32), both exact in bf16
    ids = torch.arange(2 * I, dtype=torch.float32, device="cuda")
    w = torch.zeros((2 * I, H), dtype=torch.float32, device="cuda")
    w[:, 0] = torch.div(ids, 32, rounding_mode="floor")
    w[:, 1] = ids % 32
    w = w.to(torch.bfloat16)
    wp = torch.empty_like(w)
    ppas.ppas_gateup_pack(w, wp, H, I)
    torch.cuda.synchronize()
    rows = (wp[:, 0].float() * 32 + wp[:, 1].float()).cpu().numpy()
    want = np.concatenate([np.r_[np.arange(128 * j, 128 * j + 128), np.arange(I + 128 * j, I + 128 * j + 128)]
                           for j in range(I // 128)])
    np.testing.assert_array_equal(rows, want)


def test_qwen_size_sampled_rows_and_chunk_invariance(ppas):
    T, H, I = 16384, 2048, 11008
    x, w = _inputs(T, H, I, seed=5)
    y, wp = _run(ppas, x, w, T, H, I)
    rng = np.random.default_rng(0)
    rows = sorted(set(rng.integers(0, T, size=24).tolist()) | {0, 127, 128, T - 1})
    want = mlp.gate_up_rows(x.float().cpu().numpy(), w.float().cpu().numpy(), rows)
    _check(y[rows].float().cpu().numpy(), want, "Qwen2.5-3B size")
    # the same prompt as eight 2k chunks gives the same rows, bit for bit
    yc = torch.empty_like(y)
    for c in range(8):
        ppas.ppas_gateup_swiglu(x[c * 2048:(c + 1) * 2048], wp, yc[c * 2048:(c + 1) * 2048], 2048, H, I)
    torch.cuda.synchronize()
    assert torch.equal(yc, y)
