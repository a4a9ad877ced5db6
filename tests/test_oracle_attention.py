"""Pins for the float64 attention oracle (CPU only).

Each pin checks the oracle against something other than itself: a brute
force written from the definition on tiny inputs, torch's own
``scaled_dot_product_attention`` (a library routine with its own default
scale and causal convention), closed forms, and invariants.
"""
import math

import numpy as np
import pytest
import torch

from oracle import attention as oa
from paper_2608_15171_gb300 import workloads as wl

PAGE = 16


def _random_paged(rng, ctxs, n_kv, d, num_blocks=None, dtype=np.float64):
    """Dense per-sequence K/V plus a paged copy scattered through a random pool."""
    need = [-(-c // PAGE) for c in ctxs]
    num_blocks = num_blocks or sum(need) + 3
    perm = rng.permutation(num_blocks)
    k_cache = rng.standard_normal((num_blocks, n_kv, PAGE, d))
    v_cache = rng.standard_normal((num_blocks, n_kv, PAGE, d))
    width = max(need)
    tables = np.full((len(ctxs), width), -1, dtype=np.int64)
    dense_k, dense_v, pos = [], [], 0
    for s, (c, n) in enumerate(zip(ctxs, need)):
        tables[s, :n] = perm[pos:pos + n]
        pos += n
        dk = rng.standard_normal((c, n_kv, d))
        dv = rng.standard_normal((c, n_kv, d))
        for j in range(c):
            k_cache[tables[s, j // PAGE], :, j % PAGE, :] = dk[j]
            v_cache[tables[s, j // PAGE], :, j % PAGE, :] = dv[j]
        dense_k.append(dk)
        dense_v.append(dv)
    return k_cache, v_cache, tables, dense_k, dense_v


def _brute_force(q, dense_k, dense_v, q_lens, ctx_lens, scale):
    """Definition written out with Python loops (tiny inputs only)."""
    n_q, d = q.shape[1], q.shape[2]
    n_kv = dense_k[0].shape[1]
    grp = n_q // n_kv
    out = np.zeros_like(q)
    row = 0
    for s, (ql, c) in enumerate(zip(q_lens, ctx_lens)):
        p = c - ql
        for t in range(ql):
            for h in range(n_q):
                g = h // grp
                scores = [scale * sum(q[row + t, h, x] * dense_k[s][j, g, x] for x in range(d))
                          for j in range(p + t + 1)]
                m = max(scores)
                e = [math.exp(v - m) for v in scores]
                z = sum(e)
                for x in range(d):
                    out[row + t, h, x] = sum(e[j] * dense_v[s][j, g, x] for j in range(len(e))) / z
        row += ql
    return out


def test_brute_force_tiny_mixed_step():
    rng = np.random.default_rng(1)
    q_lens, ctx_lens = [1, 5, 3, 1], [7, 5, 20, 17]
    n_q, n_kv, d = 4, 2, 8
    kc, vc, tables, dk, dv = _random_paged(rng, ctx_lens, n_kv, d)
    q = rng.standard_normal((sum(q_lens), n_q, d))
    scale = 1 / math.sqrt(d)
    got = oa.paged_attention(q, kc, vc, tables, q_lens, ctx_lens, scale)
    want = _brute_force(q, dk, dv, q_lens, ctx_lens, scale)
    assert np.max(np.abs(got - want)) <= 1e-12


@pytest.mark.parametrize("n_q,n_kv", [(16, 2), (32, 8), (4, 4)])
def test_matches_torch_sdpa_full_causal(n_q, n_kv):
    """Bottom-right alignment, scale and GQA mapping against torch SDPA.

    SDPA runs the whole square causal problem over all ``ctx`` positions with
    its default ``1/sqrt(D)`` scale and kv heads repeated in contiguous
    groups; the oracle gets only the last ``q`` rows through pages.
    """
    rng = np.random.default_rng(2)
    d, ctx, ql = 32, 75, 19
    kc, vc, tables, dk, dv = _random_paged(rng, [ctx], n_kv, d)
    q_all = rng.standard_normal((ctx, n_q, d))
    got = oa.paged_attention(q_all[ctx - ql:], kc, vc, tables, [ql], [ctx], 1 / math.sqrt(d))
    tq = torch.from_numpy(q_all).permute(1, 0, 2)[None]                       # [1, Hq, ctx, d]
    tk = torch.from_numpy(dk[0]).permute(1, 0, 2).repeat_interleave(n_q // n_kv, dim=0)[None]
    tv = torch.from_numpy(dv[0]).permute(1, 0, 2).repeat_interleave(n_q // n_kv, dim=0)[None]
    ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=True)
    ref = ref[0].permute(1, 0, 2).numpy()[ctx - ql:]
    assert np.max(np.abs(got - ref)) <= 1e-12


def test_chunk_invariance_2048_as_4x512():
    """Chunked prefill at MBT 512 equals one unchunked causal pass (P2)."""
    rng = np.random.default_rng(3)
    n_q, n_kv, d, L = 4, 2, 16, 2048
    nb = L // PAGE + 4
    perm = rng.permutation(nb)
    table = perm[: L // PAGE][None]
    q = rng.standard_normal((L, n_q, d))
    k = rng.standard_normal((L, n_kv, d))
    v = rng.standard_normal((L, n_kv, d))
    kc = np.zeros((nb, n_kv, PAGE, d))
    vc = np.zeros((nb, n_kv, PAGE, d))
    slots = np.array([table[0, j // PAGE] * PAGE + j % PAGE for j in range(L)])
    scale = 1 / math.sqrt(d)
    chunks = []
    for c0 in range(0, L, 512):
        oa.kv_append(k[c0:c0 + 512], v[c0:c0 + 512], slots[c0:c0 + 512], kc, vc)
        chunks.append(oa.paged_attention(q[c0:c0 + 512], kc, vc, table, [512], [c0 + 512], scale))
    whole = oa.paged_attention(q, kc, vc, table, [L], [L], scale)
    assert np.max(np.abs(np.concatenate(chunks) - whole)) <= 1e-12


def test_softmax_rows_sum_to_one_and_mask():
    rng = np.random.default_rng(4)
    q = rng.standard_normal((9, 8)) * 3
    k = rng.standard_normal((40, 8)) * 3
    pos = np.array([0, 1, 5, 16, 17, 30, 38, 39, 39])
    w = oa.softmax_weights(q, k, pos, 0.7)
    assert np.max(np.abs(w.sum(axis=1) - 1)) <= 1e-12
    for r, p in enumerate(pos):
        assert np.all(w[r, p + 1:] == 0)
        assert np.all(w[r, :p + 1] > 0)


def test_single_key_returns_first_value():
    """Row 0 of a prefix-0 chunk sees exactly one key, so O = V[0] (P4)."""
    rng = np.random.default_rng(5)
    kc, vc, tables, dk, dv = _random_paged(rng, [33], 2, 16)
    q = rng.standard_normal((33, 4, 16)) * 10
    out = oa.paged_attention(q, kc, vc, tables, [33], [33], 0.25)
    for h in range(4):
        assert np.array_equal(out[0, h], dv[0][0, h // 2])


def test_uniform_keys_give_prefix_mean_and_constant_values():
    """Identical keys give the mean of the visible values; constant values
    give that constant whatever the weights (P5)."""
    rng = np.random.default_rng(6)
    n_kv, d, ctx, ql = 1, 8, 50, 20
    kc, vc, tables, dk, dv = _random_paged(rng, [ctx], n_kv, d)
    kc[:] = rng.standard_normal(d)                     # every key the same vector
    q = rng.standard_normal((ql, 2, d))
    out = oa.paged_attention(q, kc, vc, tables, [ql], [ctx], 0.3)
    p = ctx - ql
    for t in range(ql):
        want = dv[0][: p + t + 1, 0].mean(axis=0)
        assert np.max(np.abs(out[t, 0] - want)) <= 1e-12
    vc[:] = 2.5
    out2 = oa.paged_attention(q, rng.standard_normal(kc.shape), vc, tables, [ql], [ctx], 0.3)
    assert np.max(np.abs(out2 - 2.5)) <= 1e-12


def test_page_permutation_invariance():
    """Moving pages to other physical blocks leaves the output unchanged (P6)."""
    rng = np.random.default_rng(7)
    q_lens, ctx_lens = [1, 40], [37, 70]
    kc, vc, tables, dk, dv = _random_paged(rng, ctx_lens, 2, 16)
    q = rng.standard_normal((41, 4, 16))
    a = oa.paged_attention(q, kc, vc, tables, q_lens, ctx_lens, 0.25)
    nb = kc.shape[0]
    relabel = rng.permutation(nb)                        # block b moves to relabel[b]
    kc2 = np.empty_like(kc)
    vc2 = np.empty_like(vc)
    kc2[relabel] = kc
    vc2[relabel] = vc
    t2 = np.where(tables >= 0, relabel[np.maximum(tables, 0)], -1)
    b = oa.paged_attention(q, kc2, vc2, t2, q_lens, ctx_lens, 0.25)
    assert np.array_equal(a, b)


def test_sampled_rows_agree_with_full_oracle():
    rng = np.random.default_rng(8)
    q_lens, ctx_lens = [1, 1, 30], [50, 64, 90]
    kc, vc, tables, _, _ = _random_paged(rng, ctx_lens, 2, 16)
    q = rng.standard_normal((32, 8, 16))
    full = oa.paged_attention(q, kc, vc, tables, q_lens, ctx_lens, 0.25)
    rows = [(0, 3), (1, 7), (2, 0), (17, 5), (31, 4)]
    samp = oa.sampled_rows(q, kc, vc, tables, q_lens, ctx_lens, 0.25, rows)
    for i, (r, h) in enumerate(rows):
        assert np.max(np.abs(samp[i] - full[r, h])) <= 1e-13


def test_thread_pool_matches_serial():
    rng = np.random.default_rng(9)
    q_lens, ctx_lens = [1, 300], [100, 700]
    kc, vc, tables, _, _ = _random_paged(rng, ctx_lens, 2, 16)
    q = rng.standard_normal((301, 4, 16))
    a = oa.paged_attention(q, kc, vc, tables, q_lens, ctx_lens, 0.25, row_block=64)
    b = oa.paged_attention(q, kc, vc, tables, q_lens, ctx_lens, 0.25, row_block=64, workers=4)
    assert np.array_equal(a, b)


def test_kv_append_writes_slots():
    rng = np.random.default_rng(10)
    kc = np.zeros((6, 2, PAGE, 4))
    vc = np.zeros((6, 2, PAGE, 4))
    k = rng.standard_normal((3, 2, 4))
    v = rng.standard_normal((3, 2, 4))
    slots = [5 * PAGE + 15, 0, 2 * PAGE + 7]
    oa.kv_append(k, v, slots, kc, vc)
    assert np.array_equal(kc[5, :, 15], k[0]) and np.array_equal(vc[2, :, 7], v[2])
    assert np.count_nonzero(kc) == k.size


def test_rejects_bad_lengths_and_missing_blocks():
    kc = np.zeros((2, 1, PAGE, 4))
    with pytest.raises(ValueError):
        oa.paged_attention(np.zeros((2, 1, 4)), kc, kc, np.zeros((1, 2), int), [2], [1], 1.0)
    with pytest.raises(ValueError):
        oa.paged_attention(np.zeros((1, 1, 4)), kc, kc, np.array([[0, -1]]), [1], [20], 1.0)


def test_bf16_inputs_widen_exactly():
    """The oracle consumes bf16 values exactly widened to float64."""
    x = wl.bf16_normal((4, 2, 8), seed=3)
    a = x.to(torch.float64).numpy()
    assert np.array_equal(a.astype(np.float32), x.to(torch.float32).numpy())
