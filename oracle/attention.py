"""float64 oracle for one mixed prefill+decode paged causal GQA attention step.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): the product path never
imports this module.

What is computed
----------------
The paper (Section 2, prefill stores keys/values in the KV cache and decode
generates tokens one at a time; Section 6.2, prefill and decode tokens of
different requests are scheduled together in one iteration) fixes the shape
of the work but defines no attention arithmetic.  The oracle therefore takes
the plain definition of causal scaled dot-product attention and applies it to
every row of the step:

* sequence ``s`` contributes ``q_s`` query tokens that are the last ``q_s``
  positions of its context ``ctx_s``; its prefix is ``p_s = ctx_s - q_s``
  (a decode row is ``q_s = 1``);
* query token ``t`` of sequence ``s`` sits at absolute position ``p_s + t``
  (bottom-right causal alignment) and sees keys ``j = 0 .. p_s + t``;
* q-head ``h`` reads kv-head ``h // (Hq / Hkv)`` (contiguous GQA groups);
* keys/values are read from 16-token pages through the block table:
  ``K_s[j] = K_cache[table_s[j // 16], kv_head, j % 16, :]``;
* ``O[s, t, h] = sum_j softmax_j(scale * Q[s, t, h] . K_s[j]) V_s[j]``.

All arithmetic is float64 on values that are exact widenings of the bf16
inputs.  There is no blocking beyond an independent split of query rows into
row blocks (each row's result does not depend on the split), no online
softmax, no split-K.
"""
from __future__ import annotations

import concurrent.futures as _cf
import os

import numpy as np

PAGE_TOKENS = 16


def kv_head_of(h: int, n_q_heads: int, n_kv_heads: int) -> int:
    """GQA mapping: contiguous groups of ``Hq / Hkv`` q-heads share a kv-head."""
    if n_q_heads % n_kv_heads != 0:
        raise ValueError("n_q_heads must be a multiple of n_kv_heads")
    return h // (n_q_heads // n_kv_heads)


def unpage(cache: np.ndarray, table: np.ndarray, ctx: int, kv_head: int) -> np.ndarray:
    """Gather the first ``ctx`` tokens of one sequence's keys (or values).

    ``cache`` is ``[num_blocks, Hkv, 16, D]``; ``table`` lists the physical
    block of each logical 16-token block.  Returns ``[ctx, D]`` float64.
    """
    j = np.arange(ctx)
    blocks = np.asarray(table)[j // PAGE_TOKENS]
    if ctx and (blocks < 0).any():
        raise ValueError("block table has no block for a context position")
    return np.asarray(cache[blocks, kv_head, j % PAGE_TOKENS, :], dtype=np.float64)


def softmax_weights(q_rows: np.ndarray, k_seq: np.ndarray, positions: np.ndarray,
                    scale: float) -> np.ndarray:
    """Causal softmax weights ``w[r, j]`` for query rows at absolute ``positions``.

    Scores ``scale * q . k_j``; keys ``j > position`` are excluded (weight 0).
    The max is subtracted before ``exp`` (a rescaling that leaves the
    normalised weights unchanged).
    """
    q_rows = np.asarray(q_rows, dtype=np.float64)
    s = scale * (q_rows @ np.asarray(k_seq, dtype=np.float64).T)
    masked = np.arange(k_seq.shape[0])[None, :] > np.asarray(positions)[:, None]
    s[masked] = -np.inf
    m = s.max(axis=1, keepdims=True)
    e = np.exp(s - m)
    return e / e.sum(axis=1, keepdims=True)


def attention_rows(q_rows, k_seq, v_seq, positions, scale):
    """Causal attention output for a block of query rows of one (sequence, head)."""
    w = softmax_weights(q_rows, k_seq, positions, scale)
    return w @ np.asarray(v_seq, dtype=np.float64)


def _seq_bounds(q_lens, ctx_lens):
    q_lens = [int(x) for x in q_lens]
    ctx_lens = [int(x) for x in ctx_lens]
    if len(q_lens) != len(ctx_lens):
        raise ValueError("q_lens and ctx_lens differ in length")
    starts, acc = [], 0
    for q, c in zip(q_lens, ctx_lens):
        if q < 1 or c < q:
            raise ValueError("need 1 <= q_len <= ctx_len")
        starts.append(acc)
        acc += q
    return q_lens, ctx_lens, starts, acc


def paged_attention(q, k_cache, v_cache, block_tables, q_lens, ctx_lens, scale,
                    n_kv_heads=None, row_block=256, workers=1):
    """Full oracle for one attention step.

    q            : ``[sum(q_lens), Hq, D]`` query rows packed sequence after
                   sequence (float64 or anything numpy widens exactly).
    k_cache/v_cache : ``[num_blocks, Hkv, 16, D]``.
    block_tables : ``[n_seqs, width]`` physical block per logical block.
    Returns ``[sum(q_lens), Hq, D]`` float64.

    ``workers > 1`` evaluates independent (sequence, head, row-block) items on
    a thread pool; numpy releases the GIL inside its loops, and each item's
    result is the same whatever the split.
    """
    q = np.asarray(q)
    n_q_heads = q.shape[1]
    n_kv_heads = k_cache.shape[1] if n_kv_heads is None else n_kv_heads
    q_lens, ctx_lens, starts, total = _seq_bounds(q_lens, ctx_lens)
    if q.shape[0] != total:
        raise ValueError("q rows do not match sum(q_lens)")
    out = np.zeros(q.shape, dtype=np.float64)

    items = []
    for s, (ql, ctx, st) in enumerate(zip(q_lens, ctx_lens, starts)):
        for h in range(n_q_heads):
            for r0 in range(0, ql, row_block):
                items.append((s, h, r0, min(ql, r0 + row_block)))

    kv_cache_memo = {}

    def run(item):
        s, h, r0, r1 = item
        g = kv_head_of(h, n_q_heads, n_kv_heads)
        key = (s, g)
        if key not in kv_cache_memo:
            kv_cache_memo[key] = (unpage(k_cache, block_tables[s], ctx_lens[s], g),
                                  unpage(v_cache, block_tables[s], ctx_lens[s], g))
        k_seq, v_seq = kv_cache_memo[key]
        prefix = ctx_lens[s] - q_lens[s]
        positions = prefix + np.arange(r0, r1)
        rows = np.asarray(q[starts[s] + r0: starts[s] + r1, h, :], dtype=np.float64)
        out[starts[s] + r0: starts[s] + r1, h, :] = attention_rows(rows, k_seq, v_seq,
                                                                  positions, scale)

    if workers <= 1:
        for it in items:
            run(it)
    else:
        # un-page once per (sequence, kv-head) before fanning out
        for s in range(len(q_lens)):
            for g in range(n_kv_heads):
                kv_cache_memo[(s, g)] = (unpage(k_cache, block_tables[s], ctx_lens[s], g),
                                         unpage(v_cache, block_tables[s], ctx_lens[s], g))
        with _cf.ThreadPoolExecutor(max_workers=workers) as ex:
            list(ex.map(run, items))
    return out


def sampled_rows(q, k_cache, v_cache, block_tables, q_lens, ctx_lens, scale, rows,
                 n_kv_heads=None):
    """Oracle output for selected ``(packed_row, q_head)`` pairs only.

    Each sampled row is exact float64 attention over that row's whole causal
    context; nothing is approximated.  Returns ``[len(rows), D]``.
    """
    q = np.asarray(q)
    n_q_heads = q.shape[1]
    n_kv_heads = k_cache.shape[1] if n_kv_heads is None else n_kv_heads
    q_lens, ctx_lens, starts, total = _seq_bounds(q_lens, ctx_lens)
    seq_of_row = np.repeat(np.arange(len(q_lens)), q_lens)
    res = np.zeros((len(rows), q.shape[2]), dtype=np.float64)
    by_seq_head = {}
    for i, (r, h) in enumerate(rows):
        s = int(seq_of_row[r])
        by_seq_head.setdefault((s, kv_head_of(h, n_q_heads, n_kv_heads)), []).append((i, r, h))
    for (s, g), lst in by_seq_head.items():
        k_seq = unpage(k_cache, block_tables[s], ctx_lens[s], g)
        v_seq = unpage(v_cache, block_tables[s], ctx_lens[s], g)
        prefix = ctx_lens[s] - q_lens[s]
        idx = [i for i, _, _ in lst]
        qrows = np.stack([np.asarray(q[r, h, :], dtype=np.float64) for _, r, h in lst])
        pos = np.array([prefix + (r - starts[s]) for _, r, _ in lst])
        res[idx] = attention_rows(qrows, k_seq, v_seq, pos, scale)
    return res


def kv_append(k_new, v_new, slot_mapping, k_cache, v_cache):
    """Write new tokens' keys/values into their pages (in place).

    ``slot = block * 16 + offset``; ``cache[block, :, offset, :] = new[t]``.
    This is the KV-cache store that prefill and decode perform for every
    scheduled token (Section 2).
    """
    slots = np.asarray(slot_mapping, dtype=np.int64)
    blk, off = slots // PAGE_TOKENS, slots % PAGE_TOKENS
    k_cache[blk, :, off, :] = k_new
    v_cache[blk, :, off, :] = v_new


def default_workers() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1
