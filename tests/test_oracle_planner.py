"""Pins for the P-PAS planner oracle (CPU only)."""
import os
from collections import Counter

import numpy as np
import pytest

from oracle import planner as op
from paper_2608_15171_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_rows(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [ln.strip() for ln in f if ln.strip() and not ln.startswith("#")]


def test_algorithm1_truth_table():
    """Algorithm 1 at N_th = 2, B_max = 16384, B_cap = 2048."""
    rows = _read_rows("alg1_truth_table.txt")
    assert len(rows) >= 10
    for ln in rows:
        n_p, n_d, b, pr = map(int, ln.split())
        assert op.prefill_budget(n_p, n_d, op.N_TH, op.B_MAX, op.B_CAP) == (b, pr)


def _single_prompt_chunks(prompt, mbt_hi, mbt_lo, th):
    reqs = [op.Request(0, prompt, 2)]
    sched = op.Scheduler(prompt // 16 + 4, range(prompt // 16 + 4))
    chunks = []
    while reqs[0].num_computed < prompt:
        st = sched.plan_step(reqs, 0, th, mbt_hi, mbt_lo)
        assert st.n_decode == 0 and st.pressure == 0
        chunks.append(st.q_len[0])
    return chunks


def test_chunking_worked_cases():
    for ln in _read_rows("chunking_cases.txt"):
        head, tail = ln.split("|")
        prompt, hi, lo, th = map(int, head.split())
        assert _single_prompt_chunks(prompt, hi, lo, th) == [int(x) for x in tail.split()]


def _trace(seed, n=16, rate=2.0):
    return [op.Request(r.arrival_us, r.prompt_len, r.output_len)
            for r in wl.poisson_burst(n, rate, seed)]


def _check_invariants(reqs, steps, num_blocks, th, hi, lo):
    prefill_tokens = Counter()
    decode_rows = Counter()
    for now, st in steps:
        # Algorithm 1 decision and both budgets
        want_b = lo if (st.n_p >= th and st.n_d > 0) else hi
        assert st.b_prefill == want_b and st.pressure == int(want_b == lo and st.n_p >= th and st.n_d > 0)
        assert st.prefill_tokens <= st.b_prefill
        assert st.total_tokens <= hi
        assert st.total_tokens == sum(st.q_len)
        # decodes first, one token each; every running decode advances (stall-free)
        assert st.q_len[: st.n_decode] == [1] * st.n_decode
        assert st.n_decode == min(st.n_d, hi)
        assert all(q >= 1 for q in st.q_len[st.n_decode:])
        assert len(st.slot_mapping) == st.total_tokens
        assert len(set(st.slot_mapping)) == len(st.slot_mapping)
        seen_blocks = set()
        for i, q, ctx, row in zip(st.req_idx, st.q_len, st.ctx_len, st.block_table):
            held = [b for b in row if b >= 0]
            assert len(held) == -(-ctx // 16)
            assert not (set(held) & seen_blocks)
            seen_blocks |= set(held)
            r = reqs[i]
            assert r.arrival_us <= now
        for idx, (i, q) in enumerate(zip(st.req_idx, st.q_len)):
            if idx < st.n_decode:
                decode_rows[i] += 1
            else:
                prefill_tokens[i] += q
    for i, r in enumerate(reqs):
        assert r.state == op.FINISHED
        assert prefill_tokens[i] == r.prompt_len
        assert decode_rows[i] == r.output_len - 1


@pytest.mark.parametrize("rate", [0.5, 1.0, 2.0, 4.0])
def test_burst_replay_invariants(rate):
    reqs = _trace(seed=11, rate=rate)
    nb = 16 * 1879
    steps = op.replay(reqs, nb, wl.page_permutation(nb, 0))
    _check_invariants(reqs, steps, nb, op.N_TH, op.B_MAX, op.B_CAP)
    assert any(st.pressure for _, st in steps) == (rate >= 0.5 and any(
        st.n_p >= 2 and st.n_d > 0 for _, st in steps))


def test_pressure_caps_prefill_and_releases():
    """Two prefills with an active decode are capped at B_cap; once only one
    prefill is left the budget returns to B_max (re-evaluated each step)."""
    reqs = [op.Request(0, 100, 5), op.Request(1, 9000, 2), op.Request(2, 9000, 2)]
    sched = op.Scheduler(4096, range(4096))
    st = sched.plan_step(reqs, 0)                  # only request 0 arrived
    assert st.q_len == [100] and st.b_prefill == op.B_MAX
    st = sched.plan_step(reqs, 10)                 # 1 decode + 2 prefills -> capped
    assert st.pressure == 1 and st.b_prefill == op.B_CAP
    assert st.q_len == [1, 2048] and st.req_idx == [0, 1]
    for _ in range(3):
        st = sched.plan_step(reqs, 10)
        assert st.q_len == [1, 2048]
    st = sched.plan_step(reqs, 10)                 # request 0 finished after 4 decodes
    assert st.n_decode == 0 and st.b_prefill == op.B_MAX
    assert st.q_len == [9000 - 4 * 2048, 9000]


def test_static_mbt_special_cases():
    reqs = _trace(seed=3, rate=4.0)
    nb = 16 * 1879
    steps = op.replay(reqs, nb, wl.page_permutation(nb, 1), threshold=2, mbt_hi=2048, mbt_lo=2048)
    assert all(st.b_prefill == 2048 for _, st in steps)
    reqs = _trace(seed=3, rate=4.0)
    steps = op.replay(reqs, nb, wl.page_permutation(nb, 1), threshold=10 ** 6)
    assert all(st.b_prefill == 16384 and st.pressure == 0 for _, st in steps)


def test_fifo_free_list_reuse_order():
    """Finished requests return their blocks to the tail at the next call."""
    reqs = [op.Request(0, 32, 1), op.Request(0, 16, 1)]
    sched = op.Scheduler(5, [4, 3, 2, 1, 0])
    st = sched.plan_step(reqs, 0)
    assert st.block_table == [[4, 3], [2, -1]]
    assert st.slot_mapping == [4 * 16 + i for i in range(16)] + [3 * 16 + i for i in range(16)] + \
        [2 * 16 + i for i in range(16)]
    assert all(r.state == op.FINISHED for r in reqs)
    reqs.append(op.Request(5, 80, 1))
    st = sched.plan_step(reqs, 5)
    assert st.block_table == [[1, 0, 4, 3, 2]]


def test_out_of_blocks_raises_without_partial_allocation():
    reqs = [op.Request(0, 64, 3)]
    sched = op.Scheduler(3, [0, 1, 2])
    with pytest.raises(op.OutOfBlocks):
        sched.plan_step(reqs, 0)
    assert list(sched.free) == [0, 1, 2] and reqs[0].blocks == []


def test_decode_context_counts_own_token():
    reqs = [op.Request(0, 20, 3)]
    sched = op.Scheduler(8, range(8))
    st = sched.plan_step(reqs, 0)
    assert st.q_len == [20] and st.ctx_len == [20] and reqs[0].num_generated == 1
    st = sched.plan_step(reqs, 0)
    assert st.q_len == [1] and st.ctx_len == [21] and st.slot_mapping == [1 * 16 + 4]
    st = sched.plan_step(reqs, 0)
    assert st.ctx_len == [22] and reqs[0].state == op.FINISHED


def test_bad_arguments():
    sched = op.Scheduler(4, range(4))
    with pytest.raises(ValueError):
        sched.plan_step([], 0, threshold=0)
    with pytest.raises(ValueError):
        sched.plan_step([], 0, mbt_hi=100, mbt_lo=200)
    with pytest.raises(ValueError):
        op.Scheduler(3, [0, 0, 1])


def test_replay_with_logged_durations():
    """Durations equal to the clock rule reproduce the default replay; other
    durations shift arrivals relative to the plan and still satisfy every
    replay invariant."""
    specs = wl.poisson_burst(8, 2.0, seed=3, prompt=(3000, 9000), output=(2, 6))
    nb = sum(wl.blocks_for(s.prompt_len + s.output_len) for s in specs) + 8
    order = wl.page_permutation(nb, 3)
    mk = lambda: [op.Request(s.arrival_us, s.prompt_len, s.output_len) for s in specs]
    ref = op.replay(mk(), nb, order, mbt_hi=4096, mbt_lo=1024)
    rule = [op.STEP_BASE_US + op.STEP_US_PER_PREFILL_TOKEN * st.prefill_tokens for _, st in ref]
    same = op.replay(mk(), nb, order, mbt_hi=4096, mbt_lo=1024, durations=rule)
    assert [(t, st.q_len, st.ctx_len, st.slot_mapping) for t, st in same] == \
           [(t, st.q_len, st.ctx_len, st.slot_mapping) for t, st in ref]
    # a fast clock (every step 1 ms): every request still gets exactly its
    # prompt and output_len - 1 decodes
    reqs = mk()
    fast = op.replay(reqs, nb, order, mbt_hi=4096, mbt_lo=1024, durations=[1000] * 100000)
    times = [t for t, _ in fast]
    assert all(b - a >= 1000 for a, b in zip(times, times[1:]))
    pre = [0] * len(specs)
    dec = [0] * len(specs)
    for _, st in fast:
        for r, i in enumerate(st.req_idx):
            if r < st.n_decode:
                dec[i] += 1
            else:
                pre[i] += st.q_len[r]
    assert pre == [s.prompt_len for s in specs]
    assert dec == [s.output_len - 1 for s in specs]
