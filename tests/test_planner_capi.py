"""C++ planner behind the C ABI vs the Python oracle: bit-exact plans (CPU)."""
import os

import numpy as np
import pytest

from oracle import planner as op
from paper_2608_15171_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def ppas():
    if not os.path.exists(os.path.join(ROOT, "paper_2608_15171_gb300", "libppas.so")):
        from paper_2608_15171_gb300 import build
        build.build()
    from paper_2608_15171_gb300 import ppas as p
    return p


WIDTH = 2048


def _compare(oracle_steps, capi_steps):
    assert len(oracle_steps) == len(capi_steps)
    for (t_o, so), (t_c, sc) in zip(oracle_steps, capi_steps):
        assert t_o == t_c
        assert (so.b_prefill, so.pressure, so.n_p, so.n_d) == (sc.b_prefill, sc.pressure, sc.n_p, sc.n_d)
        assert (so.n_decode, so.n_prefill, so.prefill_tokens, so.total_tokens) == \
            (sc.n_decode, sc.n_prefill, sc.prefill_tokens, sc.total_tokens)
        assert so.req_idx == sc.req_idx.tolist()
        assert so.q_len == sc.q_len.tolist()
        assert so.ctx_len == sc.ctx_len.tolist()
        assert np.array_equal(np.array(so.block_table, dtype=np.int32).reshape(len(so.q_len), -1),
                              sc.block_table[:, :WIDTH])
        assert so.slot_mapping == sc.slot_mapping.tolist()


def _run_both(ppas, specs, nb, seed, **kw):
    order = wl.page_permutation(nb, seed)
    reqs = [op.Request(s.arrival_us, s.prompt_len, s.output_len) for s in specs]
    o = op.replay(reqs, nb, order, width=WIDTH, **kw)
    c = ppas.replay([(s.arrival_us, s.prompt_len, s.output_len) for s in specs], nb, order,
                    cap_blocks_per_seq=WIDTH, **kw)
    return o, c


@pytest.mark.parametrize("rate", [0.5, 1.0, 2.0, 4.0])
def test_burst_replay_bit_exact(ppas, rate):
    specs = wl.poisson_burst(16, rate, seed=0)
    o, c = _run_both(ppas, specs, 16 * 1879, 0)
    _compare(o, c)


@pytest.mark.parametrize("kw", [dict(threshold=3), dict(mbt_hi=2048, mbt_lo=2048),
                                dict(mbt_hi=8192, mbt_lo=1024), dict(threshold=1)])
def test_variants_bit_exact(ppas, kw):
    specs = wl.poisson_burst(12, 2.0, seed=5)
    o, c = _run_both(ppas, specs, 12 * 1900, 3, **kw)
    _compare(o, c)


@pytest.mark.parametrize("seed", range(6))
def test_random_small_traces_bit_exact(ppas, seed):
    rng = np.random.default_rng(100 + seed)
    n = int(rng.integers(1, 9))
    specs = [wl.RequestSpec(int(a), int(p), int(o)) for a, p, o in zip(
        np.sort(rng.integers(0, 200000, n)), rng.integers(1, 3000, n), rng.integers(1, 12, n))]
    hi = int(rng.choice([64, 512, 2048]))
    lo = int(rng.integers(1, hi + 1))
    o, c = _run_both(ppas, specs, n * 200 + 8, seed, threshold=int(rng.integers(1, 4)), mbt_hi=hi, mbt_lo=lo)
    _compare(o, c)


def test_bursty_trace_bit_exact(ppas):
    specs = wl.bursty_trace(seed=1, burst_rate=1.0)
    o, c = _run_both(ppas, specs, 12000, 2)
    _compare(o, c)


def test_planner_errors_leave_state_untouched(ppas):
    sch = ppas.Scheduler(3, [0, 1, 2], cap_blocks_per_seq=8)
    sch.add_requests([(0, 64, 3)])
    with pytest.raises(ppas.PpasError) as e:
        sch.plan(0)
    assert e.value.status == ppas.PPAS_ERR_OUT_OF_BLOCKS
    assert sch.free_blocks() == 3 and sch.reqs[0].state == ppas.PPAS_REQ_PENDING
    sch2 = ppas.Scheduler(64, None, cap_blocks_per_seq=2)
    sch2.add_requests([(0, 64, 3)])
    with pytest.raises(ppas.PpasError) as e:
        sch2.plan(0)
    assert e.value.status == ppas.PPAS_ERR_CAPACITY
    with pytest.raises(ppas.PpasError) as e:
        sch2.plan(0, threshold=0)
    assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    with pytest.raises(ppas.PpasError):
        ppas.ppas_sched_create(3, [0, 0, 1])
