"""Burst replay through the P-PAS planner on the GPU.

A Poisson burst of 16 requests (prompts ~U[20000, 30000], outputs
~U[16, 64]) is planned step by step by the C++ planner (threshold 2, MBT
16384 / 2048).  Every step's new keys/values are appended with the append
kernel and its mixed attention runs on one Qwen2.5-3B-geometry layer.  The
plan sequence is compared bit for bit with the oracle planner, the cache
after the replay with the oracle's appends, and sampled attention rows of
sampled steps with the float64 oracle.
"""
import numpy as np
import pytest
import torch

from _cases import assert_close
from oracle import attention as oa
from oracle import planner as op
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


@pytest.mark.parametrize("rate", [0.5, 1.0, 2.0, 4.0])
def test_burst_replay_plans_appends_and_attention(ppas, rate):
    geo = wl.QWEN25_3B
    hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
    specs = wl.poisson_burst(16, rate, seed=0)
    nb = 16 * 1879
    order = wl.page_permutation(nb, 0)
    width = 1900
    steps = ppas.replay([(s.arrival_us, s.prompt_len, s.output_len) for s in specs], nb, order,
                        cap_blocks_per_seq=width)
    oracle_steps = op.replay([op.Request(s.arrival_us, s.prompt_len, s.output_len) for s in specs], nb, order,
                             width=width)
    assert len(steps) == len(oracle_steps)
    for (t_c, sc), (t_o, so) in zip(steps, oracle_steps):
        assert t_c == t_o and sc.q_len.tolist() == so.q_len and sc.ctx_len.tolist() == so.ctx_len
        assert sc.slot_mapping.tolist() == so.slot_mapping and sc.b_prefill == so.b_prefill

    k_cache = torch.zeros((nb, hk, 16, D), dtype=torch.bfloat16, device="cuda")
    v_cache = torch.zeros_like(k_cache)
    k_host = np.zeros((nb, hk, 16, D), dtype=np.float32)
    v_host = np.zeros_like(k_host)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    check = set(range(0, len(steps), max(1, len(steps) // 8))) | {len(steps) - 1}
    check |= {i for i, (_, st) in enumerate(steps) if st.pressure and st.n_decode > 0 and i % 5 == 0}
    rng = np.random.default_rng(7)
    checked = 0
    for i, (_, st) in enumerate(steps):
        T = st.total_tokens
        kn = wl.bf16_normal((T, hk, D), 10_000 + 3 * i, "cuda")
        vn = wl.bf16_normal((T, hk, D), 10_001 + 3 * i, "cuda")
        q = wl.bf16_normal((T, hq, D), 10_002 + 3 * i, "cuda")
        slots = torch.from_numpy(st.slot_mapping).cuda()
        ppas.ppas_kv_append(kn, vn, slots, T, k_cache, v_cache, nb, hk, D, err)
        oa.kv_append(kn.float().cpu().numpy(), vn.float().cpu().numpy(), st.slot_mapping, k_host, v_host)
        tables = torch.from_numpy(np.ascontiguousarray(st.block_table)).cuda()
        out = torch.empty((T, hq, D), dtype=torch.bfloat16, device="cuda")
        wsb = ppas.ppas_attention_workspace_size(st.q_len, st.ctx_len, hq, hk)
        ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device="cuda")
        ppas.ppas_attention_step(q, k_cache, v_cache, nb, tables, st.block_table.shape[1], st.q_len, st.ctx_len,
                                 hq, hk, D, geo.scale, out, False, ws, wsb, err)
        if i in check:
            torch.cuda.synchronize()
            rows, start = [], 0
            for ql in st.q_len.tolist():
                if ql == 1:
                    rows += [(start, h) for h in range(hq)]
                else:
                    rows += [(start + int(t), int(h)) for t, h in
                             zip(list(rng.integers(0, ql, 24)) + [ql - 1], list(rng.integers(0, hq, 24)) + [hq - 1])]
                start += ql
            want = oa.sampled_rows(q.float().cpu().numpy(), k_host, v_host, st.block_table, st.q_len.tolist(),
                                   st.ctx_len.tolist(), geo.scale, rows)
            o = out.float().cpu().numpy()
            assert_close(o[[r for r, _ in rows], [h for _, h in rows]], want, f"step {i}")
            checked += 1
    torch.cuda.synchronize()
    assert err.item() == 0
    assert checked >= 8
    # the device cache equals the oracle's appends, bit for bit
    assert np.array_equal(k_cache.float().cpu().numpy(), k_host)
    assert np.array_equal(v_cache.float().cpu().numpy(), v_host)


def test_closed_loop_with_measured_clock(ppas):
    """The closed-loop replay executes every planned step on the GPU (2
    layers) and advances the clock by its measured time; the oracle planner
    driven by the logged durations reproduces every plan and start time, and
    the request metrics are consistent with the step log."""
    from paper_2608_15171_gb300 import serving
    geo = wl.QWEN25_3B
    specs = wl.poisson_burst(6, 40.0, seed=4, prompt=(3000, 9000), output=(2, 6))
    nb = serving.blocks_needed(specs)
    width = wl.blocks_for(max(s.prompt_len + s.output_len for s in specs))
    ex = serving.StepExecutor(geo, 2, nb, max_tokens=4096 + 8, max_rows=8, max_blocks_per_seq=width)
    order = wl.page_permutation(nb, 4)
    res = serving.closed_loop(specs, ex, order, 2, 4096, 1024, record_plans=True)
    durations = [s.duration_us for s in res.steps]
    assert all(d > 0 for d in durations)
    want = op.replay([op.Request(s.arrival_us, s.prompt_len, s.output_len) for s in specs], nb, order,
                     mbt_hi=4096, mbt_lo=1024, width=width, durations=durations)
    assert len(want) == len(res.plans)
    for rec, st, (t, so) in zip(res.steps, res.plans, want):
        assert rec.now_us == t
        assert st.q_len.tolist() == so.q_len and st.ctx_len.tolist() == so.ctx_len
        assert st.slot_mapping.tolist() == so.slot_mapping and st.b_prefill == so.b_prefill
    s = res.summary
    assert s["requests"] == len(specs) and s["steps"] == len(res.steps)
    for sp, f, e in zip(specs, res.first_token_us, res.finish_us):
        assert sp.arrival_us < f <= e
    end = res.steps[-1].now_us + res.steps[-1].duration_us
    assert max(res.finish_us) == end
    assert s["makespan_s"] == pytest.approx((end - min(sp.arrival_us for sp in specs)) / 1e6)
