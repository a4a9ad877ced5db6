"""Request metrics of the closed-loop replay (Section 4.4) and the
geometric-mean improvement I_m (Section 5.1), on hand-built runs."""
import math

import numpy as np
import pytest

from paper_2608_15171_gb300 import serving
from paper_2608_15171_gb300 import workloads as wl


def _run(specs, first, finish):
    r = serving.RunResult(steps=[], first_token_us=first, finish_us=finish, specs=specs)
    return serving.summarize(r)


def test_summary_of_a_hand_built_run():
    specs = [wl.RequestSpec(0, 100, 3), wl.RequestSpec(1_000_000, 100, 1), wl.RequestSpec(2_000_000, 50, 5)]
    # request 0: first token at 0.5 s, done at 1.5 s (2 more tokens: TPOT 0.5 s)
    # request 1: one output token, first = done at 1.25 s (TPOT 0)
    # request 2: first at 2.2 s, done at 3.0 s (4 more tokens: TPOT 0.2 s)
    s = _run(specs, [500_000, 1_250_000, 2_200_000], [1_500_000, 1_250_000, 3_000_000])
    assert s["avg_latency_s"] == pytest.approx((1.5 + 0.25 + 1.0) / 3)
    assert s["avg_ttft_s"] == pytest.approx((0.5 + 0.25 + 0.2) / 3)
    assert s["avg_tpot_s"] == pytest.approx((0.5 + 0.0 + 0.2) / 3)
    assert s["makespan_s"] == pytest.approx(3.0)
    # P95 of (1.5, 0.25, 1.0) by linear interpolation between order statistics
    assert s["p95_latency_s"] == pytest.approx(1.0 + 0.9 * 0.5)


def test_improvement_is_one_minus_geometric_mean_ratio():
    assert serving.improvement([1.0, 1.0], [2.0, 2.0]) == pytest.approx(50.0)
    assert serving.improvement([2.0], [1.0]) == pytest.approx(-100.0)
    # geometric, not arithmetic: ratios 0.5 and 2 cancel
    assert serving.improvement([1.0, 4.0], [2.0, 2.0]) == pytest.approx(0.0, abs=1e-12)
    r = (0.9 * 1.1 * 0.8) ** (1 / 3)
    assert serving.improvement([0.9, 1.1, 0.8], [1, 1, 1]) == pytest.approx((1 - r) * 100)


def test_policies_are_the_papers():
    assert serving.POLICIES["P-PAS"] == (2, 16384, 2048)
    # the strict threshold reading (more than two prefills) as an ablation
    assert serving.POLICIES["P-PAS N_th=3"] == (3, 16384, 2048)
    for name, (th, hi, lo) in serving.POLICIES.items():
        if not name.startswith("P-PAS"):
            assert hi == lo and th > 10**6


def test_roofline_by_regime_sums_and_fractions():
    """Two iterations under B_max and one under B_cap: per-regime sums of the
    measured times and of n_layers x max(FLOPs / peak, bytes / bandwidth)."""
    from types import SimpleNamespace
    geo = wl.QWEN25_3B
    shapes = [([16384], [16384]), ([8616], [25000]), ([1, 1, 512], [25000, 25001, 9000])]
    budgets = [16384, 16384, 2048]
    durations = [70000, 90000, 9000]
    steps = [serving.StepRecord(0, d, 0, 1, 0, b, int(b == 2048)) for d, b in zip(durations, budgets)]
    plans = [SimpleNamespace(q_len=np.array(q), ctx_len=np.array(c)) for q, c in shapes]
    res = serving.RunResult(steps, [], [], [], plans=plans)
    tf, bw = 1920.4, 6770.5
    out = serving.roofline_by_regime(res, geo, 36, tf, bw)

    def roof(q, c):
        sh = wl.StepShape(q, c)
        return 36 * max(wl.step_flops(sh, geo) / (tf * 1e12), wl.step_bytes(sh, geo) / (bw * 1e9)) * 1e6

    hi = out["B=16384"]
    assert hi["steps"] == 2 and hi["time_us"] == 160000
    assert hi["roofline_us"] == pytest.approx(roof(*shapes[0]) + roof(*shapes[1]))
    assert hi["frac"] == pytest.approx(hi["roofline_us"] / 160000)
    lo = out["B=2048"]
    assert lo["steps"] == 1 and lo["roofline_us"] == pytest.approx(roof(*shapes[2]))
    # the 16k chunk's roofline is the tensor term: 572.6 us per layer
    assert roof(*shapes[0]) / 36 == pytest.approx(572.6, abs=0.1)
    with pytest.raises(ValueError):
        serving.roofline_by_regime(serving.RunResult(steps, [], [], []), geo, 36, tf, bw)
