"""Request metrics of the closed-loop replay (Section 4.4) and the
geometric-mean improvement I_m (Section 5.1), on hand-built runs."""
import math

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
