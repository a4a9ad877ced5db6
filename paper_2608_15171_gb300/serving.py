"""Closed-loop replay of a request trace through the P-PAS planner, with the
clock driven by measured GPU step times (Sections 4.1, 4.4 and 5.1).

Every scheduler iteration planned by ``ppas_plan_step`` (Algorithm 1 and
the chunking of Section 3) is executed on the GPU: for each of the model's
layers, the step's new keys and values are appended to that layer's paged
cache and the mixed prefill + decode attention step runs over it.  The
iteration's measured duration (CUDA events around all of its device work,
plan upload included) advances the clock, and requests that arrived in the
meantime join the next plan.  This is attention only: no projections, MLP,
norms or sampling run, so absolute latencies are far below a full model's;
the activations are synthetic (seeded normal values).

Request metrics follow Section 4.4: end-to-end latency from arrival to the
last output token, time to first token (the first token comes out of the
iteration that computes the prompt's last chunk), time per output token
over the remaining tokens, and the makespan from the first arrival to the
last completion.  ``improvement`` is the geometric-mean comparison of
Section 5.1 (I_m = (1 - R_m) x 100 %).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Sequence

import numpy as np

from . import ppas
from . import workloads as wl


@dataclass
class StepRecord:
    now_us: int          # clock at the start of the iteration
    duration_us: int     # measured device time of the iteration
    n_decode: int
    n_prefill: int
    prefill_tokens: int
    b_prefill: int
    pressure: int


@dataclass
class RunResult:
    steps: List[StepRecord]
    first_token_us: List[int]
    finish_us: List[int]
    specs: List[wl.RequestSpec]
    summary: Dict[str, float] = field(default_factory=dict)
    plans: List[ppas.StepPlan] = field(default_factory=list)  # with record_plans


class StepExecutor:
    """Device state of a closed-loop run: per-layer paged K/V caches, one
    pool of synthetic activations, plan buffers and the workspace."""

    def __init__(self, geo: wl.Geometry, n_layers: int, num_blocks: int, max_tokens: int, max_rows: int,
                 max_blocks_per_seq: int, device="cuda", seed: int = 0):
        import torch
        self.torch = torch
        self.geo, self.n_layers, self.num_blocks = geo, n_layers, num_blocks
        hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
        self.k_cache = [torch.zeros((num_blocks, hk, 16, D), dtype=torch.bfloat16, device=device)
                        for _ in range(n_layers)]
        self.v_cache = [torch.zeros((num_blocks, hk, 16, D), dtype=torch.bfloat16, device=device)
                        for _ in range(n_layers)]
        self.q = wl.bf16_normal((max_tokens, hq, D), seed * 10 + 1, device)
        self.k_new = wl.bf16_normal((max_tokens, hk, D), seed * 10 + 2, device)
        self.v_new = wl.bf16_normal((max_tokens, hk, D), seed * 10 + 3, device)
        self.out = torch.empty((max_tokens, hq, D), dtype=torch.bfloat16, device=device)
        self.tables = torch.empty((max_rows, max_blocks_per_seq), dtype=torch.int32, device=device)
        self.slots = torch.empty((max_tokens,), dtype=torch.int32, device=device)
        self.tables_pin = torch.empty((max_rows, max_blocks_per_seq), dtype=torch.int32).pin_memory()
        self.slots_pin = torch.empty((max_tokens,), dtype=torch.int32).pin_memory()
        self.err = torch.zeros(1, dtype=torch.int32, device=device)
        self.ws = torch.empty(256, dtype=torch.uint8, device=device)
        self.stream = torch.cuda.current_stream()
        self.max_tokens, self.max_rows = max_tokens, max_rows

    def run(self, st: ppas.StepPlan) -> int:
        """Execute one planned iteration over all layers; returns its device
        time in integer microseconds."""
        torch, geo = self.torch, self.geo
        hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
        n, rows = st.total_tokens, st.n_rows
        if n > self.max_tokens or rows > self.max_rows:
            raise ValueError("step larger than the executor's buffers")
        width = st.block_table.shape[1]
        ws_bytes = ppas.ppas_attention_workspace_size(st.q_len, st.ctx_len, hq, hk)
        if ws_bytes > self.ws.numel():
            self.ws = torch.empty(ws_bytes, dtype=torch.uint8, device=self.ws.device)
        self.tables_pin[:rows, :width].copy_(torch.from_numpy(st.block_table))
        self.slots_pin[:n].copy_(torch.from_numpy(st.slot_mapping))
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(self.stream)
        tables = self.tables[:rows, :width]
        tables.copy_(self.tables_pin[:rows, :width], non_blocking=True)
        self.slots[:n].copy_(self.slots_pin[:n], non_blocking=True)
        for layer in range(self.n_layers):
            ppas.ppas_kv_append(self.k_new[:n], self.v_new[:n], self.slots, n, self.k_cache[layer],
                                self.v_cache[layer], self.num_blocks, hk, D, self.err, self.stream)
            ppas.ppas_attention_step(self.q[:n], self.k_cache[layer], self.v_cache[layer], self.num_blocks, tables,
                                     width, st.q_len, st.ctx_len, hq, hk, D, geo.scale, self.out[:n], False,
                                     self.ws, ws_bytes, self.err, self.stream)
        e1.record(self.stream)
        e1.synchronize()
        return max(1, int(round(e0.elapsed_time(e1) * 1000.0)))

    def check(self) -> None:
        if int(self.err.item()) != 0:
            raise RuntimeError(f"device error flag {int(self.err.item())}")


def blocks_needed(specs: Sequence[wl.RequestSpec]) -> int:
    """A pool that never runs out: every request's full context, plus slack."""
    return sum(wl.blocks_for(s.prompt_len + s.output_len) for s in specs) + 16


def closed_loop(specs: Sequence[wl.RequestSpec], executor: StepExecutor, free_order, threshold: int = 2,
                mbt_hi: int = 16384, mbt_lo: int = 2048, max_steps: int = 1000000,
                record_plans: bool = False) -> RunResult:
    """Plan and execute every iteration until all requests finished.  With
    ``threshold`` larger than any request count (or mbt_hi == mbt_lo) the
    budget is static: the fixed-MBT baselines."""
    specs = list(specs)
    sch = ppas.Scheduler(executor.num_blocks, free_order, cap_rows=executor.max_rows,
                         cap_blocks_per_seq=executor.tables.shape[1], cap_tokens=executor.max_tokens)
    sch.add_requests([(s.arrival_us, s.prompt_len, s.output_len) for s in specs])
    now = 0
    steps: List[StepRecord] = []
    plans: List[ppas.StepPlan] = []
    first = [-1] * len(specs)
    finish = [-1] * len(specs)
    generated = [0] * len(specs)
    try:
        for _ in range(max_steps):
            if all(sch.reqs[i].state == ppas.PPAS_REQ_FINISHED for i in range(sch.n_reqs)):
                break
            st = sch.plan(now, threshold, mbt_hi, mbt_lo)
            if st.n_rows == 0:
                pending = [sch.reqs[i].arrival_us for i in range(sch.n_reqs)
                           if sch.reqs[i].state == ppas.PPAS_REQ_PENDING]
                if not pending:
                    raise RuntimeError("no runnable request and none pending")
                now = max(now, min(pending))
                continue
            dt = executor.run(st)
            end = now + dt
            for r in range(st.n_rows):
                i = int(st.req_idx[r])
                if r < st.n_decode:            # one output token
                    generated[i] += 1
                elif int(st.ctx_len[r]) == specs[i].prompt_len:  # prompt done: first token
                    generated[i] += 1
                    first[i] = end
                if generated[i] == specs[i].output_len and finish[i] < 0:
                    finish[i] = end
            steps.append(StepRecord(now, dt, st.n_decode, st.n_prefill, st.prefill_tokens, st.b_prefill,
                                    st.pressure))
            if record_plans:
                plans.append(st)
            now = end
        else:
            raise RuntimeError("closed loop did not finish")
    finally:
        sch.close()
    executor.check()
    res = RunResult(steps, first, finish, specs, plans=plans)
    res.summary = summarize(res)
    return res


def summarize(res: RunResult) -> Dict[str, float]:
    """Section 4.4 metrics of one run (seconds)."""
    arr = np.array([s.arrival_us for s in res.specs], dtype=np.float64)
    first = np.array(res.first_token_us, dtype=np.float64)
    fin = np.array(res.finish_us, dtype=np.float64)
    outs = np.array([s.output_len for s in res.specs], dtype=np.float64)
    e2e = (fin - arr) / 1e6
    ttft = (first - arr) / 1e6
    tpot = np.where(outs > 1, (fin - first) / np.maximum(outs - 1, 1), 0.0) / 1e6
    return {"avg_latency_s": float(e2e.mean()), "p95_latency_s": float(np.percentile(e2e, 95)),
            "avg_ttft_s": float(ttft.mean()), "avg_tpot_s": float(tpot.mean()),
            "makespan_s": float((fin.max() - arr.min()) / 1e6), "steps": len(res.steps),
            "requests": len(res.specs)}


def roofline_by_regime(res: RunResult, geo: wl.Geometry, n_layers: int, tflops: float,
                       gbs: float) -> Dict[str, Dict[str, float]]:
    """Time-weighted step-roofline fraction of a run recorded with its plans,
    split by the prefill budget each iteration ran under (B_max or B_cap):
    sum over its iterations of n_layers * max(FLOPs / tflops, bytes / gbs)
    over the sum of their measured times (which also hold the appends and the
    plan upload)."""
    if len(res.plans) != len(res.steps):
        raise ValueError("run was not recorded with its plans")
    out: Dict[str, Dict[str, float]] = {}
    for rec, st in zip(res.steps, res.plans):
        shape = wl.StepShape([int(x) for x in st.q_len], [int(x) for x in st.ctx_len])
        roof_us = n_layers * max(wl.step_flops(shape, geo) / (tflops * 1e12),
                                 wl.step_bytes(shape, geo) / (gbs * 1e9)) * 1e6
        d = out.setdefault(f"B={rec.b_prefill}", {"steps": 0, "time_us": 0.0, "roofline_us": 0.0})
        d["steps"] += 1
        d["time_us"] += rec.duration_us
        d["roofline_us"] += roof_us
    for d in out.values():
        d["frac"] = d["roofline_us"] / d["time_us"]
    return out


def improvement(ppas_values: Sequence[float], baseline_values: Sequence[float]) -> float:
    """I_m of Section 5.1: (1 - R_m) x 100 %, R_m the geometric mean over the
    burst rates of P-PAS's value over the baseline's."""
    r = [a / b for a, b in zip(ppas_values, baseline_values)]
    rm = math.exp(sum(math.log(x) for x in r) / len(r))
    return (1.0 - rm) * 100.0


# the policies of Sections 4.3 and 5.1: P-PAS and the static budgets, plus
# P-PAS with the strict reading of its threshold (more than two concurrent
# prefills, N_p >= 3) as an ablation
POLICIES = {"P-PAS": (2, 16384, 2048), "MBT 1k": (1 << 30, 1024, 1024), "MBT 2k": (1 << 30, 2048, 2048),
            "MBT 4k": (1 << 30, 4096, 4096), "MBT 8k": (1 << 30, 8192, 8192), "MBT 16k": (1 << 30, 16384, 16384),
            "P-PAS N_th=3": (3, 16384, 2048)}


def sweep(burst_rates, seeds, time_scale: float, policies=tuple(POLICIES), geo=wl.QWEN25_3B,
          n_layers=None, device="cuda", log=print):
    """The 50 s alternating trace of Section 4.1 at each burst rate, with
    every time compressed by ``time_scale`` (phases 10 s / time_scale,
    rates x time_scale: the same requests in the same order), replayed
    under each policy.  Returns {policy: {rate: mean summary over seeds}}."""
    n_layers = geo.n_layers if n_layers is None else n_layers
    out = {p: {} for p in policies}
    for rate in burst_rates:
        for seed in seeds:
            specs = wl.bursty_trace(seed, rate * time_scale, steady_rate=0.2 * time_scale,
                                    phase_s=10.0 / time_scale, duration_s=50.0 / time_scale)
            nb = blocks_needed(specs)
            ex = StepExecutor(geo, n_layers, nb, max_tokens=16384 + len(specs), max_rows=len(specs) + 1,
                              max_blocks_per_seq=wl.blocks_for(max(s.prompt_len + s.output_len for s in specs)),
                              device=device, seed=seed)
            for pol in policies:
                th, hi, lo = POLICIES[pol]
                r = closed_loop(specs, ex, wl.page_permutation(nb, seed), th, hi, lo)
                acc = out[pol].setdefault(rate, [])
                acc.append(r.summary)
                log(f"rate {rate} seed {seed} {pol}: " + ", ".join(f"{k} {v:.4g}" for k, v in r.summary.items()))
            del ex
    return {p: {rate: {k: float(np.mean([s[k] for s in v])) for k in v[0]} for rate, v in d.items()}
            for p, d in out.items()}


def main(argv=None):
    import argparse
    import json
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--rates", type=float, nargs="+", default=[0.4, 0.6, 0.8, 1.0, 1.2, 1.4])
    ap.add_argument("--seeds", type=int, nargs="+", default=[0])
    ap.add_argument("--time-scale", type=float, default=40.0)
    ap.add_argument("--layers", type=int, default=None)
    ap.add_argument("--policies", nargs="+", default=list(POLICIES))
    a = ap.parse_args(argv)
    res = sweep(a.rates, a.seeds, a.time_scale, a.policies, n_layers=a.layers)
    imp = {}
    if "P-PAS" in res:
        for base in (p for p in res if p != "P-PAS"):
            imp[base] = {m: improvement([res["P-PAS"][r][m] for r in a.rates], [res[base][r][m] for r in a.rates])
                         for m in ("avg_latency_s", "p95_latency_s", "avg_ttft_s", "avg_tpot_s", "makespan_s")}
    print(json.dumps({"time_scale": a.time_scale, "results": res, "improvement_pct": imp}))


if __name__ == "__main__":
    main()
