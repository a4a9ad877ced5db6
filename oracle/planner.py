"""Pure-Python oracle of the P-PAS step planner.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

Passages followed
-----------------
* Algorithm 1 (Section 3): ``N_p`` = running + waiting prefills, ``N_d`` =
  running decodes; if ``N_p >= N_th`` and ``N_d > 0`` the aggregate prefill
  tokens of the iteration are limited to ``B_cap``, else to ``B_max``.  The
  decision is re-evaluated every iteration.
* Section 3: the global token budget (vLLM's MBT) stays unchanged; P-PAS only
  adds the prefill cap.  Evaluated configuration ``N_th = 2``,
  ``B_max = 16384``, ``B_cap = 2048`` (Sections 3 and 4.3).
* Section 2: continuous batching with chunked prefill; the MBT budget is
  shared by prefill and decode work of one iteration; long prompts are split
  into chunks across iterations.
* Section 7 (Sarathi-Serve, which vLLM's chunked prefill follows): ongoing
  decodes are scheduled first and the remaining budget is filled with
  prefill work.

Readings where the paper is silent (each also listed in the design notes):
* prefill chunks are taken first-come-first-served (arrival time, then
  request index) greedily until either budget is used up;
* only arrived requests count toward ``N_p`` / ``N_d``; a request whose last
  chunk runs this iteration still counts as a prefill this iteration;
* the final prefill chunk emits the first output token, so a request makes
  ``output_len - 1`` decode iterations; a decode row's context includes the
  token it processes;
* blocks: a FIFO free list seeded with a permutation of the pool; a request
  holds ``ceil(ctx / 16)`` blocks; blocks of requests that finished are
  returned to the tail of the free list at the start of the next plan call,
  in queue order and table order;
* the replay clock: ``15000 + 27 * prefill_tokens`` microseconds per
  iteration; when nothing is runnable the clock jumps to the next arrival.
"""
from __future__ import annotations

from collections import deque
from dataclasses import dataclass, field
from typing import List

PAGE_TOKENS = 16

PENDING, WAITING, RUNNING, FINISHED = 0, 1, 2, 3

# evaluated P-PAS configuration (Section 3, Section 4.3)
N_TH = 2
B_MAX = 16384
B_CAP = 2048

# replay clock (reading of the paper; 27 us/token ~ 668.6 ms / 25k tokens of
# whole-model prefill at MBT 16k in the prefill table of Section 6.1)
STEP_BASE_US = 15000
STEP_US_PER_PREFILL_TOKEN = 27


def prefill_budget(n_p: int, n_d: int, n_th: int, b_max: int, b_cap: int):
    """Algorithm 1: returns ``(B_prefill, pressure)``."""
    pressure = (n_p >= n_th) and (n_d > 0)
    return (b_cap if pressure else b_max), int(pressure)


@dataclass
class Request:
    arrival_us: int
    prompt_len: int
    output_len: int
    num_computed: int = 0
    num_generated: int = 0
    state: int = PENDING
    blocks: List[int] = field(default_factory=list)


@dataclass
class Step:
    n_decode: int
    n_prefill: int
    b_prefill: int
    pressure: int
    n_p: int
    n_d: int
    prefill_tokens: int
    total_tokens: int
    req_idx: List[int]
    q_len: List[int]
    ctx_len: List[int]
    block_table: List[List[int]]   # each row padded with -1 to ``width``
    slot_mapping: List[int]


class OutOfBlocks(RuntimeError):
    pass


def _ceil_div(a, b):
    return -(-a // b)


class Scheduler:
    """FIFO block pool plus the per-iteration P-PAS plan."""

    def __init__(self, num_blocks: int, free_order):
        free_order = [int(b) for b in free_order]
        if sorted(free_order) != list(range(num_blocks)):
            raise ValueError("free_order must be a permutation of range(num_blocks)")
        self.num_blocks = num_blocks
        self.free = deque(free_order)

    def plan_step(self, reqs: List[Request], now_us: int, threshold: int = N_TH,
                  mbt_hi: int = B_MAX, mbt_lo: int = B_CAP, width: int | None = None) -> Step:
        if threshold < 1 or mbt_lo < 1 or mbt_hi < mbt_lo:
            raise ValueError("need threshold >= 1 and 1 <= mbt_lo <= mbt_hi")
        order = sorted(range(len(reqs)), key=lambda i: (reqs[i].arrival_us, i))
        # a failed plan leaves the pool and every request as they were
        saved = (deque(self.free), [(r.state, list(r.blocks)) for r in reqs])
        try:
            return self._plan(reqs, order, now_us, threshold, mbt_hi, mbt_lo, width)
        except (OutOfBlocks, ValueError):
            self.free = saved[0]
            for r, (st, bl) in zip(reqs, saved[1]):
                r.state, r.blocks = st, bl
            raise

    def _plan(self, reqs, order, now_us, threshold, mbt_hi, mbt_lo, width):

        # blocks of requests finished in the previous iteration go back to the tail
        for i in order:
            r = reqs[i]
            if r.state == FINISHED and r.blocks:
                self.free.extend(r.blocks)
                r.blocks = []

        # admission
        for i in order:
            if reqs[i].state == PENDING and reqs[i].arrival_us <= now_us:
                reqs[i].state = WAITING

        live = [i for i in order if reqs[i].state in (WAITING, RUNNING)]
        prefills = [i for i in live if reqs[i].num_computed < reqs[i].prompt_len]
        decodes = [i for i in live if reqs[i].num_computed == reqs[i].prompt_len]
        n_p, n_d = len(prefills), len(decodes)
        b_prefill, pressure = prefill_budget(n_p, n_d, threshold, mbt_hi, mbt_lo)

        # decodes first (one token each) under the unchanged global budget,
        # then FCFS prefill chunks under both the prefill cap and what is left
        rows = []  # (req, q, ctx, is_prefill)
        used_total = 0
        for i in decodes:
            if used_total >= mbt_hi:
                break
            r = reqs[i]
            rows.append((i, 1, r.prompt_len + r.num_generated, False))
            used_total += 1
        n_decode = len(rows)
        used_prefill = 0
        for i in prefills:
            r = reqs[i]
            q = min(r.prompt_len - r.num_computed, b_prefill - used_prefill, mbt_hi - used_total)
            if q <= 0:
                break
            rows.append((i, q, r.num_computed + q, True))
            used_prefill += q
            used_total += q

        # block allocation: all-or-nothing
        need = sum(max(0, _ceil_div(ctx, PAGE_TOKENS) - len(reqs[i].blocks)) for i, _, ctx, _ in rows)
        if need > len(self.free):
            raise OutOfBlocks(f"need {need} blocks, {len(self.free)} free")
        for i, _, ctx, _ in rows:
            r = reqs[i]
            while len(r.blocks) < _ceil_div(ctx, PAGE_TOKENS):
                r.blocks.append(self.free.popleft())

        if width is None:
            width = max([len(reqs[i].blocks) for i, *_ in rows] + [0])
        tables, slots = [], []
        for i, q, ctx, _ in rows:
            blocks = reqs[i].blocks
            if len(blocks) > width:
                raise ValueError("block table width too small")
            tables.append(list(blocks) + [-1] * (width - len(blocks)))
            for pos in range(ctx - q, ctx):
                slots.append(blocks[pos // PAGE_TOKENS] * PAGE_TOKENS + pos % PAGE_TOKENS)

        # state update
        for i, q, ctx, is_prefill in rows:
            r = reqs[i]
            r.state = RUNNING
            if is_prefill:
                r.num_computed += q
                if r.num_computed == r.prompt_len:
                    r.num_generated = 1
            else:
                r.num_generated += 1
            if r.num_computed == r.prompt_len and r.num_generated >= r.output_len:
                r.state = FINISHED

        return Step(n_decode=n_decode, n_prefill=len(rows) - n_decode, b_prefill=b_prefill,
                    pressure=pressure, n_p=n_p, n_d=n_d, prefill_tokens=used_prefill,
                    total_tokens=used_total, req_idx=[r[0] for r in rows],
                    q_len=[r[1] for r in rows], ctx_len=[r[2] for r in rows],
                    block_table=tables, slot_mapping=slots)


def replay(reqs: List[Request], num_blocks: int, free_order, threshold=N_TH, mbt_hi=B_MAX,
           mbt_lo=B_CAP, width=None, max_steps=100000, durations=None):
    """Run the planner until every request finished; returns ``[(now_us, Step)]``.

    The clock is a deterministic integer: each iteration with work advances it
    by ``15000 + 27 * prefill_tokens`` us, or, when ``durations`` is given, by
    the next logged step duration (integer us, one per iteration with work, in
    order: a closed-loop run's measured step times); with nothing runnable it
    jumps to the next arrival.
    """
    sched = Scheduler(num_blocks, free_order)
    now = 0
    out = []
    for _ in range(max_steps):
        if all(r.state == FINISHED for r in reqs):
            # release the last finished requests' blocks like a next call would
            return out
        step = sched.plan_step(reqs, now, threshold, mbt_hi, mbt_lo, width)
        if not step.req_idx:
            pending = [r.arrival_us for r in reqs if r.state == PENDING]
            if not pending:
                raise RuntimeError("no runnable request and none pending")
            now = max(now, min(pending))
            continue
        out.append((now, step))
        if durations is None:
            now += STEP_BASE_US + STEP_US_PER_PREFILL_TOKEN * step.prefill_tokens
        else:
            now += int(durations[len(out) - 1])
    raise RuntimeError("replay did not finish")
