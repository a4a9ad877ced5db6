"""GPU parity: the CUDA path through the C ABI against the float64 oracle.

Small cases compare every output element; the full-size workloads compare
sampled rows that the oracle computes exactly, in the launch configuration
the benchmark uses.
"""
import numpy as np
import pytest
import torch

from _cases import (MAX_ABS, assert_close, device_case, host32, host64, oracle_full, oracle_rows, run_step,
                    sample_rows)
from oracle import attention as oa
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

QWEN = wl.QWEN25_3B
LLAMA = wl.LLAMA31_8B
G1 = wl.Geometry("mha-4", 4, 4, 128, 1)
G2 = wl.Geometry("gqa-2", 8, 4, 128, 1)


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


SMALL_SHAPES = [
    wl.StepShape([130], [130]),                                   # prefix 0, ragged q tile
    wl.StepShape([1, 1, 1], [1, 17, 300]),                        # decodes only, tiny contexts
    wl.StepShape([1, 37, 1, 300], [40, 37, 129, 1000]),           # mixed, unaligned prefixes
    wl.StepShape([2, 257, 129], [2, 700, 129 + 384]),             # several q tiles, prefix % 128 != 0
    wl.StepShape([1] * 5 + [64], [4000, 3999, 2050, 16, 1, 5000]),  # decodes with splits
    wl.StepShape([1, 200], [5000, 6000]),                        # chunk tiles split over their KV range
]


@pytest.mark.parametrize("geo", [QWEN, LLAMA, G1, G2], ids=lambda g: g.name)
@pytest.mark.parametrize("si", range(len(SMALL_SHAPES)))
@pytest.mark.parametrize("out_fp32", [True, False])
def test_small_steps_full_parity(ppas, geo, si, out_fp32):
    c = device_case(geo, SMALL_SHAPES[si], seed=si + 10 * geo.n_q_heads)
    out = run_step(ppas, c, out_fp32)
    torch.cuda.synchronize()
    assert_close(host64(out), oracle_full(c), f"{geo.name} shape {si}")


def test_tiny_workload_four_chunks_with_decodes(ppas):
    """2048-token prompt as 4 chunks of 512 at MBT 512 (keys/values written by
    the append kernel), the last chunk batched with 2 decode rows of context
    2048; fp32 output; every element against the oracle, and the chunked
    result against one unchunked causal pass."""
    geo = QWEN
    L, hq, hk, D = 2048, geo.n_q_heads, geo.n_kv_heads, geo.head_dim
    nb = 3 * (L // 16) + 4
    perm = wl.page_permutation(nb, 1)
    tables_np = np.stack([perm[i * 128:(i + 1) * 128] for i in range(3)]).astype(np.int32)
    tables = torch.from_numpy(tables_np).cuda()
    k_cache = torch.zeros((nb, hk, 16, D), dtype=torch.bfloat16, device="cuda")
    v_cache = torch.zeros_like(k_cache)
    # decode rows 1, 2: contexts of 2048 already cached except their last token
    k_all = wl.bf16_normal((3, L, hk, D), 21, "cuda")
    v_all = wl.bf16_normal((3, L, hk, D), 22, "cuda")
    q_prompt = wl.bf16_normal((L, hq, D), 23, "cuda")
    q_dec = wl.bf16_normal((2, hq, D), 24, "cuda")

    def slots(row, lo, hi):
        pos = np.arange(lo, hi)
        return torch.from_numpy(tables_np[row][pos // 16] * 16 + pos % 16).int().cuda()

    for r in (1, 2):
        ppas.ppas_kv_append(k_all[r, :L - 1], v_all[r, :L - 1], slots(r, 0, L - 1), L - 1, k_cache, v_cache, nb,
                            hk, D)
    outs = []
    for i in range(4):
        lo, hi = 512 * i, 512 * (i + 1)
        if i < 3:
            rows, ql, cl = [0], [512], [hi]
            q = q_prompt[lo:hi]
            new_slots = slots(0, lo, hi)
            kn, vn = k_all[0, lo:hi], v_all[0, lo:hi]
        else:
            rows, ql, cl = [1, 2, 0], [1, 1, 512], [L, L, L]
            q = torch.cat([q_dec, q_prompt[lo:hi]])
            new_slots = torch.cat([slots(1, L - 1, L), slots(2, L - 1, L), slots(0, lo, hi)])
            kn = torch.cat([k_all[1, L - 1:], k_all[2, L - 1:], k_all[0, lo:hi]])
            vn = torch.cat([v_all[1, L - 1:], v_all[2, L - 1:], v_all[0, lo:hi]])
        ppas.ppas_kv_append(kn.contiguous(), vn.contiguous(), new_slots, new_slots.numel(), k_cache, v_cache, nb,
                            hk, D)
        t = tables[rows].contiguous()
        out = torch.empty((q.shape[0], hq, D), dtype=torch.float32, device="cuda")
        ws_b = ppas.ppas_attention_workspace_size(ql, cl, hq, hk)
        ws = torch.empty(max(ws_b, 1), dtype=torch.uint8, device="cuda")
        ppas.ppas_attention_step(q.contiguous(), k_cache, v_cache, nb, t, 128, ql, cl, hq, hk, D, geo.scale, out,
                                 True, ws, ws_b)
        torch.cuda.synchronize()
        want = oa.paged_attention(host64(q), host64(k_cache), host64(v_cache), tables_np[rows], ql, cl, geo.scale)
        assert_close(host64(out), want, f"chunk {i}")
        outs.append(out[-512:])
    # chunk invariance: the four chunk outputs equal one unchunked causal pass
    whole = torch.empty((L, hq, D), dtype=torch.float32, device="cuda")
    ppas.ppas_attention_step(q_prompt, k_cache, v_cache, nb, tables[:1].contiguous(), 128, [L], [L], hq, hk, D,
                             geo.scale, whole, True)
    torch.cuda.synchronize()
    diff = (torch.cat(outs) - whole).abs()
    assert diff.max().item() <= MAX_ABS and diff.mean().item() <= 2e-3


def test_kv_append_bit_exact_and_bad_slots(ppas):
    hk, D, nb, T = 8, 128, 40, 300
    k_cache = torch.zeros((nb, hk, 16, D), dtype=torch.bfloat16, device="cuda")
    v_cache = torch.zeros_like(k_cache)
    kn = wl.bf16_normal((T, hk, D), 5, "cuda")
    vn = wl.bf16_normal((T, hk, D), 6, "cuda")
    rng = np.random.default_rng(0)
    slots = rng.permutation(nb * 16)[:T].astype(np.int32)
    slots[[3, 77]] = -1                        # skipped tokens
    ppas.ppas_kv_append(kn, vn, torch.from_numpy(slots).cuda(), T, k_cache, v_cache, nb, hk, D)
    torch.cuda.synchronize()
    kc = np.zeros((nb, hk, 16, D))
    vc = np.zeros((nb, hk, 16, D))
    keep = slots >= 0
    oa.kv_append(host64(kn)[keep], host64(vn)[keep], slots[keep], kc, vc)
    assert np.array_equal(host64(k_cache), kc) and np.array_equal(host64(v_cache), vc)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    bad = torch.tensor([nb * 16 + 5], dtype=torch.int32, device="cuda")
    ppas.ppas_kv_append(kn[:1], vn[:1], bad, 1, k_cache, v_cache, nb, hk, D, err)
    torch.cuda.synchronize()
    assert err.item() == ppas.PPAS_DEVERR_BAD_INDEX
    assert np.array_equal(host64(k_cache), kc)


def test_garbage_outside_contexts_is_never_read(ppas):
    """NaN in every cache slot outside the contexts (partial last pages,
    unused blocks) must not reach the output."""
    for geo in (QWEN, LLAMA):
        shape = wl.StepShape([1, 1, 45, 200], [33, 1, 61, 777])
        c = device_case(geo, shape, seed=4, nan_fill=True)
        out = run_step(ppas, c, True)
        torch.cuda.synchronize()
        assert_close(host64(out), oracle_full(c), geo.name)


def test_single_key_uniform_keys_constant_values(ppas):
    geo = QWEN
    shape = wl.StepShape([1, 150], [1, 300])
    c = device_case(geo, shape, seed=8)
    out = run_step(ppas, c, True)
    torch.cuda.synchronize()
    # single key: the decode row with context 1 returns V[0] of its kv-head
    blk = int(c.tables_np[0, 0])
    for h in range(geo.n_q_heads):
        v0 = c.v_cache[blk, h // 8, 0].float()
        assert torch.equal(out[0, h], v0)
    # identical keys: every row is the mean of its visible values
    c.k_cache[:] = c.k_cache[0, 0, 0]
    out = run_step(ppas, c, True)
    torch.cuda.synchronize()
    assert_close(host64(out), oracle_full(c), "uniform keys")
    # constant values: output equals the constant whatever the weights (up
    # to the bf16 rounding of the weights that multiply V)
    c2 = device_case(geo, shape, seed=9)
    c2.v_cache.fill_(0.75)
    out = run_step(ppas, c2, True)
    torch.cuda.synchronize()
    assert (out - 0.75).abs().max().item() <= 0.75 * 2.0 ** -8


@pytest.mark.parametrize("growth", [0.2, 3.0])
def test_scores_growing_along_the_context(ppas, growth):
    """Keys of KV tile j (128 keys) scaled by 1 + growth * j, so every row's
    scores grow along its context.  growth 0.2: the row maximum grows by less
    than the kernel's 2^8 rescale threshold per tile, so a stale maximum stays
    in use and later exponentials exceed 1; growth 3: it grows by far more on
    almost every tile, so the maximum is raised and O rescaled in TMEM again
    and again.  Every element against the oracle."""
    geo = QWEN
    shape = wl.StepShape([1, 130, 1], [1500, 1700, 3000])
    c = device_case(geo, shape, seed=31 + int(growth * 10))
    for s_, ctx in enumerate(shape.ctx_lens):
        for b in range(wl.blocks_for(ctx)):
            c.k_cache[int(c.tables_np[s_, b])] *= 1.0 + growth * (b // 8)
    out = run_step(ppas, c, True)
    torch.cuda.synchronize()
    assert torch.isfinite(out).all()
    assert_close(host64(out), oracle_full(c), f"growth {growth}")


def test_chunk_over_a_long_prefix(ppas):
    """130 new tokens (two query tiles, the second ragged) over a 524,288-token
    prefix: every (query tile, head slot) unit is cut into stream-K pieces on
    many CTAs and merged; every element against the oracle."""
    geo = QWEN
    shape = wl.StepShape([130], [130 + (1 << 19)])
    c = device_case(geo, shape, seed=45, extra_blocks=3)
    n_kernels = ppas.ppas_attention_kernel_count(shape.q_lens, shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads,
                                                 ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens,
                                                                                    geo.n_q_heads,
                                                                                    geo.n_kv_heads))
    assert n_kernels == 2  # the prefill launch and its merge
    out = run_step(ppas, c, True)
    torch.cuda.synchronize()
    want = oa.paged_attention(host64(c.q), host32(c.k_cache), host32(c.v_cache), c.tables_np, shape.q_lens,
                              shape.ctx_lens, c.scale, workers=oa.default_workers())
    assert_close(host64(out), want, "chunk over a 512k prefix")


def test_dirty_and_reused_workspace(ppas):
    """The workspace is the caller's uninitialised memory: filled with random
    bytes, then reused by two more steps (the split units' partials, the
    decode partials and tickets of the step before left in it), the step
    gives the oracle's result, bit for bit the same every time."""
    geo = QWEN
    hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
    shape = wl.StepShape([1, 256, 130], [20000, 40000, 9000])
    c = device_case(geo, shape, seed=61)
    ws_bytes = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, hq, hk)
    # the chunks' units are cut: more workspace than the decode row's partials
    assert ws_bytes > ppas.ppas_attention_workspace_size([1], [20000], hq, hk)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(5)
    ws = torch.randint(0, 256, (ws_bytes,), dtype=torch.uint8, device="cuda", generator=gen)
    outs = []
    for _ in range(3):
        out = torch.empty((shape.total_q, hq, D), dtype=torch.float32, device="cuda")
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        ppas.ppas_attention_step(c.q, c.k_cache, c.v_cache, c.num_blocks, c.tables, c.width, shape.q_lens,
                                 shape.ctx_lens, hq, hk, D, c.scale, out, True, ws, ws_bytes, err)
        torch.cuda.synchronize()
        assert err.item() == 0
        outs.append(out)
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])
    assert_close(host64(outs[0]), oracle_full(c), "dirty and reused workspace")


def test_chunk_at_the_longest_prefill_context(ppas):
    """A 130-token chunk whose context ends at the longest the boundary
    accepts for prefill rows (65535 KV tiles of 128 keys: the items' 16-bit
    tile indices), with constant values: the output is that constant
    whatever the weights (up to their bf16 rounding)."""
    geo = QWEN
    hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
    ctx = 65535 * 128
    shape = wl.StepShape([130], [ctx])
    nb = wl.blocks_for(ctx)
    k_cache = torch.empty((nb, hk, 16, D), dtype=torch.bfloat16, device="cuda")
    step = 1 << 17
    for b0 in range(0, nb, step):
        k_cache[b0:b0 + step] = wl.bf16_normal((min(step, nb - b0), hk, 16, D), 700 + b0 // step, "cuda")
    v_cache = torch.full((nb, hk, 16, D), -1.25, dtype=torch.bfloat16, device="cuda")
    tables = torch.from_numpy(wl.page_permutation(nb, 47).reshape(1, nb)).cuda()
    q = wl.bf16_normal((130, hq, D), 48, "cuda")
    out = torch.empty((130, hq, D), dtype=torch.float32, device="cuda")
    ws_bytes = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, hq, hk)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ppas.ppas_attention_step(q, k_cache, v_cache, nb, tables, nb, shape.q_lens, shape.ctx_lens, hq, hk, D,
                             geo.scale, out, True, ws, ws_bytes, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert (out + 1.25).abs().max().item() <= 1.25 * 2.0 ** -8


def test_long_decode_rows(ppas):
    """Decode rows far longer than the workloads': 2,097,157 tokens (129
    splits of 1024 pages, merged in several rounds) against the oracle for
    every head, and the longest row the boundary accepts, 2^25 tokens (2048
    splits), with constant values, whose output is that constant whatever
    the weights (up to the bf16 rounding of the weights)."""
    geo = QWEN
    hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
    shape = wl.StepShape([1], [(1 << 21) + 5])
    c = device_case(geo, shape, seed=41, extra_blocks=3)
    out = run_step(ppas, c, True)
    torch.cuda.synchronize()
    rows = [(0, h) for h in range(hq)]
    assert_close(host64(out)[0], oracle_rows(c, rows), "2M-token decode row")
    del c, out
    torch.cuda.empty_cache()

    ctx = 1 << 25
    nb = wl.blocks_for(ctx)
    k_cache = torch.empty((nb, hk, 16, D), dtype=torch.bfloat16, device="cuda")
    step = 1 << 17
    for b0 in range(0, nb, step):  # N(0,1) keys, drawn in slices to bound the float32 scratch
        k_cache[b0:b0 + step] = wl.bf16_normal((min(step, nb - b0), hk, 16, D), 900 + b0 // step, "cuda")
    v_cache = torch.full((nb, hk, 16, D), 0.75, dtype=torch.bfloat16, device="cuda")
    tables = torch.from_numpy(wl.page_permutation(nb, 43).reshape(1, nb)).cuda()
    q = wl.bf16_normal((1, hq, D), 44, "cuda")
    out = torch.empty((1, hq, D), dtype=torch.float32, device="cuda")
    ws_bytes = ppas.ppas_attention_workspace_size([1], [ctx], hq, hk)
    ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ppas.ppas_attention_step(q, k_cache, v_cache, nb, tables, nb, [1], [ctx], hq, hk, D, geo.scale, out, True,
                             ws, ws_bytes, err)
    torch.cuda.synchronize()
    assert err.item() == 0
    assert (out - 0.75).abs().max().item() <= 0.75 * 2.0 ** -8


def test_page_permutation_invariance_bitwise(ppas):
    geo = LLAMA
    shape = wl.StepShape([1, 1, 300], [2000, 77, 900])
    c = device_case(geo, shape, seed=12)
    a = run_step(ppas, c, False)
    relabel = torch.from_numpy(np.random.default_rng(3).permutation(c.num_blocks)).cuda()
    k2 = torch.empty_like(c.k_cache)
    v2 = torch.empty_like(c.v_cache)
    k2[relabel] = c.k_cache
    v2[relabel] = c.v_cache
    c.k_cache, c.v_cache = k2, v2
    t = torch.from_numpy(c.tables_np).long().cuda()
    c.tables = torch.where(t >= 0, relabel[t.clamp(min=0)], t).int().contiguous()
    b = run_step(ppas, c, False)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


def test_bad_block_id_sets_error_flag(ppas):
    geo = QWEN
    c = device_case(geo, wl.StepShape([1, 40], [100, 40]), seed=2)
    c.tables[0, 2] = c.num_blocks + 100
    c.tables[1, 0] = -7
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    run_step(ppas, c, True, err=err)
    torch.cuda.synchronize()
    assert err.item() == ppas.PPAS_DEVERR_BAD_INDEX


def test_repeated_calls_reuse_workspace(ppas):
    """The split-K counters in the workspace are ready for the next call."""
    geo = QWEN
    c = device_case(geo, wl.StepShape([1] * 8, [25000 + i for i in range(8)]), seed=3)
    a = run_step(ppas, c, True)
    for _ in range(3):
        b = run_step(ppas, c, True)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    rows = sample_rows(c.shape, geo.n_q_heads, 0, 0)
    assert_close(host64(a)[[r for r, _ in rows], [h for _, h in rows]], oracle_rows(c, rows), "decodes 25k")


# ---------------------------------------------------------------- full sizes
FULL = [
    ("low-pressure s1 (16384, p=0)", QWEN, lambda: wl.low_pressure_steps()[0]),
    ("low-pressure s2 (8616, p=16384)", QWEN, lambda: wl.low_pressure_steps()[1]),
    ("high-pressure 4x512 + 8 decodes", QWEN, lambda: wl.high_pressure_step(0)),
    ("llama 16384 + 4 decodes", LLAMA, lambda: wl.llama_hi_step(0)),
    ("llama 3 chunks + 16 decodes", LLAMA, lambda: wl.llama_lo_step(0)),
    # the decode rows of the Llama MBT 2k step alone (1.97 GB of K/V)
    ("llama_decodes_only_16x30k", LLAMA,
     lambda: wl.StepShape(wl.llama_lo_step(0).q_lens[:16], wl.llama_lo_step(0).ctx_lens[:16])),
]


@pytest.mark.parametrize("name,geo,mk", FULL, ids=[f[0] for f in FULL])
def test_full_size_sampled_rows(ppas, name, geo, mk):
    shape = mk()
    c = device_case(geo, shape, seed=0, extra_blocks=64)
    out = run_step(ppas, c, False)
    torch.cuda.synchronize()
    o = out.float().cpu().numpy()
    assert np.all(np.isfinite(o))
    rows = sample_rows(shape, geo.n_q_heads, 96, seed=1)
    got = o[[r for r, _ in rows], [h for _, h in rows]]
    assert_close(got, oracle_rows(c, rows), name)


@pytest.mark.parametrize("name,geo,mk", FULL, ids=[f[0] for f in FULL])
def test_full_layer_every_element(ppas, name, geo, mk):
    """One whole layer of every full-size workload, in the launch
    configuration the benchmark times (whole units or stream-K pieces with
    their merge; a mixed step's decode rows in the same launch as its
    prefill tiles): every output element against the float64 oracle."""
    shape = mk()
    c = device_case(geo, shape, seed=2, extra_blocks=64)
    out = run_step(ppas, c, False)
    torch.cuda.synchronize()
    want = oa.paged_attention(host64(c.q), host32(c.k_cache), host32(c.v_cache), c.tables_np, shape.q_lens,
                              shape.ctx_lens, c.scale, workers=oa.default_workers())
    assert_close(host64(out), want, name)


def test_split_kv_and_unsplit_fallback_agree(ppas):
    """A chunk over a long prefix runs split over its KV range (partials merged
    by the merge kernel); with a workspace too small for the partials the same
    step runs unsplit.  Both match the oracle."""
    geo = QWEN
    shape = wl.StepShape([1, 300, 130], [9000, 12000, 7000])
    c = device_case(geo, shape, seed=21, nan_fill=True)
    want = oracle_full(c)
    full = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads)
    outs = []
    for ws_bytes in (full, 1 << 20):
        out = torch.empty((shape.total_q, geo.n_q_heads, geo.head_dim), dtype=torch.float32, device="cuda")
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device="cuda")
        ppas.ppas_attention_step(c.q, c.k_cache, c.v_cache, c.num_blocks, c.tables, c.width, shape.q_lens,
                                 shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads, geo.head_dim, c.scale, out, True,
                                 ws, ws_bytes)
        torch.cuda.synchronize()
        assert_close(host64(out), want, f"workspace {ws_bytes}")
        outs.append(out)
    assert full > 1 << 20


def _many_short_chunks():
    # 130 prefill chunks (more than one launch holds) plus 3 decode rows
    rng = np.random.default_rng(5)
    q = [int(x) for x in rng.integers(2, 300, size=130)] + [1, 1, 1]
    p = [int(x) for x in rng.integers(0, 3000, size=130)] + [4000, 5000, 6000]
    return wl.StepShape(q, [a + b for a, b in zip(q, p)])


MULTI = [
    ("130 chunks + 3 decodes", QWEN, _many_short_chunks),
    # 157 query tiles x 16 head slots: more items than one launch holds
    ("one 20000-token chunk", LLAMA, lambda: wl.StepShape([20000], [20500])),
]


@pytest.mark.parametrize("name,geo,mk", MULTI, ids=[m[0] for m in MULTI])
def test_steps_planned_over_several_launches(ppas, name, geo, mk):
    shape = mk()
    c = device_case(geo, shape, seed=9, extra_blocks=16, nan_fill=True)
    out = run_step(ppas, c, False)
    torch.cuda.synchronize()
    o = out.float().cpu().numpy()
    rows = sample_rows(shape, geo.n_q_heads, 4 if len(shape.q_lens) > 10 else 256, seed=2)
    got = o[[r for r, _ in rows], [h for _, h in rows]]
    assert_close(got, oracle_rows(c, rows), name)
