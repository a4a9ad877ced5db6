"""The attention entry point that allocates nothing.

Some callers cannot call cudaMalloc (a serving loop that gave all of HBM to
its KV-cache pool at start-up, or a program whose device memory belongs to
another allocator).  ``ppas_attention_step_noalloc`` takes only inputs and
outputs and keeps its scratch in the library's fixed device array.

These tests run it through the C ABI, two calls in a row each time, and check
every output against the float64 oracle:

* the MBT 2048 step (4 chunks + 8 multi-split decode rows in one mixed
  launch), whose whole plan (decode split partials and the prefill tiles'
  stream-K partials, merged by the merge launch) fits the array: it must also
  equal the ordinary entry point with a caller-owned workspace bit for bit
  (same plan);
* a 130-token chunk over a ~100k-token prefix plus a decode row, whose prefill
  units are longer than one piece may be and are always cut: the stream-K
  partials live in the fixed array beside the decode partials;
* a step whose prefill partials do not fit beside the decode partials, so the
  prefill tiles run unsplit (sampled rows against the oracle);
* a step whose decode scratch alone exceeds the array is rejected.

The file is collected last, so a run that stops at the first failure has run
every other test before it.
"""
import numpy as np
import pytest
import torch

from _cases import assert_close, device_case, host64, oracle_full, oracle_rows, run_step, sample_rows
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


def _noalloc(ppas, c, out_fp32=True):
    geo, shape = c.geo, c.shape
    out = torch.full((shape.total_q, geo.n_q_heads, geo.head_dim), float("nan"),
                     dtype=torch.float32 if out_fp32 else torch.bfloat16, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ppas.ppas_attention_step_noalloc(c.q, c.k_cache, c.v_cache, c.num_blocks, c.tables, c.width, shape.q_lens,
                                     shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads, geo.head_dim, c.scale, out,
                                     out_fp32, err)
    torch.cuda.synchronize()
    assert err.item() == 0, f"device error flag {err.item()}"
    return out


def _kernels(ppas, shape, geo, ws):
    return ppas.ppas_attention_kernel_count(shape.q_lens, shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads, ws)


def test_noalloc_mbt2k_step_against_oracle_twice(ppas):
    geo = wl.QWEN25_3B
    shape = wl.high_pressure_step(0)          # 8 decode rows of ~25k context (several splits) + 4 chunks
    full = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads)
    assert 0 < full <= ppas.PPAS_NOALLOC_SCRATCH_BYTES
    # one mixed launch + the merge of the cut units, as with a full workspace
    assert _kernels(ppas, shape, geo, ppas.PPAS_NOALLOC_SCRATCH_BYTES) == _kernels(ppas, shape, geo, full) == 2
    c = device_case(geo, shape, seed=5)
    want = oracle_full(c)
    ref = host64(run_step(ppas, c, out_fp32=True))
    for _ in range(2):
        got = host64(_noalloc(ppas, c))
        assert_close(got, want, "noalloc MBT 2k step vs oracle")
        assert np.array_equal(got, ref), "noalloc differs from the workspace entry point on the same plan"


def test_noalloc_stream_k_pieces_in_the_fixed_array(ppas):
    geo = wl.QWEN25_3B
    shape = wl.StepShape([1, 130], [25003, 100130])
    full = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads)
    dec = ppas.ppas_attention_workspace_size([1], [25003], geo.n_q_heads, geo.n_kv_heads)
    assert dec < full <= ppas.PPAS_NOALLOC_SCRATCH_BYTES   # prefill partials beside the decode partials
    assert _kernels(ppas, shape, geo, ppas.PPAS_NOALLOC_SCRATCH_BYTES) == 2   # mixed launch + merge
    c = device_case(geo, shape, seed=9)
    want = oracle_full(c)
    ref = host64(run_step(ppas, c, out_fp32=True))
    for _ in range(2):
        got = host64(_noalloc(ppas, c))
        assert_close(got, want, "noalloc stream-K step vs oracle")
        assert np.array_equal(got, ref), "noalloc differs from the workspace entry point on the same plan"


def test_noalloc_prefill_unsplit_when_its_partials_do_not_fit(ppas):
    geo = wl.QWEN25_3B
    shape = wl.StepShape([1] + [1024] * 4, [25011] + [65536 + 1024] * 4)
    full = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads)
    assert full > ppas.PPAS_NOALLOC_SCRATCH_BYTES
    # without room for the pieces the plan keeps every unit whole (one mixed launch)
    assert _kernels(ppas, shape, geo, ppas.PPAS_NOALLOC_SCRATCH_BYTES) == 1
    c = device_case(geo, shape, seed=13)
    rows = sample_rows(shape, geo.n_q_heads, 48, seed=13)
    want = oracle_rows(c, rows)
    for _ in range(2):
        got = _noalloc(ppas, c)
        sel = np.stack([host64(got[r, h]) for r, h in rows])
        assert_close(sel, want, "noalloc unsplit prefill vs oracle (sampled rows)")


def test_noalloc_rejects_steps_beyond_its_scratch(ppas):
    geo = wl.LLAMA31_8B
    q_lens, ctx_lens = [1] * 4, [1 << 25] * 4          # 2048 decode splits a row
    need = ppas.ppas_attention_workspace_size(q_lens, ctx_lens, geo.n_q_heads, geo.n_kv_heads)
    assert need > ppas.PPAS_NOALLOC_SCRATCH_BYTES
    # rejected on the host before anything touches the (dummy) pointers
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_attention_step_noalloc(16, 16, 16, 1, 16, 1 << 21, q_lens, ctx_lens, geo.n_q_heads,
                                         geo.n_kv_heads, geo.head_dim, geo.scale, 16, True)
    assert e.value.status == ppas.PPAS_ERR_CAPACITY
