"""The attention entry point that allocates nothing.

Some callers cannot call cudaMalloc (a serving loop that gave all of HBM to
its KV-cache pool at start-up, or a program whose device memory belongs to
another allocator).  ``ppas_attention_step_noalloc`` takes only inputs and
outputs and keeps its split-K scratch in the library's fixed device array.
This test checks it against the ordinary entry point (with a caller-owned
workspace) on a step with multi-split decode rows, for two calls in a row,
and that a step needing more scratch than the array holds is rejected.
"""
import pytest
import torch

from _cases import assert_close, device_case, host64, run_step
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


def test_noalloc_matches_workspace_entry_point_twice(ppas):
    geo = wl.QWEN25_3B
    shape = wl.high_pressure_step(0)          # 8 decode rows of ~25k context (several splits) + 4 chunks
    # the decode rows' split scratch fits the fixed array; the prefill chunks
    # then run without KV splits (their partials would not fit)
    dec = [i for i, q in enumerate(shape.q_lens) if q == 1]
    need = ppas.ppas_attention_workspace_size([1] * len(dec), [shape.ctx_lens[i] for i in dec], geo.n_q_heads,
                                              geo.n_kv_heads)
    assert 0 < need <= ppas.PPAS_NOALLOC_SCRATCH_BYTES
    c = device_case(geo, shape, seed=5)
    want = run_step(ppas, c, out_fp32=True)
    for _ in range(2):
        out = torch.full_like(want, float("nan"))
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        ppas.ppas_attention_step_noalloc(c.q, c.k_cache, c.v_cache, c.num_blocks, c.tables, c.width,
                                         shape.q_lens, shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads,
                                         geo.head_dim, c.scale, out, True, err)
        torch.cuda.synchronize()
        assert err.item() == 0
        assert_close(host64(out), host64(want), "noalloc vs workspace entry point")


def test_noalloc_rejects_steps_beyond_its_scratch(ppas):
    geo = wl.LLAMA31_8B
    q_lens, ctx_lens = [1] * 256, [30000] * 256
    need = ppas.ppas_attention_workspace_size(q_lens, ctx_lens, geo.n_q_heads, geo.n_kv_heads)
    assert need > ppas.PPAS_NOALLOC_SCRATCH_BYTES
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_attention_step_noalloc(16, 16, 16, 1, 16, 2048, q_lens, ctx_lens, geo.n_q_heads, geo.n_kv_heads,
                                         geo.head_dim, geo.scale, 16, True)
    assert e.value.status == ppas.PPAS_ERR_CAPACITY
