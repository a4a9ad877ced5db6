"""GPU parity of decode-only steps of a few rows.

On a GB300 the plan runs the splits of these Qwen2.5-3B steps (one to
three or six rows; four rows keep plain CTAs) in thread-block clusters of
4: each CTA stores its partial into shared memory of the cluster's first
CTA, which merges them into one partial slot, so the last CTA of a (row,
kv-head) reads one partial per cluster.  Every output element is compared with the
float64 oracle; two calls over a workspace of random bytes give the same
bits; the step is one launch.
"""
import numpy as np
import pytest
import torch

from _cases import assert_close, device_case, host64, oracle_full
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

QWEN = wl.QWEN25_3B


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


@pytest.mark.parametrize("out_fp32", [False, True])
@pytest.mark.parametrize("varied", [False, True])
@pytest.mark.parametrize("n_rows", [1, 2, 3, 4, 6])
def test_decode_only_steps_of_a_few_rows(ppas, n_rows, varied, out_fp32):
    geo = QWEN
    hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
    rng = np.random.default_rng(100 + n_rows)
    if varied:
        ctx = [int(x) for x in rng.integers(9000, 31000, n_rows)]
    else:
        ctx = [int(x) for x in rng.integers(25000, 25032, n_rows)]
    shape = wl.StepShape([1] * n_rows, ctx)
    c = device_case(geo, shape, seed=70 + n_rows)
    ws_bytes = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, hq, hk)
    assert ppas.ppas_attention_kernel_count(shape.q_lens, shape.ctx_lens, hq, hk, ws_bytes) == 1
    gen = torch.Generator(device="cuda")
    gen.manual_seed(9 + n_rows)
    ws = torch.randint(0, 256, (max(ws_bytes, 1),), dtype=torch.uint8, device="cuda", generator=gen)
    outs = []
    for _ in range(2):
        out = torch.empty((shape.total_q, hq, D), dtype=torch.float32 if out_fp32 else torch.bfloat16,
                          device="cuda")
        err = torch.zeros(1, dtype=torch.int32, device="cuda")
        ppas.ppas_attention_step(c.q, c.k_cache, c.v_cache, c.num_blocks, c.tables, c.width, shape.q_lens,
                                 shape.ctx_lens, hq, hk, D, c.scale, out, out_fp32, ws, ws_bytes, err)
        torch.cuda.synchronize()
        assert err.item() == 0
        outs.append(out)
    assert torch.equal(outs[0], outs[1])
    assert_close(host64(outs[0]), oracle_full(c), f"{n_rows} decode rows")
