"""Seeded random mixed steps against the float64 oracle: random group sizes,
chunk lengths (ragged query tiles), prefixes (unaligned pages), decode rows,
and both a full workspace (stream-K cuts and their merge, split decode) and
none at all (whole-unit plans, no prefill splits).  All decode rows and
sampled (token, head) rows of every chunk are compared."""
import numpy as np
import pytest
import torch

from _cases import assert_close, device_case, oracle_rows, sample_rows
from paper_2608_15171_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ppas():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_15171_gb300 import ppas as p
    return p


def _random_step(seed):
    rng = np.random.default_rng(1000 + seed)
    hk = int(rng.choice([1, 2, 4, 8]))
    g = int(rng.choice([1, 2, 4, 8]))
    geo = wl.Geometry(f"random{seed}", hk * g, hk, 128, 1)
    n = int(rng.integers(1, 9))
    q, c = [], []
    for _ in range(n):
        ql = 1 if rng.random() < 0.35 else int(rng.integers(2, 1500))
        p = int(rng.integers(0, 9000))
        q.append(ql)
        c.append(ql + p)
    return geo, wl.StepShape(q, c)


@pytest.mark.parametrize("seed", range(12))
@pytest.mark.parametrize("with_workspace", [True, False])
def test_random_mixed_step(ppas, seed, with_workspace):
    geo, shape = _random_step(seed)
    c = device_case(geo, shape, seed=seed, nan_fill=True)
    hq, hk, D = geo.n_q_heads, geo.n_kv_heads, geo.head_dim
    ws_full = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, hq, hk)
    # the smaller workspace holds exactly the decode rows' partials: the
    # prefill plan keeps every unit whole
    ws_bytes = ws_full
    if not with_workspace:
        dec = [(q, x) for q, x in zip(shape.q_lens, shape.ctx_lens) if q == 1]
        ws_bytes = ppas.ppas_attention_workspace_size([d[0] for d in dec], [d[1] for d in dec], hq, hk) if dec else 0
    out = torch.empty((shape.total_q, hq, D), dtype=torch.float32, device="cuda")
    ws = torch.empty(max(ws_bytes, 256), dtype=torch.uint8, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    ppas.ppas_attention_step(c.q, c.k_cache, c.v_cache, c.num_blocks, c.tables, c.width, shape.q_lens,
                             shape.ctx_lens, hq, hk, D, c.scale, out, True, ws, ws_bytes, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    o = out.cpu().numpy()
    rows = sample_rows(shape, hq, 24, seed=seed)
    got = o[[r for r, _ in rows], [h for _, h in rows]]
    assert_close(got, oracle_rows(c, rows), f"seed {seed} ws {ws_bytes} {geo.name} q={shape.q_lens}")
