"""Shared helpers for the GPU parity tests: build a seeded step on the device,
run it through the C ABI, and compare with the oracle."""
import numpy as np
import torch

from oracle import attention as oa
from paper_2608_15171_gb300 import workloads as wl

# attention tolerance on bf16 inputs with fp32 accumulation
MAX_ABS = 2e-2
MEAN_ABS = 2e-3


class Case:
    pass


def device_case(geo, shape, seed, nan_fill=False, extra_blocks=5, device="cuda"):
    """Q, paged K/V caches and block tables for one literal step shape.

    Every context token of every sequence holds N(0,1) bf16 keys/values; with
    ``nan_fill`` every slot that no sequence's context covers (the tail of the
    last page, unused blocks) holds NaN, which the kernels must never read
    into a result.
    """
    c = Case()
    c.geo, c.shape = geo, shape
    need = sum(wl.blocks_for(x) for x in shape.ctx_lens)
    c.num_blocks = need + extra_blocks
    perm = wl.page_permutation(c.num_blocks, seed)
    c.tables_np = wl.literal_tables(shape, perm)
    c.width = c.tables_np.shape[1]
    D, hq, hk = geo.head_dim, geo.n_q_heads, geo.n_kv_heads
    c.k_cache = wl.bf16_normal((c.num_blocks, hk, 16, D), seed * 7 + 1, device)
    c.v_cache = wl.bf16_normal((c.num_blocks, hk, 16, D), seed * 7 + 2, device)
    if nan_fill:
        covered = torch.zeros(c.num_blocks * 16, dtype=torch.bool)
        for s, ctx in enumerate(shape.ctx_lens):
            pos = torch.arange(ctx)
            blk = torch.from_numpy(c.tables_np[s]).long()[pos // 16]
            covered[blk * 16 + pos % 16] = True
        hole = (~covered).view(c.num_blocks, 1, 16, 1).to(device)
        c.k_cache.masked_fill_(hole, float("nan"))
        c.v_cache.masked_fill_(hole, float("nan"))
    c.q = wl.bf16_normal((shape.total_q, hq, D), seed * 7 + 3, device)
    c.tables = torch.from_numpy(c.tables_np).to(device)
    c.scale = geo.scale
    return c


def run_step(ppas, c, out_fp32=False, stream=None, err=None):
    geo = c.geo
    out = torch.empty((c.shape.total_q, geo.n_q_heads, geo.head_dim),
                      dtype=torch.float32 if out_fp32 else torch.bfloat16, device=c.q.device)
    ws_bytes = ppas.ppas_attention_workspace_size(c.shape.q_lens, c.shape.ctx_lens, geo.n_q_heads,
                                                  geo.n_kv_heads)
    ws = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=c.q.device)
    ppas.ppas_attention_step(c.q, c.k_cache, c.v_cache, c.num_blocks, c.tables, c.width,
                             c.shape.q_lens, c.shape.ctx_lens, geo.n_q_heads, geo.n_kv_heads,
                             geo.head_dim, c.scale, out, out_fp32, ws, ws_bytes, err, stream)
    return out


def host64(t):
    return t.detach().to("cpu", torch.float64).numpy()


def oracle_full(c):
    return oa.paged_attention(host64(c.q), host64(c.k_cache), host64(c.v_cache), c.tables_np,
                              c.shape.q_lens, c.shape.ctx_lens, c.scale)


def host32(t):
    """float32 host copy (exact for bf16; the oracle widens to float64)."""
    return t.detach().to("cpu", torch.float32).numpy()


def oracle_rows(c, rows, kc=None, vc=None):
    kc = host32(c.k_cache) if kc is None else kc
    vc = host32(c.v_cache) if vc is None else vc
    return oa.sampled_rows(host64(c.q), kc, vc, c.tables_np, c.shape.q_lens, c.shape.ctx_lens, c.scale, rows)


def sample_rows(shape, n_q_heads, per_chunk, seed):
    """All heads of every decode row plus ``per_chunk`` seeded (token, head)
    pairs per prefill chunk, always including each chunk's first and last
    token."""
    rng = np.random.default_rng(seed)
    rows, start = [], 0
    for q in shape.q_lens:
        if q == 1:
            rows += [(start, h) for h in range(n_q_heads)]
        else:
            ts = list(rng.integers(0, q, size=per_chunk)) + [0, q - 1]
            hs = list(rng.integers(0, n_q_heads, size=per_chunk)) + [0, n_q_heads - 1]
            rows += [(start + int(t), int(h)) for t, h in zip(ts, hs)]
        start += q
    return rows


def assert_close(got, want, what=""):
    got = np.asarray(got, dtype=np.float64)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    err = np.abs(got - want)
    assert err.max() <= MAX_ABS, f"{what}: max abs err {err.max():.3e}"
    assert err.mean() <= MEAN_ABS, f"{what}: mean abs err {err.mean():.3e}"
    return float(err.max()), float(err.mean())
