"""The C-ABI library loads and exports every entry point ``include/ppas.h``
declares; host-side argument checks reject bad input before any device work
(CPU only: no compute call reaches a kernel)."""
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def ppas():
    lib = os.path.join(ROOT, "paper_2608_15171_gb300", "libppas.so")
    if not os.path.exists(lib):
        from paper_2608_15171_gb300 import build
        build.build()
    from paper_2608_15171_gb300 import ppas as p
    return p


def _declared():
    src = open(os.path.join(ROOT, "include", "ppas.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ppas_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(ppas):
    names = _declared()
    assert len(names) == len(ppas.EXPORTED)
    for n in names:
        assert hasattr(ppas._lib, n), n
    assert sorted(ppas.EXPORTED) == names


def test_status_strings_and_version(ppas):
    assert ppas.ppas_abi_version() == 1
    for code in (0, -1, -2, -3, -4, -5):
        assert ppas.ppas_status_string(code) != "unknown status"


def test_attention_argument_errors_before_device_work(ppas):
    E = ppas.PpasError
    ok = dict(q=16, k_cache=16, v_cache=16, num_blocks=4, d_block_tables=16, max_blocks_per_seq=4,
              q_lens=[2], ctx_lens=[5], n_q_heads=16, n_kv_heads=2, head_dim=128, scale=0.1, out=16,
              out_is_fp32=False, stream=0)

    def call(**kw):
        a = dict(ok)
        a.update(kw)
        ppas.ppas_attention_step(**a)

    with pytest.raises(E) as e:
        call(head_dim=64)
    assert e.value.status == ppas.PPAS_ERR_UNSUPPORTED
    with pytest.raises(E) as e:
        call(n_q_heads=12, n_kv_heads=1)
    assert e.value.status == ppas.PPAS_ERR_UNSUPPORTED
    with pytest.raises(E) as e:
        call(n_q_heads=15)
    assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    for ql, cl in (([0], [5]), ([6], [5]), ([2], [65])):
        with pytest.raises(E) as e:
            call(q_lens=ql, ctx_lens=cl)
        assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    with pytest.raises(E) as e:
        call(q=8)  # not 16-byte aligned
    assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    with pytest.raises(E) as e:
        call(scale=-1.0)
    assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    # a prefill row past 65535 KV tiles of 128 keys (16-bit tile indices) is refused
    with pytest.raises(E) as e:
        call(q_lens=[2], ctx_lens=[65535 * 128 + 1], max_blocks_per_seq=65535 * 8 + 1)
    assert e.value.status == ppas.PPAS_ERR_UNSUPPORTED
    assert ppas.ppas_attention_kernel_count([2], [65535 * 128], 16, 2, 0) >= 1  # the limit itself is accepted
    # a decode row longer than 2^25 tokens (2048 splits of 1024 pages) is refused
    big = (1 << 25) + 16
    with pytest.raises(E) as e:
        call(q_lens=[1], ctx_lens=[big], max_blocks_per_seq=big // 16 + 1)
    assert e.value.status == ppas.PPAS_ERR_UNSUPPORTED
    # empty step is a no-op
    call(q_lens=[], ctx_lens=[])


def test_kv_append_argument_errors(ppas):
    with pytest.raises(ppas.PpasError):
        ppas.ppas_kv_append(16, 16, 16, -1, 16, 16, 4, 2, 128, None, 0)
    with pytest.raises(ppas.PpasError):
        ppas.ppas_kv_append(16, 16, 16, 3, 16, 16, 4, 2, 12, None, 0)
    ppas.ppas_kv_append(16, 16, 16, 0, 16, 16, 4, 2, 128, None, 0)  # no-op
    # 2^27 tokens x 2 heads x 16 chunks = 2^32 elements: over the 32-bit index range
    with pytest.raises(ppas.PpasError, match="UNSUPPORTED|unsupported"):
        ppas.ppas_kv_append(16, 16, 16, 1 << 27, 16, 16, 4, 2, 128, None, 0)


def test_workspace_size_is_a_pure_function_of_lengths(ppas):
    a = ppas.ppas_attention_workspace_size([1, 1, 512], [25000, 25010, 3000], 16, 2)
    b = ppas.ppas_attention_workspace_size([1, 1, 512], [25000, 25010, 3000], 16, 2)
    assert a == b and a > 0 and a % 256 == 0
    # a short chunk with no prefix: no decode rows and no split-KV ranges
    assert ppas.ppas_attention_workspace_size([512], [512], 16, 2) == 0
    # a chunk over a long prefix is split over its KV range: partials need room
    assert ppas.ppas_attention_workspace_size([512], [24000], 16, 2) > 0
    assert ppas.ppas_attention_workspace_size([], [], 16, 2) == 0


def test_kernel_count_follows_the_plan(ppas):
    from paper_2608_15171_gb300 import workloads as wl
    # one prefill launch (whole units) for the 16k chunk with no prefix
    it1, it2 = wl.low_pressure_steps()
    assert ppas.ppas_attention_kernel_count(it1.q_lens, it1.ctx_lens, 16, 2, 0) == 1
    # the chunk over a 16k prefix is cut into pieces when the workspace holds
    # their partials: prefill launch + merge launch; without it, one launch
    ws = ppas.ppas_attention_workspace_size(it2.q_lens, it2.ctx_lens, 16, 2)
    assert ws > 0
    assert ppas.ppas_attention_kernel_count(it2.q_lens, it2.ctx_lens, 16, 2, ws) == 2
    assert ppas.ppas_attention_kernel_count(it2.q_lens, it2.ctx_lens, 16, 2, 0) == 1
    # decode rows alone: one decode launch; decode rows with a chunk: one
    # mixed launch, and its merge launch when the plan cuts units
    assert ppas.ppas_attention_kernel_count([1, 1], [3000, 5000], 16, 2, 1 << 30) == 1
    assert ppas.ppas_attention_kernel_count([1, 1, 512], [3000, 5000, 9000], 16, 2, 1 << 30) == 2
    assert ppas.ppas_attention_kernel_count([1, 1, 512], [3000, 5000, 9000], 16, 2, 0) == 1
    # the paper's mixed workloads: the MBT 16k Llama step (whole units) is one
    # launch; the MBT 2k steps cut units to balance the SMs (mixed + merge)
    for shape, hq, hk, n in ((wl.high_pressure_step(0), 16, 2, 2), (wl.llama_hi_step(0), 32, 8, 1),
                             (wl.llama_lo_step(0), 32, 8, 2)):
        ws = ppas.ppas_attention_workspace_size(shape.q_lens, shape.ctx_lens, hq, hk)
        assert ppas.ppas_attention_kernel_count(shape.q_lens, shape.ctx_lens, hq, hk, ws) == n
        assert ppas.ppas_attention_kernel_count(shape.q_lens, shape.ctx_lens, hq, hk, 0) == 1
    # more sequences than one launch holds (whole units): two prefill launches,
    # and with decode rows beside them a decode launch as well
    assert ppas.ppas_attention_kernel_count([200] * 150, [200 + 37 * i for i in range(150)], 16, 2, 1 << 30) == 2
    assert ppas.ppas_attention_kernel_count([1] + [200] * 150, [900] + [200 + 37 * i for i in range(150)], 16, 2,
                                            1 << 30) == 3
    assert ppas.ppas_attention_kernel_count([], [], 16, 2, 0) == 0
    with pytest.raises(ppas.PpasError):
        ppas.ppas_attention_kernel_count([0], [5], 16, 2, 0)
    with pytest.raises(ppas.PpasError):
        ppas.ppas_attention_kernel_count([4], [8], 16, 3, 0)


def test_gateup_argument_errors_before_device_work(ppas):
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_gateup_swiglu(16, 16, 16, 4, 100, 256, None, 0)   # hidden not a multiple of 64
    assert e.value.status == ppas.PPAS_ERR_UNSUPPORTED
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_gateup_swiglu(16, 16, 16, 4, 128, 200, None, 0)   # inter not a multiple of 128
    assert e.value.status == ppas.PPAS_ERR_UNSUPPORTED
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_gateup_swiglu(0, 16, 16, 4, 128, 256, None, 0)    # null input
    assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_gateup_swiglu(16, 16, 16, -1, 128, 256, None, 0)
    assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
    ppas.ppas_gateup_swiglu(16, 16, 16, 0, 128, 256, None, 0)       # no tokens: no-op
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_gateup_pack(16, 16, 64, 100, 0)
    assert e.value.status == ppas.PPAS_ERR_UNSUPPORTED
    with pytest.raises(ppas.PpasError) as e:
        ppas.ppas_gateup_pack(8, 16, 64, 128, 0)                     # misaligned
    assert e.value.status == ppas.PPAS_ERR_INVALID_ARG
