"""Host plan of the split-K decode kernel (CPU).

A small C++ program (tests/native/decode_plan_check.cpp), compiled against
the built library, plans each step's decode rows the way the attention call
does and checks what the kernel indexes from the plan: which rows decode,
the pages each split covers (every page exactly once, no empty split), the
split bounds the kernel's shared memory relies on, and the workspace sizes.
The paper's decode workloads must fit one wave of CTAs unless the
1024-page limit of a split needs more.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

from paper_2608_15171_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2608_15171_gb300")
LIB = os.path.join(PKG, "libppas.so")


@pytest.fixture(scope="module")
def checker(tmp_path_factory):
    if not os.path.exists(LIB):
        pytest.skip("libppas.so is not built")
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("no g++")
    exe = str(tmp_path_factory.mktemp("dplan") / "decode_plan_check")
    cmd = [gxx, "-std=c++17", "-O1", "-I", os.path.join(ROOT, "include"), "-I", os.path.join(PKG, "csrc"),
           "-I", "/usr/local/cuda/include", os.path.join(ROOT, "tests", "native", "decode_plan_check.cpp"),
           "-o", exe, "-L", PKG, "-lppas", f"-Wl,-rpath,{PKG}", "-L/usr/local/cuda/lib64", "-lcudart"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    return exe


def _run(exe, cases, sms=152):
    text = "".join(f"{sms} {hq} {hk} {len(q)} " + " ".join(map(str, q)) + " " + " ".join(map(str, c)) + "\n"
                   for hq, hk, q, c in cases)
    out = subprocess.run([exe], input=text, capture_output=True, text=True, check=True).stdout.split("\n")
    lines = [l for l in out if l]
    assert len(lines) == len(cases)
    return lines


@pytest.mark.parametrize("sms", [152, 148, 132])
def test_paper_decode_workloads_fit_one_wave_unless_capped(checker, sms):
    q3, l8 = wl.QWEN25_3B, wl.LLAMA31_8B
    cases = [("MBT 2k + 8 decodes", q3, wl.high_pressure_step(0)),
             ("Llama 16384 + 4 decodes", l8, wl.llama_hi_step(0)),
             ("Llama 3 chunks + 16 decodes", l8, wl.llama_lo_step(0))]
    cases += [(f"tiny step {i}", q3, s) for i, s in enumerate(wl.tiny_steps()) if 1 in s.q_lens]
    lines = _run(checker, [(g.n_q_heads, g.n_kv_heads, list(s.q_lens), list(s.ctx_lens)) for _, g, s in cases],
                 sms)
    for (name, geo, shape), line in zip(cases, lines):
        assert line.startswith("ok"), f"{name}: {line}"
        # one wave of CTAs (one per SM), unless rows need more splits than
        # their share because a split holds at most 1024 pages
        capped = sum(-(-wl.blocks_for(c) // 1024) for q, c in zip(shape.q_lens, shape.ctx_lens) if q == 1)
        assert int(line.split()[1]) <= max(sms, capped * geo.n_kv_heads), f"{name}: {line}"


@pytest.mark.parametrize("sms", [152, 132])
def test_random_and_extreme_decode_plans(checker, sms):
    rng = np.random.default_rng(5)
    cases = []
    for _ in range(80):
        n = int(rng.integers(1, 40))
        q = [1 if rng.random() < 0.7 else int(rng.integers(2, 3000)) for _ in range(n)]
        c = [x + int(rng.integers(0, 120000)) for x in q]
        hk = int(rng.choice([1, 2, 4, 8]))
        g = int(rng.choice([1, 2, 4, 8]))
        cases.append((hk * g, hk, q, c))
    cases.append((16, 2, [1] * 300, [1 + 97 * i for i in range(300)]))  # more rows than CTAs
    cases.append((32, 8, [1], [1]))                                      # one key
    cases.append((16, 2, [1, 1], [1 << 20, 17]))                         # a million-token row
    cases.append((16, 2, [1], [1 << 25]))                                 # the longest decode row
    for case, line in zip(cases, _run(checker, cases, sms)):
        assert line.startswith("ok"), f"{case[:2]} {len(case[2])} rows: {line}"


def test_cluster_plans_only_where_the_merge_bounds_the_step(checker):
    """With the co-resident cluster capacity of a GB300 (36 clusters of 4 of
    the decode kernel), the plan puts the splits of a Qwen2.5-3B step of one
    or two decode rows into clusters of 4 (the split merge reads a quarter of
    the partials) and keeps plain CTAs where clusters would leave SMs idle or
    unbalance the splits (4 and 8 rows, 16 Llama rows), and for any step with
    prefill rows (a mixed launch has no clusters)."""
    q3, l8 = wl.QWEN25_3B, wl.LLAMA31_8B
    cases = [("qwen 1 row", q3, [1], [25000], 4),
             ("qwen 2 rows", q3, [1, 1], [25000, 25020], 4),
             ("qwen 4 rows", q3, [1] * 4, [25000, 25010, 25020, 25030], 1),
             ("qwen 8 rows", q3, [1] * 8, [25000 + 4 * i for i in range(8)], 1),
             ("llama 16 rows", l8, [1] * 16, [30000 + 4 * i for i in range(16)], 1),
             ("qwen 1 row beside a chunk", q3, [1, 512], [25000, 2048], 1)]
    lines = _run(checker, [(g.n_q_heads, g.n_kv_heads, q, c) for _, g, q, c, _ in cases])
    for (name, _, _, _, want), line in zip(cases, lines):
        assert line.startswith("ok"), f"{name}: {line}"
        assert int(line.split()[3]) == want, f"{name}: {line}"
