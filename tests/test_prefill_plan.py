"""Host plan of the persistent prefill kernel (CPU).

A small C++ program (tests/native/plan_check.cpp), compiled against the
built library, plans each step the way the attention call does and checks
every index the kernel derives from the plan (capacities, KV ranges, pages
read, partial slots, merge entries) and that the items of every (query tile,
head slot) cover its causal KV tiles exactly once, with and without splits.
The paper's workloads must also come out balanced over the CTAs.
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
    exe = str(tmp_path_factory.mktemp("plan") / "plan_check")
    cuda_inc = "/usr/local/cuda/include"
    cmd = [gxx, "-std=c++17", "-O1", "-I", os.path.join(ROOT, "include"), "-I", os.path.join(PKG, "csrc"),
           "-I", cuda_inc, os.path.join(ROOT, "tests", "native", "plan_check.cpp"), "-o", exe,
           "-L", PKG, "-lppas", f"-Wl,-rpath,{PKG}", "-L/usr/local/cuda/lib64", "-lcudart"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    return exe


def _run(exe, cases, sms=152):
    text = "".join(f"{sms} {hq} {hk} {len(q)} " + " ".join(map(str, q)) + " " + " ".join(map(str, c)) + "\n"
                   for hq, hk, q, c in cases)
    out = subprocess.run([exe], input=text, capture_output=True, text=True, check=True).stdout.split("\n")
    lines = [l for l in out if l]
    assert len(lines) == 2 * len(cases)
    return [(lines[2 * i], lines[2 * i + 1]) for i in range(len(cases))]


def _paper_cases():
    q3, l8 = wl.QWEN25_3B, wl.LLAMA31_8B
    cases = [(name, geo, shape) for name, geo, shape in [
        ("MBT 16k iteration 1", q3, wl.low_pressure_steps()[0]),
        ("MBT 16k iteration 2", q3, wl.low_pressure_steps()[1]),
        ("MBT 2k + 8 decodes", q3, wl.high_pressure_step(0)),
        ("Llama 16384 + 4 decodes", l8, wl.llama_hi_step(0)),
        ("Llama 3 chunks + 16 decodes", l8, wl.llama_lo_step(0)),
    ]]
    cases += [(f"tiny step {i}", q3, s) for i, s in enumerate(wl.tiny_steps())]
    return cases


@pytest.mark.parametrize("sms", [152, 148, 132])
def test_paper_workloads_plan_valid_and_balanced(checker, sms):
    """Plans for GB300's 152 SMs and for parts (or partitions) with fewer."""
    cases = _paper_cases()
    res = _run(checker, [(g.n_q_heads, g.n_kv_heads, list(s.q_lens), list(s.ctx_lens)) for _, g, s in cases], sms)
    for (name, _, _), (split, whole) in zip(cases, res):
        assert split.startswith("ok"), f"{name}: {split}"
        assert whole.startswith("ok"), f"{name}: {whole}"
        if not name.startswith("tiny"):
            f = split.split()
            assert int(f[1]) == 1, f"{name}: one launch expected"
            assert float(f[5]) <= 1.10 * float(f[6]), f"{name}: CTA loads {f[5]} vs mean {f[6]}"


@pytest.mark.parametrize("sms", [152, 132, 256])
def test_random_steps_plan_valid(checker, sms):
    rng = np.random.default_rng(11)
    cases = []
    for _ in range(60):
        n = int(rng.integers(1, 24))
        q = [1 if rng.random() < 0.4 else int(rng.integers(2, 4000)) for _ in range(n)]
        c = [x + int(rng.integers(0, 40000)) for x in q]
        hk = int(rng.choice([1, 2, 4, 8]))
        g = int(rng.choice([1, 2, 4, 8]))
        cases.append((hk * g, hk, q, c))
    # more sequences than one launch holds, and more items than one launch holds
    cases.append((16, 2, [200] * 150 + [1] * 5, [200 + 37 * i for i in range(150)] + [30000] * 5))
    cases.append((32, 8, [20000], [20500]))
    cases.append((32, 8, [65536], [66536]))
    cases.append((16, 2, [130], [130 + (1 << 19)]))  # a chunk over a 512k-token prefix
    # chunks at the longest context the kernel takes, and units just over,
    # at and under the piece cap
    cases.append((16, 2, [256], [65535 * 128]))
    cases.append((32, 8, [128, 300], [65535 * 128 - 7, 4_000_000]))
    for kt in (511, 512, 513, 515, 516, 1024, 1025):
        cases.append((16, 2, [128], [kt * 128]))
    for case, (split, whole) in zip(cases, _run(checker, cases, sms)):
        assert split.startswith("ok"), f"{case[:2]} {len(case[2])} seqs: {split}"
        assert whole.startswith("ok"), f"{case[:2]} {len(case[2])} seqs: {whole}"
