"""Host side of the multi-rank bench path, on CPU with gloo (world size 2).

`bench.py --gpus N` runs N independent replicas (the step has no exchange
between GPUs); the only cross-rank work is the barrier and the max over
ranks of the timed region, which is what these tests exercise.
"""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


_WORKER = r"""
import os, sys, json
sys.path.insert(0, os.environ["ROOT"])
import torch.distributed as dist
import bench
dist.init_process_group("gloo")
rank = dist.get_rank()
dist.barrier()
got = bench._max_over_ranks(dist, 10.0 + 7.5 * rank)
print(json.dumps({"rank": rank, "max": got}), flush=True)
dist.destroy_process_group()
"""


def _launch(world, code, extra_env=None):
    port = _free_port()
    procs = []
    for r in range(world):
        env = dict(os.environ, ROOT=ROOT, RANK=str(r), LOCAL_RANK=str(r), WORLD_SIZE=str(world),
                   MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), CUDA_VISIBLE_DEVICES="")
        env.update(extra_env or {})
        procs.append(subprocess.Popen([sys.executable, "-c", code], env=env, stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True, cwd=ROOT))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=180)
        assert p.returncode == 0, err[-2000:]
        outs.append(out)
    return outs


def test_max_over_ranks_gloo_world2():
    outs = _launch(2, _WORKER)
    lines = [json.loads(o.strip().splitlines()[-1]) for o in outs]
    assert sorted(l["rank"] for l in lines) == [0, 1]
    assert all(l["max"] == 17.5 for l in lines)


def test_max_over_ranks_single_process():
    sys.path.insert(0, ROOT)
    import bench
    assert bench._max_over_ranks(None, 3.25) == 3.25


def test_reference_arm_nonzero_rank_does_no_work():
    # ranks other than 0 of the reference arm return without timing anything
    sys.path.insert(0, ROOT)
    import bench

    class Args:
        steps, warmup, cpu_seconds = 1, 0, 0.1

    assert bench.run_reference(Args(), 1, 2) is None


def test_traffic_key_follows_the_device_code(tmp_path, monkeypatch):
    """The ncu traffic in the bench line is keyed by a hash of the prefill
    kernel's device code: comment and host-launcher edits keep the key, an
    edit of the kernel's code changes it (and the bench then reports null)."""
    sys.path.insert(0, ROOT)
    import bench
    src = os.path.join(ROOT, "paper_2608_15171_gb300", "csrc", "attn_prefill.cu")
    text = open(src, encoding="utf-8").read()
    assert bench.PREFILL_TRAFFIC.get(bench._src_hash("attn_prefill.cu")) is not None
    csrc = tmp_path / "paper_2608_15171_gb300" / "csrc"
    csrc.mkdir(parents=True)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))

    def key(t):
        (csrc / "attn_prefill.cu").write_text(t, encoding="utf-8")
        return bench._src_hash("attn_prefill.cu")

    base = key(text)
    cut = text.index("\ncudaError_t launch_")
    assert key(text.replace("// ", "//  note: ", 1)) == base
    assert key(text[:cut] + "\n// a launcher comment" + text[cut:].replace("return", "return ", 1)) == base
    assert key(text[:cut].replace("kNK = 3", "kNK = 2", 1) + text[cut:]) != base
