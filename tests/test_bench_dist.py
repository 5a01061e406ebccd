"""bench.py's multi-process timing path on CPU: two gloo ranks, the max-over-ranks reduction,
the whole-job (weak scaling) rate, and the reference arm's rank handling.  No GPU, no kernels."""
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_WORKER = r'''
import os, sys, json
sys.path.insert(0, sys.argv[1])
import bench
world, rank, local = bench.dist_setup(2, backend="gloo")
ms = 10.0 * (rank + 1)                      # rank 1 is the slower one
ms_max = bench.barrier_max(ms, world)
rate = bench.whole_job_rate(world, 65536, ms_max)
print(json.dumps({"rank": rank, "world": world, "ms_max": ms_max, "rate": rate}))
import torch.distributed as dist
dist.destroy_process_group()
'''


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_reduce_max_and_weak_scaling_rate():
    port = _free_port()
    procs = []
    for rank in range(2):
        env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2",
                   MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        procs.append(subprocess.Popen([sys.executable, "-c", _WORKER, ROOT], env=env,
                                      stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=120)
        assert p.returncode == 0, err
        outs.append(__import__("json").loads(out.strip().splitlines()[-1]))
    for o in outs:
        assert o["world"] == 2
        assert o["ms_max"] == 20.0                       # the slowest rank's time
        assert o["rate"] == pytest.approx(2 * 65536 / 0.020)   # all ranks' tokens over that time
    assert sorted(o["rank"] for o in outs) == [0, 1]


def test_single_process_needs_no_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.barrier_max(3.5, 1) == 3.5
    assert bench.whole_job_rate(1, 1000, 1.0) == pytest.approx(1e6)


def test_reference_arm_non_zero_rank_exits_quietly():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""


def _bench_module():
    import importlib.util
    spec = importlib.util.spec_from_file_location("bench_for_digest", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    argv = sys.argv
    sys.argv = ["bench.py"]
    try:
        spec.loader.exec_module(mod)
    finally:
        sys.argv = argv
    return mod


def test_source_digest_ignores_comments_only():
    b = _bench_module()
    src = 'int a = 1; // note\nconst char *s = "//kept"; /* block\n comment */ char c = \'/\';\n'
    assert b._strip_comments(src) == 'int a = 1; \nconst char *s = "//kept";  char c = \'/\';\n'
    # a comment edit keeps the stripped text, a code edit changes it
    assert b._strip_comments(src.replace("note", "other note")) == b._strip_comments(src)
    assert b._strip_comments(src.replace("a = 1", "a = 2")) != b._strip_comments(src)
    # the digest also ignores line breaks and indentation (a comment that grows by a line)
    def digest(text):
        return " ".join(b._strip_comments(text).split())
    assert digest(src.replace("// note", "// note\n    // more")) == digest(src)


def test_stored_traffic_is_plausible_when_current():
    # bench.py reports a pass's DRAM traffic only while the figure under profiles/ was captured from
    # the current pass kernels; such a figure lies near the pass's algorithmic bytes (809.5 MB)
    b = _bench_module()
    for kern in ("kpass", "vpass"):
        t = b.stored_traffic(kern, 65536)
        if t is None:
            pytest.skip("the %s traffic figure predates the current sources" % kern)
        assert 7e8 < t < 1e9, (kern, t)
        assert b.stored_traffic(kern, 32768) == t / 2
