"""bench.py host logic on CPU: multi-rank aggregation (two gloo ranks) and the
reference arm's JSON line."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, ms, units, out_q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        out_q.put((rank, bench.aggregate(ms[rank], units[rank], world, device="cpu")))
    finally:
        dist.destroy_process_group()


def test_aggregate_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ms, units = [0.25, 0.4], [16, 16]
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, ms, units, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        assert res[r] == (0.4, 32.0)      # max step time, branches summed over ranks


def test_aggregate_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate(1.5, 7, 1) == (1.5, 7)


def test_reference_arm_json_line():
    env = {**os.environ, "OMP_NUM_THREADS": "2"}
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--config", "1", "--steps", "3", "--warmup", "3"],
                         capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert res.returncode == 0, res.stderr[-2000:]
    line = json.loads(res.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "branch-tokens/s"
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0
    assert line["config"]["workload"] == "tiny_fork_h8_2_d64"


def test_kernel_source_hash_ignores_comments_only():
    """The hash that keys the stored DRAM counters sees code, not comments or
    layout: a comment edit keeps it, a code edit (even inside a string
    literal that looks like a comment) changes it."""
    sys.path.insert(0, ROOT)
    import bench
    tok = bench._code_tokens
    base = 'int a = 1; // note\n/* block\n comment */ const char *s = "// kept";\n'
    assert tok(base) == tok(base.replace("note", "other note").replace("block", "x"))
    assert tok(base) == tok(base.replace("int a = 1;", "int  a =\n 1;"))
    assert tok(base) != tok(base.replace("int a = 1;", "int a = 2;"))
    assert tok(base) != tok(base.replace('"// kept"', '"// changed"'))
    assert "kept" in tok(base) and "note" not in tok(base) and "block" not in tok(base)
    assert tok("char c = '\\'';  // q") == "char c = '\\'';"
    h = bench.kernel_source_hash()
    assert len(h) == 16 and int(h, 16) >= 0
