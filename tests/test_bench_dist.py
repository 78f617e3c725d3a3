"""bench.py's multi-rank aggregation (replicas only): each rank times its own
replica; the job reports the maximum time over ranks and the sum of the
tokens.  Two gloo ranks on the CPU."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    r, w, local = bench.dist_env()
    d = bench.Dist(w, local)
    d.barrier()
    t_max = d.max(10.0 + rank)          # slowest rank decides the job time
    tokens = d.sum(64.0 * (rank + 1))   # every rank's replica contributes its tokens
    d.close()
    q.put((r, w, t_max, tokens))


def test_two_ranks_take_max_time_and_sum_tokens():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in procs)
    assert [x[0] for x in res] == [0, 1]
    for _, w, t_max, tokens in res:
        assert w == 2
        assert t_max == pytest.approx(11.0)
        assert tokens == pytest.approx(64.0 + 128.0)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    d = bench.Dist(1, 0)
    assert d.max(3.5) == 3.5 and d.sum(2.0) == 2.0
    d.barrier()
    d.close()


def test_timed_steps_are_exact_with_several_steps_per_graph():
    sys.path.insert(0, ROOT)
    import bench
    for steps in (1, 4, 7, 11, 16, 32, 64, 100):
        k = bench.steps_per_graph(steps)
        assert 1 <= k <= bench.GRAPH_STEPS and steps % k == 0
        assert (steps // k) * k == steps
        # eager warm-up, whole graphs of warm-up, then the timed steps
        for warmup in (1, 3, 5):
            cap = bench.graph_capacity(steps, warmup)
            assert cap == warmup + k * -(-warmup // k) + steps
            assert k * -(-warmup // k) >= warmup
    assert bench.steps_per_graph(64) == 8 and bench.steps_per_graph(7) == 7 and bench.steps_per_graph(11) == 1


def test_reference_arm_prints_one_json_line_on_the_cpu():
    # the reference arm is the oracle on the host cores: one JSON line with
    # the contract's keys, its e2e equal to its value (no device copies)
    import json
    import subprocess
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny",
                          "--steps", "2", "--warmup", "3"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    rec = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
                "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in rec, key
    assert rec["impl"] == "reference" and rec["value"] > 0 and rec["higher_is_better"] is True
    assert rec["cpu_baseline"]["kind"] == "oracle" and rec["cpu_baseline"]["cores"] >= 1
    assert rec["e2e"]["value"] == rec["value"] and rec["e2e"]["h2d_bytes_per_step"] == 0
    assert rec["config"]["workload"].startswith("tiny")
