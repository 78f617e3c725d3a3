"""The expert-partitioned step on the CPU: Eq. 3 couples a query's experts
only through the maximum over them, so ranks holding disjoint experts (the
amateur replicated) agree on the token through one all-reduce-max of packed
int64 keys.  (1) The key's signed order is Eq. 3's order and unpacks
exactly.  (2) Two gloo ranks, each scoring its half of the experts with the
oracle, reduce their keys and obtain the single-rank oracle's token and
expert."""
import math
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def pced():
    from paper_2601_08670_gb300 import build
    build.build()
    import paper_2601_08670_gb300 as p
    return p


def test_key_order_is_eq3_order_and_round_trips(pced):
    rng = np.random.default_rng(7)
    special = [0.0, -0.0, 1.0, -1.0, math.inf, -math.inf, 3.4e38, -3.4e38, 1e-40, -1e-40]
    scores = np.concatenate([rng.normal(0, 10, 60), np.repeat(rng.normal(0, 1, 5), 8), special]).astype(np.float32)
    cands = [(float(s), int(rng.integers(0, 1 << 20)), int(rng.integers(1, 4097))) for s in scores]
    # ties in score with different tokens / experts, and in token with different experts
    cands += [(2.5, 100, 7), (2.5, 99, 9), (2.5, 100, 3), (2.5, (1 << 20) - 1, 4096), (2.5, 0, 1)]
    keys = [pced.select_key(*c) for c in cands]
    by_key = [c for _, c in sorted(zip(keys, cands), key=lambda kc: kc[0])]
    # Eq. 3: higher score first, then lower token, then lower expert (+0 above -0)
    by_rule = sorted(cands, key=lambda c: (c[0], math.copysign(1.0, c[0]) if c[0] == 0 else 0.0, -c[1], -c[2]))
    assert by_key == by_rule
    for c, k in zip(cands, keys):
        s, t, e = pced.select_key_unpack(k)
        assert (t, e) == (c[1], c[2]) and np.float32(s).tobytes() == np.float32(c[0]).tobytes()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _problem(B=3, N=6, V=64, seed=11):
    rng = np.random.default_rng(seed)
    z = rng.normal(0, 2, size=(B * (N + 1), V))
    lp = z - np.log(np.exp(z).sum(1, keepdims=True))
    beta = rng.uniform(0.2, 1.0, size=(B, N)).astype(np.float32)
    r = rng.uniform(0.05, 1.0, size=(B, N)).astype(np.float32)
    return lp, beta, r, 2.5


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    import oracle
    import paper_2601_08670_gb300 as pced
    dist.init_process_group("gloo", rank=rank, world_size=world)
    lp, beta, r, gamma = _problem()
    B, N = beta.shape
    per = N // world
    e0, e1 = rank * per, (rank + 1) * per
    # this rank's sequences: every query's amateur and its experts [e0, e1)
    rows = [b * (N + 1) + j for b in range(B) for j in [0] + list(range(1 + e0, 1 + e1))]
    sel = oracle.contrastive_select(lp[rows], beta[:, e0:e1], r[:, e0:e1], gamma, B, e1 - e0)
    keys = torch.tensor([pced.select_key(np.float32(sel["score"][b]), int(sel["token"][b]), e0 + int(sel["expert"][b]))
                         for b in range(B)], dtype=torch.int64)
    dist.all_reduce(keys, op=dist.ReduceOp.MAX)
    out = [pced.select_key_unpack(int(k)) for k in keys]
    dist.destroy_process_group()
    q.put((rank, out))


def test_two_ranks_with_half_the_experts_each_choose_like_one(pced):
    import oracle
    lp, beta, r, gamma = _problem()
    B, N = beta.shape
    full = oracle.contrastive_select(lp, beta, r, gamma, B, N)
    # no near tie in this problem, so fp32 keys cannot reorder the candidates
    assert np.all(full["token_gap"] > 1e-4) and np.all(full["expert_gap"] > 1e-4)
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(rk, 2, port, q)) for rk in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rk in range(2):
        for b in range(B):
            s, t, e = res[rk][b]
            assert t == full["token"][b] and e == full["expert"][b]
            assert abs(s - full["score"][b]) <= 1e-5 * max(1.0, abs(full["score"][b]))
