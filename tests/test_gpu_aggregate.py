"""The aggregation variants (MoE / PoE, the appendix's aggregation ablation)
and the raw-logit reading of Eq. 2 in pced_step, against the oracle run with
the same settings: tokens and experts exact except near ties, log-sum-exps
and hidden states as for the plain step, the reported score within 2e-2."""
import numpy as np
import pytest
import torch

import synth
from gpu_util import near_tie
from oracle.run import OracleRun
from test_gpu_step import check_stats, compare_step, host_ram_gb, new_stats

pytestmark = pytest.mark.gpu

SCORE_TOL = 2e-2


def run_variant(name, steps, ram, paged=0, overrides=None, **kw):
    import paper_2601_08670_gb300 as pced
    if host_ram_gb() < ram:
        pytest.skip(f"needs {ram} GB of free host memory for the oracle's caches")
    w = synth.get(name, **(overrides or {}))
    t = synth.device_inputs(w, "cuda", paged=paged)
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True, **kw)
    run = OracleRun(w, **kw)
    stats = new_stats()
    for s in range(steps):
        dec.step()
        torch.cuda.synchronize()
        ref = run.step()
        sc = dec.score_trace[:, s].cpu().numpy()
        for j, b in enumerate(run.queries):
            if not near_tie(ref, j):
                assert abs(sc[b] - ref["score"][j]) <= SCORE_TOL, f"step {s} query {b}: score {sc[b]} vs {ref['score'][j]}"
        compare_step(dec, ref, run, s, stats)
    assert dec.status() == 0
    check_stats(stats, f"{name} {kw}")
    return stats


@pytest.mark.parametrize("rule", [1, 2])
def test_moe_poe_tiny(cuda_ok, rule):
    run_variant("tiny", 4, 0, aggregation=rule)


@pytest.mark.parametrize("rule", [1, 2])
def test_moe_poe_llama8(cuda_ok, rule):
    run_variant("llama8", 2, 8, aggregation=rule)


def test_raw_logit_mode(cuda_ok):
    run_variant("tiny", 4, 0, score_mode=1)
    run_variant("llama8", 2, 8, score_mode=1)


@pytest.mark.parametrize("rule,paged,theta", [(1, 64, 0.0), (2, 128, 5e5), (1, 0, 1e4)])
def test_aggregation_with_paged_caches_and_rotary(cuda_ok, rule, paged, theta):
    # the aggregation kernels after attention over paged caches and / or
    # rotary positions (the options compose: they touch different stages)
    run_variant("tiny", 3, 0, paged=paged, aggregation=rule, rope_theta=theta)
    run_variant("llama8", 2, 2, paged=paged, overrides={"L": 4}, aggregation=rule, rope_theta=theta)


def test_dynamic_beta_with_rotary_and_raw_logits(cuda_ok):
    run_variant("tiny", 3, 0, dynamic_beta=True, rope_theta=1e4)
    run_variant("tiny", 3, 0, score_mode=1, rope_theta=1e4)


def test_moe_with_dynamic_beta_and_graph_replay(cuda_ok):
    # dynamic beta's first step feeds the aggregation; later steps replay from a graph
    import paper_2601_08670_gb300 as pced
    w = synth.get("tiny")
    t = synth.device_inputs(w, "cuda")
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True,
                                   aggregation=1, dynamic_beta=True)
    run = OracleRun(w, aggregation=1, dynamic_beta=True)
    stats = new_stats()
    dec.step()
    torch.cuda.synchronize()
    compare_step(dec, run.step(), run, 0, stats)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        dec.step()
    for i in range(1, 3):
        with torch.cuda.stream(s):
            g.replay()
        torch.cuda.synchronize()
        compare_step(dec, run.step(), run, i, stats)
    assert dec.status() == 0
    check_stats(stats, "tiny moe dynamic beta graph")
