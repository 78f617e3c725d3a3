"""The expert-partitioned decode step on one GPU: two decoders, each with
every query's amateur and half of its contextual experts (the contents of
the full workload's sequences), run pced_step with key_out; the packed keys
are reduced with an elementwise max (what an all-reduce-max over GPUs
computes) and pced_step_commit appends the common token on both.  Tokens,
experts and the hidden states of both halves must match the oracle run over
all experts (Eq. 3 couples experts only through the max).  Each step is
teacher-forced with the oracle's token."""
import numpy as np
import pytest
import torch

import synth
from gpu_util import bf16_bits, near_tie
from oracle.run import OracleRun
from test_gpu_step import compare_hidden, host_ram_gb, new_stats

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,steps,ram,dyn", [("tiny", 4, 0, False), ("llama8", 3, 8, False), ("tiny", 3, 0, True)])
def test_two_halves_of_the_experts_choose_like_the_whole(cuda_ok, name, steps, ram, dyn):
    import paper_2601_08670_gb300 as pced
    if host_ram_gb() < ram:
        pytest.skip(f"needs {ram} GB of free host memory for the oracle's caches")
    w = synth.get(name)
    half = w.N // 2
    parts = [(0, half), (half, w.N)]
    decs, ids = [], []
    for e0, e1 in parts:
        t = synth.device_inputs(w, "cuda", part=(e0, e1))
        wp = t["w"]
        dm = pced.dims(wp.B, wp.N, wp.L, wp.Hq, wp.Hkv, wp.D, wp.V)
        decs.append(pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True,
                                             dynamic_beta=dyn))
        ids.append(synth.expert_part(w, e0, e1)[1])
    run = OracleRun(w, dynamic_beta=dyn)
    keys = [torch.zeros(w.B, dtype=torch.int64, device="cuda") for _ in parts]
    stats = new_stats()
    compared = 0
    for s in range(steps):
        for dec, k, (e0, _) in zip(decs, keys, parts):
            dec.step_partial(k, e0)
        red = torch.maximum(keys[0], keys[1])
        for dec in decs:
            dec.commit(red)
        torch.cuda.synchronize()
        ref = run.step()
        for dec, sid in zip(decs, ids):
            tok = dec.history[:, s].cpu().numpy()
            ex = dec.expert_trace[:, s].cpu().numpy()
            for b in range(w.B):
                if not near_tie(ref, b):
                    assert tok[b] == ref["token"][b], f"step {s} query {b}: token {tok[b]} vs {ref['token'][b]}"
                    assert ex[b] == ref["expert"][b], f"step {s} query {b}: expert {ex[b]} vs {ref['expert'][b]}"
                    compared += 1
                dec.history[b, s] = int(ref["token"][b])
            compare_hidden(bf16_bits(dec.hidden), ref["h"][sid], w.Hq, f"step {s}", stats)
    for dec in decs:
        assert dec.status() == 0
        assert int(dec.step_t.item()) == steps
    assert compared > 0
    assert stats["h_bits_diff"] <= 0.02 * stats["h_elems"]
    print(f"{name} dyn={dyn}: {stats}")


def test_partitioned_step_refuses_moe_and_large_expert_indices(cuda_ok):
    import paper_2601_08670_gb300 as pced
    w = synth.get("tiny")
    t = synth.device_inputs(w, "cuda")
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    keys = torch.zeros(w.B, dtype=torch.int64, device="cuda")
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, aggregation=1)
    with pytest.raises(pced.PcedError):
        dec.step_partial(keys, 0)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos)
    with pytest.raises(pced.PcedError):
        dec.step_partial(keys, 4095)
    assert int(dec.step_t.item()) == 0
