"""pced_step_host_io: the decode step with its per-step inputs (beta, r) and
outputs (token, expert, score) in host memory, eagerly and replayed from one
captured CUDA graph per step.

The step's kernels are the same as pced_step's and deterministic, so every
choice, score and hidden state must be bit-identical to a plain pced_step
decode over the same inputs; that decode is checked against the oracle by
the parity tests, and the first choice here is also checked against the
oracle directly."""
from dataclasses import replace

import numpy as np
import pytest
import torch

import synth
from gpu_util import bf16_bits, near_tie
from oracle.run import OracleRun

pytestmark = pytest.mark.gpu


def workload():
    # three queries, so uploads and read-backs carry more than one row
    return replace(synth.get("tiny"), B=3, steps=5, seed=7)


def decoder(w, dev, **kw):
    import paper_2601_08670_gb300 as pced
    t = synth.device_inputs(w, dev)
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    return pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True, **kw)


def host_buffers(w, beta, r):
    pin = lambda x: x.cpu().contiguous().pin_memory()
    return dict(beta=pin(beta), r=pin(r), token=torch.zeros(w.B, dtype=torch.int32).pin_memory(),
                expert=torch.zeros(w.B, dtype=torch.int32).pin_memory(),
                score=torch.zeros(w.B, dtype=torch.float32).pin_memory())


def adjacent_host_buffers(dec, beta, r):
    # r right after beta and the choice as one block, as on the device: the
    # call moves each side in one copy
    br = torch.stack([beta.cpu(), r.cpu()]).pin_memory()
    tok, exp, sc = dec.choice_buffers()
    assert exp.data_ptr() == tok.data_ptr() + 4 * tok.numel() and sc.data_ptr() == exp.data_ptr() + 4 * tok.numel()
    assert dec.r.data_ptr() == dec.beta.data_ptr() + 4 * dec.beta.numel()
    return dict(beta=br[0], r=br[1], token=tok, expert=exp, score=sc)


def per_query_beta(w):
    # a different contrast strength per (query, expert), so a lost upload shows
    return torch.from_numpy(np.random.default_rng(5).uniform(0.1, 0.9, (w.B, w.N)).astype(np.float32))


def expect_same_step(ref, hb, t, dec=None):
    """ref: plain decoder after step t; hb: host outputs of the same step."""
    assert torch.equal(hb["token"], ref.history[:, t].cpu())
    assert torch.equal(hb["expert"], ref.expert_trace[:, t].cpu())
    assert torch.equal(hb["score"].view(torch.int32), ref.score_trace[:, t].cpu().view(torch.int32))
    if dec is not None:
        assert np.array_equal(bf16_bits(dec.hidden), bf16_bits(ref.hidden))
        assert torch.equal(dec.history[:, : t + 1], ref.history[:, : t + 1])


def test_eager_host_io_matches_the_device_step(cuda_ok):
    w = workload()
    dev = torch.device("cuda")
    beta = per_query_beta(w)
    ref = decoder(w, dev)
    ref.beta.copy_(beta)
    dec = decoder(w, dev)
    dec.beta.fill_(float("nan"))  # only the uploads give it values
    hb = host_buffers(w, beta, ref.r)
    for t in range(w.steps):
        ref.step()
        dec.step_host_io(hb["beta"], hb["r"], hb["token"], hb["expert"], hb["score"])
        torch.cuda.synchronize()
        expect_same_step(ref, hb, t, dec)
        assert torch.equal(dec.token_out.cpu(), hb["token"])
    assert ref.status() == 0 and dec.status() == 0
    assert torch.equal(dec.beta.cpu(), beta)


def test_first_choice_matches_the_oracle(cuda_ok):
    w = workload()
    dev = torch.device("cuda")
    dec = decoder(w, dev)
    hb = host_buffers(w, dec.beta, dec.r)
    dec.step_host_io(hb["beta"], hb["r"], hb["token"], hb["expert"], hb["score"])
    torch.cuda.synchronize()
    assert dec.status() == 0
    ref = OracleRun(w).step()
    for b in range(w.B):
        if near_tie(ref, b):
            continue
        assert int(hb["token"][b]) == ref["token"][b]
        assert int(hb["expert"][b]) == ref["expert"][b]


def test_graph_of_one_host_io_step_replays_step_after_step(cuda_ok):
    w = workload()
    dev = torch.device("cuda")
    beta = per_query_beta(w)
    ref = decoder(w, dev)
    ref.beta.copy_(beta)
    dec = decoder(w, dev)
    hb = adjacent_host_buffers(dec, beta, ref.r)
    dec.beta.fill_(float("nan"))
    dec.r.fill_(float("nan"))
    g = dec.capture_host_io(**hb)
    torch.cuda.synchronize()
    assert int(dec.step_t.item()) == 0  # capturing runs nothing
    for t in range(w.steps):
        ref.step()
        hb["token"].fill_(-1)
        g.replay()
        torch.cuda.synchronize()
        expect_same_step(ref, hb, t, dec)
    assert int(dec.step_t.item()) == w.steps
    assert ref.status() == 0 and dec.status() == 0


def test_host_io_with_dynamic_beta_and_moe(cuda_ok):
    import paper_2601_08670_gb300 as pced
    w = workload()
    dev = torch.device("cuda")
    # dynamic beta: the first step computes beta on the device (nothing
    # uploaded), the later steps replay a graph that uploads r only
    ref = decoder(w, dev, dynamic_beta=True)
    dec = decoder(w, dev, dynamic_beta=True)
    hb = host_buffers(w, ref.beta, ref.r)
    ref.step()
    dec.step_host_io(None, hb["r"], hb["token"], hb["expert"], hb["score"])
    torch.cuda.synchronize()
    expect_same_step(ref, hb, 0, dec)
    assert torch.equal(dec.beta, ref.beta)
    g = dec.capture_host_io(None, hb["r"], hb["token"], hb["expert"], hb["score"])
    for t in range(1, w.steps):
        ref.step()
        g.replay()
        torch.cuda.synchronize()
        expect_same_step(ref, hb, t, dec)
    assert ref.status() == 0 and dec.status() == 0
    # MoE: the aggregation kernels write the fixed-address outputs too
    ref = decoder(w, dev, aggregation=pced.AGG_MOE)
    dec = decoder(w, dev, aggregation=pced.AGG_MOE)
    hb = adjacent_host_buffers(dec, ref.beta, ref.r)
    for t in range(2):
        ref.step()
        dec.step_host_io(hb["beta"], hb["r"], hb["token"], hb["expert"], hb["score"])
        torch.cuda.synchronize()
        expect_same_step(ref, hb, t, dec)
    assert ref.status() == 0 and dec.status() == 0


def test_host_io_refuses_device_buffers_as_host_buffers(cuda_ok):
    import paper_2601_08670_gb300 as pced
    w = workload()
    dev = torch.device("cuda")
    dec = decoder(w, dev)
    L = pced.lib()
    import ctypes
    rc = L.pced_step_host_io(ctypes.byref(dec.args), dec.beta.data_ptr(), None, None, None, None,
                             torch.cuda.current_stream().cuda_stream)
    assert rc == 1
    assert b"device memory" in L.pced_last_error()
    torch.cuda.synchronize()
    assert int(dec.step_t.item()) == 0  # nothing was enqueued
