"""Checkpoint / resume on the GPU: a decode checkpointed after k steps and
resumed on a fresh decoder over regenerated caches (replaying the saved
history) continues exactly like the uninterrupted decode: the same tokens,
experts and scores, bit-identical hidden states and lengths."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


def _decoder(w, dyn, steps):
    import paper_2601_08670_gb300 as pced
    t = synth.device_inputs(w, "cuda", extra_steps=steps)
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    return pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=steps, bos=w.bos, keep_hidden=True,
                                    dynamic_beta=dyn), t


@pytest.mark.parametrize("name,over,k,total,dyn", [("tiny", {}, 3, 6, False), ("tiny", {}, 2, 5, True),
                                                     ("llama8", {"L": 4}, 2, 4, False)])
def test_resumed_decode_continues_like_the_uninterrupted_one(cuda_ok, tmp_path, name, over, k, total, dyn):
    from paper_2601_08670_gb300 import checkpoint
    w = synth.get(name, **over)
    ref, tr = _decoder(w, dyn, total)
    for _ in range(total):
        ref.step()
    torch.cuda.synchronize()
    ref_h = ref.hidden.clone()

    a, ta = _decoder(w, dyn, total)
    for _ in range(k):
        a.step()
    path = str(tmp_path / "ckpt.npz")
    checkpoint.save(a, path, meta={"workload": name, "overrides": over, "dynamic_beta": dyn})
    del a, ta
    torch.cuda.empty_cache()

    st = checkpoint.load(path)
    b, tb = _decoder(w, dyn, total)  # caches regenerated from the same seed and configuration
    checkpoint.resume(b, st)
    for _ in range(total - k):
        b.step()
    torch.cuda.synchronize()
    assert b.status() == 0 and ref.status() == 0
    assert torch.equal(b.history[:, :total], ref.history[:, :total])
    assert torch.equal(b.expert_trace[:, :total], ref.expert_trace[:, :total])
    assert torch.equal(b.score_trace[:, :total], ref.score_trace[:, :total])
    assert torch.equal(b.seq_len, ref.seq_len)
    assert torch.equal(b.beta, ref.beta)
    assert torch.equal(b.hidden.view(torch.int16), ref_h.view(torch.int16))
