"""Checkpoint / resume host logic on the CPU: the file round trip, its
validation, and the replay's forcing of the saved choices, with a stand-in
decoder whose step() appends a token that depends on the previous one (the
dependency a real step has through the embedding of y_{t-1})."""
import types

import numpy as np
import pytest
import torch

from paper_2601_08670_gb300 import checkpoint


class FakeDecoder:
    """step(): y_t = (7 * y_{t-1} + 3 + bias) mod 101, appended at t; lengths +1;
    with a pending dynamic beta the first step writes beta."""

    def __init__(self, B=2, N=3, max_steps=10, bias=0, dyn=False):
        self.dm = types.SimpleNamespace(B=B, N=N)
        self.max_steps = max_steps
        self.step_t = torch.zeros(1, dtype=torch.int32)
        self.history = torch.zeros((B, max_steps), dtype=torch.int32)
        self.expert_trace = torch.zeros((B, max_steps), dtype=torch.int32)
        self.score_trace = torch.zeros((B, max_steps), dtype=torch.float32)
        self.beta = torch.full((B, N), 0.5)
        self.r = torch.linspace(0.1, 0.9, B * N).reshape(B, N)
        self.seq_len = torch.arange(B * (N + 1), dtype=torch.int32) + 5
        self.args = types.SimpleNamespace(beta_from_step=1 if dyn else 0)
        self.bias = bias

    def step(self):
        t = int(self.step_t.item())
        prev = self.history[:, t - 1] if t > 0 else torch.zeros(self.dm.B, dtype=torch.int32)
        self.history[:, t] = (7 * prev + 3 + self.bias) % 101
        self.expert_trace[:, t] = 1 + t % self.dm.N
        self.score_trace[:, t] = -0.25 * t
        if self.args.beta_from_step:
            self.beta.fill_(0.125)
            self.args.beta_from_step = 0
        self.seq_len += 1
        self.step_t += 1

    def status(self):
        return 0


def test_save_load_round_trip(tmp_path):
    dec = FakeDecoder(dyn=True)
    for _ in range(4):
        dec.step()
    st = checkpoint.save(dec, str(tmp_path / "c.npz"), meta={"workload": "tiny", "seed": 0})
    back = checkpoint.load(str(tmp_path / "c.npz"))
    assert back["meta"] == {"workload": "tiny", "seed": 0}
    assert back["step"] == 4 and back["beta_pending"] is False
    for k in ("history", "expert_trace", "score_trace", "beta", "r", "seq_len"):
        assert np.array_equal(back[k], st[k]), k
        assert back[k].dtype == st[k].dtype


def test_resume_replays_and_forces_the_saved_tokens(tmp_path):
    a = FakeDecoder(dyn=True)
    for _ in range(3):
        a.step()
    checkpoint.save(a, str(tmp_path / "c.npz"))
    st = checkpoint.load(str(tmp_path / "c.npz"))
    # a decoder whose own choices differ (as after a numerics change): the
    # replay still lands on the saved history, and later steps continue from it
    b = FakeDecoder(dyn=True, bias=1)
    checkpoint.resume(b, st)
    assert torch.equal(b.history[:, :3], a.history[:, :3])
    assert torch.equal(b.expert_trace[:, :3], a.expert_trace[:, :3])
    a.step()
    b.bias = 0
    b.step()
    assert torch.equal(b.history[:, :4], a.history[:, :4])
    assert torch.equal(b.seq_len, a.seq_len)


def test_resume_rejects_mismatched_decoders(tmp_path):
    a = FakeDecoder()
    for _ in range(2):
        a.step()
    checkpoint.save(a, str(tmp_path / "c.npz"))
    st = checkpoint.load(str(tmp_path / "c.npz"))
    with pytest.raises(ValueError):
        checkpoint.resume(FakeDecoder(B=3), st)        # other batch
    used = FakeDecoder()
    used.step()
    with pytest.raises(ValueError):
        checkpoint.resume(used, st)                    # not fresh
    other = FakeDecoder()
    other.seq_len -= 1
    with pytest.raises(ValueError):
        checkpoint.resume(other, st)                   # other caches
    with pytest.raises(ValueError):
        checkpoint.resume(FakeDecoder(dyn=True), st)   # other beta mode
    np.savez(str(tmp_path / "bad.npz"), header=np.frombuffer(b'{"format": "x"}', dtype=np.uint8))
    with pytest.raises(ValueError):
        checkpoint.load(str(tmp_path / "bad.npz"))
