"""Checkpoint and resume of a decode by replaying its history.

The decode state of PCED is (KV caches, sequence lengths, history, beta): the
caches hold the prefill rows, which the caller can regenerate from the same
inputs, plus one appended K/V row per generated token and layer, which is a
function of the history alone (Sec. 3: every expert appends the shared token
y_t).  A checkpoint therefore stores only the small host-side state -- the
step counter, the generated tokens with their experts and scores, beta, r and
the lengths -- and `resume` rebuilds the rest by running the saved number of
pced_step calls on a fresh decoder over the regenerated caches, each forced
to the saved token before the next step reads it.  The step is deterministic
(fixed reduction orders), so on the same GPU type the replay chooses the same
tokens anyway; forcing makes the resumed history exact everywhere.  Host
logic only: every replayed step runs in the library's kernels.
"""
from __future__ import annotations

import json

import numpy as np
import torch

FORMAT = "pced-checkpoint-1"


def state(dec) -> dict:
    """Host copy of a decoder's state after its last completed step."""
    if dec.history.is_cuda:
        torch.cuda.synchronize(dec.history.device)
    t = int(dec.step_t.item())
    return {"format": FORMAT, "step": t, "B": dec.dm.B, "N": dec.dm.N,
            "history": dec.history[:, :t].cpu().numpy().copy(),
            "expert_trace": dec.expert_trace[:, :t].cpu().numpy().copy(),
            "score_trace": dec.score_trace[:, :t].cpu().numpy().copy(),
            "beta": dec.beta.cpu().numpy().copy(), "r": dec.r.cpu().numpy().copy(),
            "seq_len": dec.seq_len.cpu().numpy().copy(),
            "beta_pending": bool(dec.args.beta_from_step)}


def save(dec, path: str, meta: dict | None = None) -> dict:
    """Writes state(dec) and the caller's `meta` (what regenerates the
    caches: workload, seed, options) to `path` (.npz)."""
    st = state(dec)
    arrays = {k: v for k, v in st.items() if isinstance(v, np.ndarray)}
    head = {k: v for k, v in st.items() if not isinstance(v, np.ndarray)}
    head["meta"] = meta or {}
    np.savez(path, header=np.frombuffer(json.dumps(head).encode(), dtype=np.uint8), **arrays)
    return st


def load(path: str) -> dict:
    """Reads a checkpoint written by save(); returns its state and `meta`."""
    with np.load(path) as z:
        head = json.loads(bytes(z["header"]).decode())
        if head.get("format") != FORMAT:
            raise ValueError(f"{path}: not a {FORMAT} file")
        st = dict(head)
        for k in z.files:
            if k != "header":
                st[k] = z[k]
    t, B = st["step"], st["B"]
    for k in ("history", "expert_trace", "score_trace"):
        if st[k].shape != (B, t):
            raise ValueError(f"{path}: {k} has shape {st[k].shape}, expected {(B, t)}")
    return st


def resume(dec, st: dict) -> None:
    """Brings `dec` -- a fresh decoder over the regenerated prefill caches and
    inputs of the checkpointed decode, with its step counter at 0 -- to the
    state `st`: replays st['step'] steps, forcing each step's token, expert
    and score to the saved ones, then checks that the lengths and beta agree.
    Raises ValueError on a mismatch."""
    if (dec.dm.B, dec.dm.N) != (st["B"], st["N"]):
        raise ValueError(f"checkpoint of B={st['B']} N={st['N']}, decoder of B={dec.dm.B} N={dec.dm.N}")
    if int(dec.step_t.item()) != 0:
        raise ValueError("resume needs a fresh decoder (step counter 0)")
    T = st["step"]
    if T > dec.max_steps:
        raise ValueError(f"checkpoint has {T} steps, the decoder holds {dec.max_steps}")
    dev = dec.history.device
    hist = torch.as_tensor(st["history"], dtype=torch.int32).to(dev)
    ex = torch.as_tensor(st["expert_trace"], dtype=torch.int32).to(dev)
    sc = torch.as_tensor(st["score_trace"], dtype=torch.float32).to(dev)
    for s in range(T):
        dec.step()
        # the next step embeds history[:, s]: force the saved choice first
        dec.history[:, s].copy_(hist[:, s])
        dec.expert_trace[:, s].copy_(ex[:, s])
        dec.score_trace[:, s].copy_(sc[:, s])
    if dec.history.is_cuda:
        torch.cuda.synchronize(dev)
    status = dec.status()
    if status:
        raise ValueError(f"replay ended with device status {status:#x}")
    if int(dec.step_t.item()) != T:
        raise ValueError("replay did not reach the saved step")
    if not np.array_equal(dec.seq_len.cpu().numpy(), st["seq_len"]):
        raise ValueError("replayed sequence lengths differ from the checkpoint's")
    if not np.array_equal(dec.beta.cpu().numpy(), st["beta"]):
        raise ValueError("replayed beta differs from the checkpoint's (different inputs or options?)")
    if bool(dec.args.beta_from_step) != bool(st["beta_pending"]):
        raise ValueError("dynamic-beta state differs from the checkpoint's")
