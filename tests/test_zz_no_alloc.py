"""pced_decode_attention_noalloc, the attention entry point for callers that
cannot allocate device memory when they call it (a locked or shutting-down
allocator, host callbacks, a capped memory pool owned by someone else).

It keeps its partial records in one fixed device array inside the library, so
the checks here are (1) its output matches pced_decode_attention's on the
same inputs, for two different calls in a row (the second one runs over the
scratch the first one left behind), (2) it matches the fp64 oracle's
brute-force attention directly, so a fault of the shared array that hit both
entry points alike would still show, (3) a length beyond its capacity comes
back as a bit of the caller's status word, and (4) shapes whose scratch would
exceed the fixed maximum are refused before anything is launched.

The file name sorts last so that a run stopping at the first failure has
already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import to_dev_bf16

# same bound as the attention parity tests: 2e-2 of each (sequence, head)
# row's largest magnitude
REL_TOL = 2e-2


def make_case(lens, Hq, Hkv, D, seed, extra=5):
    from dataclasses import replace
    S = len(lens)
    lens = np.asarray(lens, np.int32)
    w = replace(synth.get("tiny"), L=1, Hq=Hq, Hkv=Hkv, D=D, seed=seed)
    lay = synth.cache_layout(w, lens, extra)
    kc, vc = synth.host_caches(w, lay, lens, np.arange(S, dtype=np.int32))
    q = synth.host_normal_bf16(S * Hq * D, seed + 1).reshape(S, Hq, D)
    dev = torch.device("cuda")
    return dict(q=to_dev_bf16(q), k=to_dev_bf16(kc), v=to_dev_bf16(vc),
                off=torch.from_numpy(lay.kv_offset).to(dev), cap=torch.from_numpy(lay.cap).to(dev),
                lens=torch.from_numpy(lens).to(dev), Hkv=Hkv, total_cap=int(lay.cap.sum()),
                host=(q, kc, vc, lay.kv_offset, lay.cap, lens, Hq, Hkv, D))


def within_tol(got, ref):
    err = np.abs(got - ref).max(axis=2)
    mag = np.abs(ref).max(axis=2)
    assert np.all(np.isfinite(got))
    assert np.all(err <= REL_TOL * mag), f"max rel err {np.max(err / mag):.3e}"


def compare(c):
    import paper_2601_08670_gb300 as pced
    want = pced.decode_attention(c["q"], c["k"], c["v"], c["off"], c["cap"], c["lens"], c["Hkv"], c["total_cap"])
    out = torch.full_like(want, float("nan"))
    status = torch.zeros(1, dtype=torch.int32, device=want.device)
    pced.decode_attention_noalloc(c["q"], c["k"], c["v"], c["off"], c["cap"], c["lens"], c["Hkv"], c["total_cap"],
                                  out, status=status)
    torch.cuda.synchronize()
    got, ref = out.cpu().numpy().astype(np.float64), want.cpu().numpy().astype(np.float64)
    assert int(status.item()) == 0
    within_tol(got, ref)
    return got


@pytest.mark.gpu
def test_noalloc_matches_workspace_entry_point_on_two_calls(cuda_ok):
    # first call: D=128, GQA 4, ragged lengths spanning several CTAs and tails
    compare(make_case([1, 63, 64, 65, 700, 2081, 130, 33], Hq=32, Hkv=8, D=128, seed=21))
    # second call, different shape over the scratch left by the first one:
    # D=64, more sequences, different grouping
    compare(make_case(list(np.random.default_rng(3).integers(1, 300, size=40)), Hq=16, Hkv=2, D=64, seed=22))


@pytest.mark.gpu
def test_noalloc_matches_the_oracle(cuda_ok):
    # the tiny workload's attention shape (8 q / 2 kv heads, D = 64, two
    # documents of 256 keys and an amateur of 32), then a ragged D = 128 case
    for lens, Hq, Hkv, D, seed in (([32, 256, 256], 8, 2, 64, 31), ([1, 65, 2081, 130], 32, 8, 128, 32)):
        c = make_case(lens, Hq=Hq, Hkv=Hkv, D=D, seed=seed)
        got = compare(c)
        q, kc, vc, off, cap, ln, Hq_, Hkv_, D_ = c["host"]
        within_tol(got, oracle.attention(q, kc, vc, off, cap, ln, Hq_, Hkv_, D_))


@pytest.mark.gpu
def test_noalloc_reports_bad_lengths_through_the_status_word(cuda_ok):
    import paper_2601_08670_gb300 as pced
    dev = torch.device("cuda")
    S, Hq, Hkv, D = 2, 4, 1, 64
    cap = torch.tensor([8, 8], dtype=torch.int32, device=dev)
    off = torch.tensor([0, 8 * D], dtype=torch.int64, device=dev)
    lens = torch.tensor([9, 3], dtype=torch.int32, device=dev)  # the first is beyond its capacity
    k = torch.zeros(2 * 8 * D, dtype=torch.bfloat16, device=dev)
    q = torch.zeros((S, Hq, D), dtype=torch.bfloat16, device=dev)
    out = torch.full((S, Hq, D), float("nan"), dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    pced.decode_attention_noalloc(q, k, k, off, cap, lens, Hkv, 16, out, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & pced.PCED_DEV_BAD_LENGTH
    assert torch.isfinite(out).all()


@pytest.mark.gpu
def test_noalloc_refuses_shapes_beyond_its_scratch(cuda_ok):
    import paper_2601_08670_gb300 as pced
    L = pced.lib()
    S, Hq, Hkv, D = 1024, 64, 8, 128  # 8192 segments x 8 heads x 128 fp32 ~ 33.6 MB of records
    assert S * Hkv * (Hq // Hkv) * D * 4 > pced.NOALLOC_SCRATCH_BYTES
    dev = torch.device("cuda")
    # valid, fully sized buffers (every sequence: one live row of a 1-row slab
    # at offset 0), so that the refusal is the only thing under test
    q = torch.zeros((S, Hq, D), dtype=torch.bfloat16, device=dev)
    kv = torch.zeros(Hkv * D, dtype=torch.bfloat16, device=dev)
    idx = torch.zeros(S, dtype=torch.int64, device=dev)
    i32 = torch.ones(S, dtype=torch.int32, device=dev)
    out = torch.zeros((S, Hq, D), dtype=torch.float32, device=dev)
    rc = L.pced_decode_attention_noalloc(q.data_ptr(), kv.data_ptr(), kv.data_ptr(), kv.numel(),
                                         idx.data_ptr(), i32.data_ptr(), i32.data_ptr(), S, Hq, Hkv, D, S,
                                         ctypes.c_float(0.1), out.data_ptr(), None, None)
    assert rc == 3
    assert b"above the fixed maximum" in L.pced_last_error()


def test_noalloc_rejects_null_arguments_on_the_host():
    # host validation only: no device is touched
    from paper_2601_08670_gb300 import build
    build.build()
    import paper_2601_08670_gb300 as pced
    L = pced.lib()
    fake = 1 << 12
    assert L.pced_decode_attention_noalloc(None, fake, fake, 1 << 20, fake, fake, fake, 2, 8, 2, 64, 100,
                                           ctypes.c_float(0.1), fake, None, None) == 1
    assert L.pced_decode_attention_noalloc(fake, fake, fake, 1 << 20, fake, fake, fake, 2, 8, 2, 96, 100,
                                           ctypes.c_float(0.1), fake, None, None) == 3
