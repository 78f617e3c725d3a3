"""pced_decode_attention against the fp64 oracle on the same seeded inputs."""
import math
from dataclasses import replace

import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import to_dev_bf16

pytestmark = pytest.mark.gpu

# Attention tolerance (bf16 in, fp32 accumulate): 2e-2
# relative.  The kernel keeps QK^T exact in fp32 and P to ~16 bits, so the
# observed error is far below; the bound is applied per (sequence, head) row
# relative to that row's largest magnitude.
REL_TOL = 2e-2


def run_case(lens, Hq, Hkv, D, extra=7, seed=11, scale=None):
    import paper_2601_08670_gb300 as pced
    S = len(lens)
    lens = np.asarray(lens, np.int32)
    w = replace(synth.get("tiny"), L=1, Hq=Hq, Hkv=Hkv, D=D, seed=seed)
    lay = synth.cache_layout(w, lens, extra)
    kc, vc = synth.host_caches(w, lay, lens, np.arange(S, dtype=np.int32))
    q = synth.host_normal_bf16(S * Hq * D, seed + 1).reshape(S, Hq, D)
    ref = oracle.attention(q, kc, vc, lay.kv_offset, lay.cap, lens, Hq, Hkv, D, scale)
    dev = torch.device("cuda")
    out = pced.decode_attention(to_dev_bf16(q), to_dev_bf16(kc), to_dev_bf16(vc),
                                torch.from_numpy(lay.kv_offset).to(dev), torch.from_numpy(lay.cap).to(dev),
                                torch.from_numpy(lens).to(dev), Hkv, int(lay.cap.sum()), scale)
    got = out.cpu().numpy().astype(np.float64)
    err = np.abs(got - ref).max(axis=2)
    mag = np.abs(ref).max(axis=2)
    assert np.all(np.isfinite(got))
    assert np.all(err <= REL_TOL * mag), f"max rel err {np.max(err / mag):.3e}"
    return float(np.max(err / mag))


def test_tiny_geometry(cuda_ok):
    rel = run_case([33, 257, 257], Hq=8, Hkv=2, D=64)
    assert rel < 1e-4


def test_ragged_d128_gqa4(cuda_ok):
    rel = run_case([1, 5, 63, 64, 65, 200, 1000, 2081, 130], Hq=32, Hkv=8, D=128)
    assert rel < 1e-4


def test_gqa7_qwen_heads(cuda_ok):
    rel = run_case([33, 4128, 700, 1, 2049], Hq=28, Hkv=4, D=128)
    assert rel < 1e-4


@pytest.mark.parametrize("Hq,Hkv", [(2, 2), (16, 2)])
def test_gqa_1_and_8(cuda_ok, Hq, Hkv):
    run_case([17, 300, 64], Hq=Hq, Hkv=Hkv, D=64)


def test_many_short_sequences_span_ctas(cuda_ok):
    # more sequences than keys per CTA: CTA ranges cross many segment boundaries
    rng = np.random.default_rng(5)
    run_case(list(rng.integers(1, 40, size=200)), Hq=8, Hkv=2, D=128)


def test_length_equal_to_capacity(cuda_ok):
    run_case([64, 128, 1], Hq=8, Hkv=2, D=128, extra=0)


def test_custom_scale(cuda_ok):
    run_case([100, 7], Hq=4, Hkv=1, D=64, scale=0.3)


def test_bad_length_sets_device_status_without_faulting(cuda_ok):
    import paper_2601_08670_gb300 as pced
    dev = torch.device("cuda")
    S, Hq, Hkv, D = 2, 4, 1, 64
    cap = torch.tensor([8, 8], dtype=torch.int32, device=dev)
    off = torch.tensor([0, 8 * D], dtype=torch.int64, device=dev)
    lens = torch.tensor([9, 0], dtype=torch.int32, device=dev)  # > cap and < 1
    k = torch.zeros(2 * 8 * D, dtype=torch.bfloat16, device=dev)
    q = torch.zeros((S, Hq, D), dtype=torch.bfloat16, device=dev)
    ws = pced.workspace(pced.decode_attention_workspace_size(S, Hq, Hkv, D), dev)
    out = pced.decode_attention(q, k, k, off, cap, lens, Hkv, 16, ws=ws)
    torch.cuda.synchronize()
    assert pced.device_status(ws) & pced.PCED_DEV_BAD_LENGTH
    assert torch.isfinite(out).all()
