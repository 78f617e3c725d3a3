"""pced_lm_head_logprobs (tcgen05 GEMM + log-softmax) against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import to_dev_bf16

pytestmark = pytest.mark.gpu

# Log-prob tolerance: 1e-2 absolute (bf16 inputs, fp32
# accumulation).  Products of bf16 operands are exact in fp32 and the sums run
# over d <= 4096 terms, so the observed error is ~1e-5.
ABS_TOL = 1e-2


def run_case(S, d, V, seed=3, wscale=0.02):
    import paper_2601_08670_gb300 as pced
    h = synth.host_normal_bf16(S * d, seed).reshape(S, d)
    w = synth.host_normal_bf16(V * d, seed + 1, wscale).reshape(V, d)
    lp_ref, lse_ref = oracle.lm_head_logprobs(h, w)
    lp, lse = pced.lm_head_logprobs(to_dev_bf16(h), to_dev_bf16(w))
    lp = lp.cpu().numpy().astype(np.float64)
    lse = lse.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(lp))
    err = np.abs(lp - lp_ref).max()
    assert err <= ABS_TOL, f"max abs err {err:.3e}"
    assert np.abs(lse - lse_ref).max() <= ABS_TOL
    return err


def test_tiny_shapes(cuda_ok):
    assert run_case(3, 512, 8192) < 1e-4


def test_ragged_vocab_tail(cuda_ok):
    assert run_case(9, 4096, 4096 + 77) < 1e-4


def test_s33_d1024(cuda_ok):
    assert run_case(33, 1024, 2000) < 1e-4


def test_single_row(cuda_ok):
    assert run_case(1, 64, 128) < 1e-4


def test_two_mma_chunks_s272(cuda_ok):
    assert run_case(272, 256, 1000) < 1e-4


def test_larger_logits_scale(cuda_ok):
    # logits with std ~ 6: exercises the max-subtracted sums
    assert run_case(17, 1024, 3000, wscale=0.2) < 1e-3


@pytest.mark.parametrize("S", [272, 300, 340, 512])
def test_many_tiles_per_cta_with_two_n_chunks(cuda_ok, S):
    # more than 256 hidden rows: two N chunks in one TMEM accumulator, several
    # vocabulary tiles per CTA (the accumulator is reused), ragged tail; 512
    # rows is the maximum (two 256-column chunks in all 512 TMEM columns)
    assert run_case(S, 256, 48000 + 77) < 1e-4
