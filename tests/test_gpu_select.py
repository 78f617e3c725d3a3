"""pced_contrastive_select (Eq. 2 + Eq. 3 on materialised log-probs) against the oracle."""
import numpy as np
import pytest
import torch

import oracle
import synth
from gpu_util import near_tie

pytestmark = pytest.mark.gpu


def run_case(B, N, V, seed, gamma=2.5, beta_val=None):
    import paper_2601_08670_gb300 as pced
    rng = np.random.default_rng(seed)
    z = rng.normal(size=(B * (N + 1), V)) * 1.5
    z -= z.max(axis=1, keepdims=True)
    lp = (z - np.log(np.exp(z).sum(axis=1, keepdims=True))).astype(np.float32)
    beta = (rng.uniform(0, 1, size=(B, N)) if beta_val is None else np.full((B, N), beta_val)).astype(np.float32)
    r = rng.uniform(0, 1, size=(B, N)).astype(np.float32)
    ref = oracle.contrastive_select(lp.astype(np.float64), beta, r, gamma, B, N)
    dev = torch.device("cuda")
    tok, exp, sc = pced.contrastive_select(torch.from_numpy(lp).to(dev), torch.from_numpy(beta).to(dev),
                                           torch.from_numpy(r).to(dev), gamma)
    tok, exp, sc = tok.cpu().numpy(), exp.cpu().numpy(), sc.cpu().numpy()
    for b in range(B):
        if near_tie(ref, b):
            continue
        assert tok[b] == ref["token"][b] and exp[b] == ref["expert"][b], f"query {b}"
        assert abs(sc[b] - ref["score"][b]) < 1e-4


def test_llama_vocab_n8(cuda_ok):
    run_case(1, 8, 128256, 1)


def test_batch16_n16(cuda_ok):
    run_case(16, 16, 8192, 2)


def test_single_expert(cuda_ok):
    run_case(4, 1, 5000, 3)


def test_n32_no_contrast(cuda_ok):
    run_case(2, 32, 3000, 4, beta_val=0.0)


def test_exact_ties_follow_lowest_token_then_expert(cuda_ok):
    import paper_2601_08670_gb300 as pced
    V, N = 10, 3
    lp = np.full((N + 1, V), -5.0, np.float32)
    lp[2, 7] = lp[2, 4] = lp[3, 4] = -0.5  # equal best: tokens 4 and 7 of expert 2, token 4 of expert 3
    beta = np.zeros((1, N), np.float32)
    r = np.full((1, N), 0.5, np.float32)
    dev = torch.device("cuda")
    tok, exp, _ = pced.contrastive_select(torch.from_numpy(lp).to(dev), torch.from_numpy(beta).to(dev),
                                          torch.from_numpy(r).to(dev), 2.5)
    ref = oracle.contrastive_select(lp.astype(np.float64), beta, r, 2.5, 1, N)
    assert int(tok[0]) == ref["token"][0] == 4 and int(exp[0]) == ref["expert"][0] == 2
