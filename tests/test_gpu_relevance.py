"""pced_relevance against the oracle: the retriever / reranker score maps and
the harmonic-mean fusion (Sec. 3; appendix on normalising the scores), on
random scores and on the maps' edge values."""
import math

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _check(got, want):
    want32 = want.astype(np.float32)
    ulp = np.spacing(np.abs(want32)).astype(np.float64)
    diff = np.abs(got.astype(np.float64) - want32.astype(np.float64))
    assert np.all(diff <= ulp), f"max diff {diff.max()}"
    assert np.mean(got == want32) >= 0.99


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("with_reranker", [False, True])
def test_relevance_matches_oracle(cuda_ok, mode, with_reranker):
    import paper_2601_08670_gb300 as pced
    rng = np.random.default_rng(7 + mode)
    n = 1000
    s = (rng.uniform(-1.2, 1.2, n) if mode == 0 else rng.exponential(3.0, n) - 0.5).astype(np.float32)
    edge = [-1.0, 1.0, 0.0, -5.0, 5.0, 1e-30, -1e-30, 0.5] if mode == 0 else [0.0, -1.0, 1.0, 1e6, 1e30, 1e-30, 0.25, 3.0]
    s[:len(edge)] = np.array(edge, np.float32)
    z = (rng.normal(size=n) * 4).astype(np.float32)
    z[:8] = np.array([0.0, -50.0, 50.0, 1e4, -1e4, 1e-30, math.log(3.0), -0.5], np.float32)
    zd = torch.from_numpy(z).cuda() if with_reranker else None
    r = pced.relevance(torch.from_numpy(s).cuda(), mode, zd).cpu().numpy()
    want = oracle.relevance(s.astype(np.float64), mode, z.astype(np.float64) if with_reranker else None)
    _check(r, want)
    assert np.all((r >= 0) & (r <= 1))


def test_relevance_feeds_the_prior(cuda_ok):
    # relevance scores go straight into the step's r: clip away from 0 inside the step
    import paper_2601_08670_gb300 as pced
    s = torch.tensor([-1.0, 0.0, 1.0], device="cuda")
    r = pced.relevance(s, pced.RET_DENSE)
    assert r.tolist() == [0.0, 0.5, 1.0]  # 1 - 1e-8 is 1.0 in fp32
    empty = torch.empty(0, device="cuda")
    assert pced.relevance(empty).numel() == 0
