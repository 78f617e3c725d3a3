"""pced_adacad_beta (the dynamic contrast strength of the first generated
token, Sec. 3 after Eq. 2) against the fp64 oracle, and the decode step with
dynamic beta against the oracle run with dynamic beta."""
import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

BETA_TOL = 2e-5  # fp32 terms summed in fp64 on the GPU vs fp64 throughout


def _logprob_rows(rng, rows, V, spread):
    z = rng.normal(0.0, spread, size=(rows, V))
    z -= z.max(axis=1, keepdims=True)
    return z - np.log(np.exp(z).sum(axis=1, keepdims=True))


def _gpu_beta(lp, B, N):
    import paper_2601_08670_gb300 as pced
    t = torch.from_numpy(np.ascontiguousarray(lp, np.float32)).cuda()
    beta = pced.adacad_beta(t, B, N)
    torch.cuda.synchronize()
    return beta.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("B,N,V,spread", [(1, 2, 1, 1.0), (1, 3, 255, 0.5), (2, 4, 8192, 1.3), (3, 5, 128256, 1.3),
                                          (1, 16, 151936, 3.0)])
def test_adacad_beta_matches_oracle(cuda_ok, B, N, V, spread):
    rng = np.random.default_rng(B * 1000 + N * 10 + V % 97)
    lp = _logprob_rows(rng, B * (N + 1), V, spread)
    lp32 = lp.astype(np.float32).astype(np.float64)  # both sides read the same fp32 log-probs
    want = oracle.adacad_beta(lp32, B, N)
    got = _gpu_beta(lp32, B, N)
    assert np.all(np.isfinite(got))
    assert np.max(np.abs(got - want)) <= BETA_TOL, f"max err {np.max(np.abs(got - want)):.2e}"


def test_adacad_beta_degenerate_rows(cuda_ok):
    V = 1000
    rng = np.random.default_rng(5)
    p = _logprob_rows(rng, 1, V, 1.0)[0]
    one_a = np.full(V, -np.inf)
    one_a[3] = 0.0
    one_b = np.full(V, -np.inf)
    one_b[999] = 0.0
    # query 0: expert equal to the amateur (0 bits); query 1: disjoint one-hot
    # supports (1 bit); query 2: the same one-hot on both sides (0 bits)
    lp = np.stack([p, p, one_a, one_b, one_b, one_b]).astype(np.float32)
    got = _gpu_beta(lp, 3, 1)
    assert abs(got[0, 0]) <= 1e-6
    assert abs(got[1, 0] - 1.0) <= 1e-6
    assert abs(got[2, 0]) <= 1e-6


@pytest.mark.parametrize("name,steps,ram", [("tiny", 4, 0), ("llama8", 2, 8)])
def test_step_with_dynamic_beta(cuda_ok, name, steps, ram):
    from test_gpu_step import check_stats, compare_step, host_ram_gb, new_stats
    import paper_2601_08670_gb300 as pced
    if host_ram_gb() < ram:
        pytest.skip(f"needs {ram} GB of free host memory for the oracle's caches")
    w = synth.get(name)
    dev = torch.device("cuda")
    t = synth.device_inputs(w, dev)
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True,
                                   dynamic_beta=True)
    from oracle.run import OracleRun
    run = OracleRun(w, dynamic_beta=True)
    stats = new_stats()
    for s in range(steps):
        dec.step()
        torch.cuda.synchronize()
        ref = run.step()
        if s == 0:
            got = dec.beta.cpu().numpy().astype(np.float64)
            assert np.max(np.abs(got - run.beta.astype(np.float64))) <= 1e-4
            # the frozen beta is what the later steps read
            assert not np.allclose(got, synth.betas(w))
        compare_step(dec, ref, run, s, stats)
    assert dec.status() == 0
    check_stats(stats, name)
