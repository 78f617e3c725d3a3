"""Near-tie margins reported by the device with every choice (Eq. 3): the
token gap (the chosen score minus the best score at any other token, over
all experts) and the expert gap (minus the best other expert's score at the
chosen token), against the oracle's brute-force gaps on the same inputs, for
the max rule of Eq. 3 and for the MoE / PoE aggregation variants (whose
expert gap is the attribution's margin in log(w p)).  Each step is
teacher-forced with the oracle's token."""
import numpy as np
import pytest
import torch

import synth
from oracle.run import OracleRun
from test_gpu_step import host_ram_gb

pytestmark = pytest.mark.gpu

# The device's gaps against the oracle's Eq. 2 / Eq. 3 (or MoE / PoE) on the
# device's own hidden states: fp32 against fp64 arithmetic only.
GAP_TOL = 1e-4
# Against the full oracle run: its hidden state rounds to bf16 differently
# in about 1 % of the elements (one ulp, ~4e-3 at unit scale), which moves a
# single logit by ~sqrt(40) * 4e-3 * 0.02 ~ 5e-4 at d = 4096; a gap, the
# difference of two scores, within 2e-3.
GAP_TOL_E2E = 2e-3


@pytest.mark.parametrize("name,steps,kw,ram", [("tiny", 4, {}, 0), ("llama8", 3, {}, 8),
                                               ("tiny", 4, {"aggregation": 1}, 0),
                                               ("tiny", 4, {"aggregation": 2}, 0),
                                               ("llama8", 2, {"aggregation": 1}, 8),
                                               ("tiny", 3, {"score_mode": 1}, 0)])
def test_device_gaps_match_the_oracle(cuda_ok, name, steps, kw, ram):
    import oracle
    import paper_2601_08670_gb300 as pced
    from gpu_util import bf16_bits
    if host_ram_gb() < ram:
        pytest.skip(f"needs {ram} GB of free host memory for the oracle's caches")
    w = synth.get(name)
    t = synth.device_inputs(w, "cuda")
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True, **kw)
    run = OracleRun(w, **kw)
    beta, r = synth.betas(w), synth.retrieval_scores(w)
    worst = worst_e2e = 0.0
    for s in range(steps):
        dec.step()
        torch.cuda.synchronize()
        ref = run.step()
        got = dec.gap_trace[:, s].cpu().numpy().astype(np.float64)
        # the oracle's selection on the device's hidden states
        lp, lse = oracle.lm_head_logprobs(bf16_bits(dec.hidden), run.w_bits)
        if kw.get("aggregation"):
            own = oracle.aggregate_select(lp, beta, r, kw["aggregation"])
        else:
            if kw.get("score_mode") == 1:
                lp = lp + lse[:, None]
            own = oracle.contrastive_select(lp, beta, r, w.gamma, w.B, w.N)
        for b in range(w.B):
            for col, key in ((0, "token_gap"), (1, "expert_gap")):
                want = float(own[key][b])
                assert np.isfinite(want) and want >= 0.0
                err = abs(got[b, col] - want)
                worst = max(worst, err)
                assert err <= GAP_TOL, f"step {s} query {b}: {key} {got[b, col]:.6f} vs oracle {want:.6f}"
                e2e = abs(got[b, col] - float(ref[key][b]))
                worst_e2e = max(worst_e2e, e2e)
                assert e2e <= GAP_TOL_E2E, f"step {s} query {b}: {key} {got[b, col]:.6f} vs oracle run {ref[key][b]:.6f}"
            dec.history[b, s] = int(ref["token"][b])
    assert dec.status() == 0
    print(f"{name} {kw}: worst gap difference {worst:.2e} (own hidden state), {worst_e2e:.2e} (oracle run)")


def test_single_expert_has_no_expert_gap(cuda_ok):
    import paper_2601_08670_gb300 as pced
    w = synth.get("tiny", N=1)
    t = synth.device_inputs(w, "cuda")
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos)
    dec.step()
    torch.cuda.synchronize()
    g = dec.gap_trace[:, 0].cpu().numpy()
    assert np.isinf(g[0, 1]) and np.isfinite(g[0, 0])
