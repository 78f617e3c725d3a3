"""Rotary position embedding in pced_step (the decoders the paper runs are
rotary models): queries and the appended key row rotated by the new token's
position, values not.  Checked against the oracle (which applies the same
rotation in fp64 from fp32 angles) on whole steps, and on the appended rows
themselves."""
import numpy as np
import pytest
import torch

import synth
from gpu_util import bf16_bits, bits_to_f64
from oracle.run import OracleRun
from test_gpu_step import check_stats, compare_step, host_ram_gb, new_stats

pytestmark = pytest.mark.gpu


def _rows(cache, base, D):
    return cache[base:base + D]


@pytest.mark.parametrize("name,theta,steps,paged,ram", [("tiny", 1e4, 4, 0, 0), ("tiny", 5e5, 3, 64, 0),
                                                         ("llama8", 5e5, 2, 0, 8)])
def test_rope_step_matches_oracle(cuda_ok, name, theta, steps, paged, ram):
    import paper_2601_08670_gb300 as pced
    if host_ram_gb() < ram:
        pytest.skip(f"needs {ram} GB of free host memory for the oracle's caches")
    w = synth.get(name)
    t = synth.device_inputs(w, "cuda", paged=paged)
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True,
                                   rope_theta=theta)
    run = OracleRun(w, rope_theta=theta)
    stats = new_stats()
    for s in range(steps):
        pos = run.lens.copy()  # the new token's position in every sequence
        dec.step()
        torch.cuda.synchronize()
        compare_step(dec, run.step(), run, s, stats)
        if name != "tiny":
            continue
        # the appended rows: keys rotated, values not (bf16, fp32 vs fp64 rotation)
        kc = bf16_bits(t["k_cache"])
        vc = bf16_bits(t["v_cache"])
        lay = t["paged_layout"] if paged else t["layout"]
        same = total = 0
        for l in range(w.L):
            for q in range(w.S):
                for h in range(w.Hkv):
                    ref = run.layout.kv_offset[q] + (h * run.layout.cap[q] + pos[q]) * w.D
                    ref += l * run.layout.layer_elems
                    if paged:
                        blk = int(lay.table[q, pos[q] // lay.P])
                        got = l * lay.layer_elems + ((blk * w.Hkv + h) * lay.P + pos[q] % lay.P) * w.D
                    else:
                        got = l * lay.layer_elems + lay.kv_offset[q] + (h * lay.cap[q] + pos[q]) * w.D
                    for cache, oc in ((kc, run.kc), (vc, run.vc)):
                        a, b = _rows(cache, got, w.D), _rows(oc, ref, w.D)
                        diff = np.abs(bits_to_f64(a) - bits_to_f64(b))
                        assert np.all(diff <= np.abs(bits_to_f64(b)) * 2.0 ** -7 + 1e-30)
                        same += int((a == b).sum())
                        total += a.size
        assert same >= 0.98 * total, f"{same}/{total} appended elements bit-equal"
    assert dec.status() == 0
    check_stats(stats, f"{name} rope {theta}")


def test_rope_changes_the_step_and_zero_theta_is_the_plain_step(cuda_ok):
    # theta = 0 leaves the step as it was; a rotary base changes the hidden states
    import paper_2601_08670_gb300 as pced
    w = synth.get("tiny")
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    outs = []
    for theta in (0.0, 1e4):
        t = synth.device_inputs(w, "cuda")
        dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True,
                                       rope_theta=theta)
        dec.step()
        dec.step()
        torch.cuda.synchronize()
        outs.append(bf16_bits(dec.hidden).copy())
    run = OracleRun(w)
    run.step()
    plain = run.step()
    assert np.mean(outs[0] == plain["h"]) >= 0.98
    assert np.mean(outs[1] != outs[0]) > 0.5


def test_rope_theta_is_validated(cuda_ok):
    import paper_2601_08670_gb300 as pced
    w = synth.get("tiny")
    t = synth.device_inputs(w, "cuda")
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    for bad in (-1.0, float("inf"), float("nan")):
        dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, rope_theta=bad)
        with pytest.raises(pced.PcedError):
            dec.step()
