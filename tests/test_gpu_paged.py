"""Paged KV caches (PagedAttention-style block tables, the paper's serving
setup): the generator's paged pool holds the same logical cache, the decode
step over it matches the oracle and the step over slab caches (up to the
summation order), and a block id outside the pool is flagged, not followed."""
import numpy as np
import pytest
import torch

import synth
from gpu_util import bf16_bits

pytestmark = pytest.mark.gpu


def test_paged_pool_holds_the_logical_cache(cuda_ok):
    w = synth.get("tiny")
    t = synth.device_inputs(w, "cuda", paged=64)
    lay = t["paged_layout"]
    bl = synth.base_lengths(w)
    ref_lay = synth.cache_layout(w, bl)
    kc, vc = synth.host_caches(w, ref_lay, bl, np.arange(w.S, dtype=np.int32))
    pool_k = bf16_bits(t["k_cache"]).reshape(w.L, lay.num_blocks, w.Hkv, lay.P, w.D)
    pool_v = bf16_bits(t["v_cache"]).reshape(w.L, lay.num_blocks, w.Hkv, lay.P, w.D)
    for l in range(w.L):
        for s in range(w.S):
            for h in range(w.Hkv):
                base = l * ref_lay.layer_elems + ref_lay.kv_offset[s] + h * ref_lay.cap[s] * w.D
                for pos in range(bl[s]):
                    blk = lay.table[s, pos // lay.P]
                    want_k = kc[base + pos * w.D: base + (pos + 1) * w.D]
                    want_v = vc[base + pos * w.D: base + (pos + 1) * w.D]
                    assert np.array_equal(pool_k[l, blk, h, pos % lay.P], want_k)
                    assert np.array_equal(pool_v[l, blk, h, pos % lay.P], want_v)


@pytest.mark.parametrize("name,P,steps,queries,ram,over", [
    ("tiny", 64, 4, None, 0, {}), ("tiny", 192, 3, None, 0, {}),
    # seven query heads per kv head at D = 128 (the Qwen grouping) in 128-row blocks
    ("tiny", 128, 3, None, 0, dict(Hq=14, Hkv=2, D=128)),
    ("llama8", 256, 2, None, 8, {}), ("manydoc", 64, 1, [0, 15], 8, {}),
    # Qwen2-7B shapes (28 layers, G = 7, 4096 + 32 keys) over 64-row blocks
    ("qwen_flat", 64, 1, None, 8, {})])
def test_paged_step_matches_oracle(cuda_ok, name, P, steps, queries, ram, over):
    import paper_2601_08670_gb300 as pced
    from oracle.run import OracleRun
    from test_gpu_step import check_stats, compare_step, host_ram_gb, new_stats
    if host_ram_gb() < ram:
        pytest.skip(f"needs {ram} GB of free host memory for the oracle's caches")
    w = synth.get(name, **over)
    t = synth.device_inputs(w, "cuda", paged=P)
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True)
    run = OracleRun(w, queries=queries)
    stats = new_stats()
    for s in range(steps):
        dec.step()
        torch.cuda.synchronize()
        compare_step(dec, run.step(), run, s, stats)
    assert dec.status() == 0
    check_stats(stats, f"{name} paged {P}")


def test_paged_agrees_with_slab(cuda_ok):
    # same logical caches; the paged partition rounds extents and CTA
    # boundaries to 64-key tiles, so the pieces and the summation order (not
    # the result) differ
    import paper_2601_08670_gb300 as pced
    w = synth.get("llama8")
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    outs = []
    for P in (0, 128):
        t = synth.device_inputs(w, "cuda", paged=P)
        dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True)
        rec = []
        for _ in range(3):
            dec.step()
            torch.cuda.synchronize()
            rec.append((bf16_bits(dec.hidden).copy(), dec.lse.cpu().numpy().copy()))
        assert dec.status() == 0
        outs.append((rec, dec.history[:, :3].cpu().numpy().copy(), dec.expert_trace[:, :3].cpu().numpy().copy()))
        del dec, t
        torch.cuda.empty_cache()
    (ra, ha, ea), (rb, hb, eb) = outs
    assert np.array_equal(ha, hb) and np.array_equal(ea, eb)
    for (h1, l1), (h2, l2) in zip(ra, rb):
        assert np.max(np.abs(l1.astype(np.float64) - l2)) <= 1e-3
        assert np.mean(h1 == h2) >= 0.98


def test_paged_bad_block_is_flagged(cuda_ok):
    # a table entry outside the pool: its keys read as zeros, the appended row
    # is not stored and PCED_DEV_BAD_BLOCK is set
    import paper_2601_08670_gb300 as pced
    w = synth.get("tiny")
    t = synth.device_inputs(w, "cuda", paged=64)
    lay = t["paged_layout"]
    s_bad = 1
    blk = int(lay.table[s_bad, 0])
    table = t["block_table"]
    table[s_bad, 0] = lay.num_blocks  # one past the pool
    k_before = t["k_cache"].clone()
    dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
    dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos)
    dec.step()
    torch.cuda.synchronize()
    assert dec.status() & pced.PCED_DEV_BAD_BLOCK
    # the block the entry used to name was not written (its row was not appended)
    per_layer = lay.layer_elems
    blk_elems = w.Hkv * lay.P * w.D
    for l in range(w.L):
        lo = l * per_layer + blk * blk_elems
        assert torch.equal(t["k_cache"][lo:lo + blk_elems], k_before[lo:lo + blk_elems])
