"""Seeded input generator: determinism, distribution, subset consistency.  No GPU."""
import numpy as np

import oracle
import synth
from oracle.run import OracleRun


def test_generator_is_deterministic_and_normal_like():
    w = synth.get("tiny")
    a = synth.host_matrix(w, synth.T_EMBED, 0, 64)
    b = synth.host_matrix(w, synth.T_EMBED, 0, 64)
    assert np.array_equal(a, b)
    x = oracle.bf16_to_f64(a)
    assert abs(x.mean()) < 0.02 and abs(x.std() - 1.0) < 0.02
    assert np.abs(x).max() <= 3.47
    u = oracle.bf16_to_f64(synth.host_matrix(w, synth.T_UNEMBED, 0, 64))
    assert abs(u.std() - 0.02) < 0.001


def test_matrix_row_ranges_are_slices_of_the_full_matrix():
    w = synth.get("tiny", V=300)
    full = synth.host_matrix(w, synth.T_UNEMBED)
    part = synth.host_matrix(w, synth.T_UNEMBED, 123, 7)
    assert np.array_equal(full[123:130], part)


def test_cache_subset_generation_matches_full_layout():
    w = synth.get("manydoc", B=3, N=2, L=2, Hq=4, Hkv=2, D=8, V=64)
    bl = synth.base_lengths(w)
    lay = synth.cache_layout(w, bl)
    kc, vc = synth.host_caches(w, lay, bl)
    ids = np.array([3, 4, 5], np.int32)  # query 1
    sub = synth.cache_layout(synth.get("manydoc", B=1, N=2, L=2, Hq=4, Hkv=2, D=8, V=64), bl[ids])
    kc1, vc1 = synth.host_caches(w, sub, bl[ids], ids)
    for l in range(w.L):
        for j, s in enumerate(ids):
            for h in range(w.Hkv):
                a = l * lay.layer_elems + lay.kv_offset[s] + h * lay.cap[s] * w.D
                b = l * sub.layer_elems + sub.kv_offset[j] + h * sub.cap[j] * w.D
                n = bl[s] * w.D
                assert np.array_equal(kc[a:a + n], kc1[b:b + n]) and np.array_equal(vc[a:a + n], vc1[b:b + n])


def test_workload_recipes():
    for name in synth.WORKLOADS:
        w = synth.get(name)
        bl = synth.base_lengths(w)
        assert len(bl) == w.S and np.all(bl[:: w.N + 1] == w.amateur_len)
        r = synth.retrieval_scores(w)
        assert r.shape == (w.B, w.N) and np.all(r > 0) and np.all(r <= 1)
    w = synth.get("llama32")
    docs = np.delete(synth.base_lengths(w), np.arange(0, w.S, w.N + 1)) - 32
    assert docs.min() >= 512 and docs.max() <= 8192
    assert abs(synth.retrieval_scores(w).sum() - 1.0) < 1e-5
    w = synth.get("manydoc")
    docs = np.delete(synth.base_lengths(w), np.arange(0, w.S, w.N + 1)) - 32
    assert docs.min() >= 256 and docs.max() <= 2048


def test_oracle_queries_are_independent():
    # running a subset of queries gives the same result as the full batch:
    # experts of different queries never interact (each query is its own Eq. 3)
    w = synth.get("manydoc", B=3, N=2, L=2, Hq=4, Hkv=2, D=16, V=256, steps=2)
    full = OracleRun(w)
    one = OracleRun(w, queries=[2])
    for _ in range(2):
        a = full.step()
        b = one.step()
        assert a["token"][2] == b["token"][0] and a["expert"][2] == b["expert"][0]
        assert np.array_equal(a["h"][6:9], b["h"])


def test_paged_layout_hands_out_every_block_once():
    # a seeded shuffled pool: every sequence gets ceil(cap / P) distinct blocks,
    # the blocks of all sequences are a permutation of the pool, -1 pads the table
    for name, P in (("tiny", 64), ("llama8", 256), ("manydoc", 64), ("tiny", 192)):
        w = synth.get(name)
        bl = synth.base_lengths(w)
        lay = synth.paged_layout(w, bl, P)
        nblk = (lay.cap.astype(np.int64) + P - 1) // P
        assert lay.num_blocks == int(nblk.sum())
        assert lay.layer_elems == lay.num_blocks * w.Hkv * P * w.D
        used = np.concatenate([lay.table[s, :n] for s, n in enumerate(nblk)])
        assert np.array_equal(np.sort(used), np.arange(lay.num_blocks))
        for s, n in enumerate(nblk):
            assert np.all(lay.table[s, n:] == -1)
        assert np.all(lay.cap <= lay.max_blocks * P)
        # same seed, same pool
        assert np.array_equal(synth.paged_layout(w, bl, P).table, lay.table)
