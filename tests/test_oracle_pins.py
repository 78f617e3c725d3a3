"""Pins of the CPU oracle against facts fixed by the paper and by mathematics
(closed forms, invariants, special cases reducing to textbook rules, brute
force on tiny inputs).  No GPU."""
import math

import numpy as np
import pytest

import oracle
import synth

rng0 = np.random.default_rng(1234)


def bf16_bits(x):
    """nearest-bf16 bit patterns of fp64 values, through the pinned scalar rounding"""
    x = np.asarray(x, np.float64)
    return np.array([oracle.round_bf16(v) for v in x.ravel()], np.uint16).reshape(x.shape)


# ---------------------------------------------------------------- bf16 / norm
def test_bf16_round_known_values():
    assert oracle.round_bf16(1.0) == 0x3F80
    assert oracle.round_bf16(-2.5) == 0xC020
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: ties go to the even significand (1.0)
    assert oracle.round_bf16(1.0 + 2.0 ** -8) == 0x3F80
    # 1 + 3*2^-8 is halfway between 1 + 2^-7 (odd) and 1 + 2^-6 (even)
    assert oracle.round_bf16(1.0 + 3 * 2.0 ** -8) == 0x3F82
    # just above a tie rounds up
    assert oracle.round_bf16(1.0 + 2.0 ** -8 + 2.0 ** -30) == 0x3F81
    assert oracle.round_bf16(0.0) == 0
    assert oracle.bf16_value(0x3F80) == 1.0
    assert oracle.bf16_value(0xC020) == -2.5


def test_bf16_round_trip_all_finite_patterns():
    for b in range(0, 1 << 16, 7):
        exp = (b >> 7) & 0xFF
        if exp == 0xFF or b == 0x8000:
            continue
        assert oracle.round_bf16(oracle.bf16_value(b)) == b


def test_bf16_rounding_agrees_with_generator_integer_rounding():
    # the generator rounds fp32 -> bf16 with integer arithmetic; the oracle rounds
    # fp64 -> bf16 through frexp.  On fp32 inputs the two must agree.
    lib = synth.host_lib()
    key = lib.synth_key(7, 1, 0, 0, 0)
    for i in range(2000):
        f = lib.synth_value_f32(key, i, synth.normal_scale(1.0))
        assert lib.synth_value_bf16(key, i, synth.normal_scale(1.0)) == oracle.round_bf16(f)


def test_rmsnorm_closed_forms():
    c, eps = 3.0, 1e-6
    y = oracle.rmsnorm(np.full(64, c), eps)
    assert np.allclose(y, c / math.sqrt(c * c + eps), rtol=0, atol=1e-15)
    x = rng0.normal(size=512)
    y = oracle.rmsnorm(x, 0.0)
    assert abs(np.mean(y * y) - 1.0) < 1e-12
    assert np.allclose(y / x, y[0] / x[0])  # a pure rescaling


# ------------------------------------------------------------------ attention
def make_cache(slabs, cap, D):
    """slabs: list over sequences of [Hkv][len][D] float arrays -> (kc-or-vc bits, kv_off)"""
    S = len(slabs)
    Hkv = len(slabs[0])
    off = np.zeros(S, np.int64)
    total = 0
    for s in range(S):
        off[s] = total
        total += Hkv * cap[s] * D
    buf = np.zeros(total, np.uint16)
    for s in range(S):
        for h in range(Hkv):
            rows = np.asarray(slabs[s][h], np.float64)
            n = rows.shape[0]
            base = off[s] + h * cap[s] * D
            buf[base:base + n * D] = bf16_bits(rows).ravel()
    return buf, off


def run_attn(q, K, V, lens, cap, Hq, Hkv, D, scale=None):
    kc, off = make_cache(K, cap, D)
    vc, _ = make_cache(V, cap, D)
    return oracle.attention(bf16_bits(q), kc, vc, off, np.asarray(cap, np.int32), np.asarray(lens, np.int32),
                            Hq, Hkv, D, scale)


def test_attention_single_key_returns_its_value():
    D = 4
    v = np.array([[[0.5, -1.25, 2.0, 3.0]]])
    k = np.array([[[1.0, 2.0, -1.0, 0.5]]])
    q = np.array([[[0.25, 0.5, -0.75, 1.0]]])
    o = run_attn(q, [k], [v], [1], [3], 1, 1, D)
    assert np.array_equal(o[0, 0], v[0, 0])


def test_attention_zero_query_is_mean_of_values():
    D, n = 8, 5
    K = rng0.normal(size=(1, n, D))
    V = np.round(rng0.normal(size=(1, n, D)) * 8) / 8  # exactly representable
    o = run_attn(np.zeros((1, 1, D)), [K], [V], [n], [n], 1, 1, D)
    assert np.allclose(o[0, 0], V[0].mean(axis=0), atol=1e-15)


def test_attention_two_keys_logistic_closed_form():
    D = 4
    q = np.array([[[1.0, 0.5, 0.0, -1.0]]])
    k = np.array([[[1.0, 1.0, 0.0, 0.0], [0.0, -1.0, 2.0, 1.0]]])
    v = np.array([[[1.0, 0.0, 0.0, 2.0], [0.0, 1.0, -3.0, 0.0]]])
    scale = 0.7
    s1, s2 = scale * (1.0 + 0.5), scale * (-0.5 - 1.0)
    p1 = 1.0 / (1.0 + math.exp(s2 - s1))
    expect = p1 * v[0, 0] + (1 - p1) * v[0, 1]
    o = run_attn(q, [k], [v], [2], [2], 1, 1, D, scale)
    assert np.allclose(o[0, 0], expect, atol=1e-15)


def test_attention_gqa_head_mapping():
    # Hq = 4, Hkv = 2: query heads 0,1 read kv-head 0; heads 2,3 read kv-head 1
    D, n = 4, 3
    K = [rng0.normal(size=(n, D)), rng0.normal(size=(n, D))]
    V = [np.ones((n, D)), -np.ones((n, D))]
    q = rng0.normal(size=(1, 4, D))
    o = run_attn(q, [K], [V], [n], [n], 4, 2, D)
    assert np.allclose(o[0, 0], 1) and np.allclose(o[0, 1], 1)
    assert np.allclose(o[0, 2], -1) and np.allclose(o[0, 3], -1)


def test_attention_ignores_rows_beyond_length_and_uses_own_slab():
    D = 4
    big = np.full((2, D), 50.0)
    K0 = np.concatenate([rng0.normal(size=(3, D)), big])
    V0 = np.concatenate([np.full((3, D), 2.0), np.full((2, D), -100.0)])
    K1 = rng0.normal(size=(5, D))
    V1 = np.full((5, D), -7.0)
    q = np.ones((2, 1, D))
    o = run_attn(q, [[K0], [K1]], [[V0], [V1]], [3, 5], [5, 6], 1, 1, D)
    assert np.allclose(o[0, 0], 2.0) and np.allclose(o[1, 0], -7.0)


def test_attention_random_tiny_against_logsumexp_route_and_invariants():
    for trial in range(20):
        n, D, Hq, Hkv = int(rng0.integers(1, 9)), 4, 2, 1
        K = rng0.normal(size=(1, n, D))
        V = rng0.normal(size=(1, n, D))
        q = rng0.normal(size=(1, Hq, D))
        o = run_attn(q, [K], [V], [n], [n], Hq, Hkv, D)
        Kb = oracle.bf16_to_f64(bf16_bits(K[0]))
        Vb = oracle.bf16_to_f64(bf16_bits(V[0]))
        qb = oracle.bf16_to_f64(bf16_bits(q[0]))
        for h in range(Hq):
            s = np.array([math.fsum(qb[h] * Kb[j]) for j in range(n)]) / 2.0
            lse = max(s) + math.log(math.fsum(math.exp(x - max(s)) for x in s))
            p = np.array([math.exp(x - lse) for x in s])
            expect = np.array([math.fsum(p * Vb[:, i]) for i in range(D)])
            assert np.allclose(o[0, h], expect, atol=1e-13)
            assert np.all(o[0, h] <= Vb.max(axis=0) + 1e-12) and np.all(o[0, h] >= Vb.min(axis=0) - 1e-12)
        perm = rng0.permutation(n)
        o2 = run_attn(q, [K[:, perm]], [V[:, perm]], [n], [n], Hq, Hkv, D)
        assert np.allclose(o, o2, atol=1e-13)


# ------------------------------------------------------- unembedding / softmax
def test_lm_head_rows_are_normalised_log_probs():
    S, d, V = 3, 16, 40
    h = bf16_bits(rng0.normal(size=(S, d)))
    w = bf16_bits(rng0.normal(size=(V, d)) * 0.3)
    lp, lse = oracle.lm_head_logprobs(h, w)
    assert np.all(lp <= 0)
    assert np.allclose(np.exp(lp).sum(axis=1), 1.0, atol=1e-12)
    z = oracle.bf16_to_f64(h) @ oracle.bf16_to_f64(w).T  # independent library matmul
    m = z.max(axis=1, keepdims=True)
    ref_lse = (m + np.log(np.exp(z - m).sum(axis=1, keepdims=True)))[:, 0]
    assert np.allclose(lse, ref_lse, atol=1e-12)
    assert np.allclose(lp, z - ref_lse[:, None], atol=1e-12)


def test_lm_head_one_hot_hidden_selects_weight_column():
    d, V, i = 8, 12, 5
    h = np.zeros((1, d))
    h[0, i] = 1.0
    wv = rng0.normal(size=(V, d))
    lp, lse = oracle.lm_head_logprobs(bf16_bits(h), bf16_bits(wv))
    col = oracle.bf16_to_f64(bf16_bits(wv))[:, i]  # z_v = W[v][i]: a transposed W would give a row
    assert np.allclose(lp[0], col - math.log(np.exp(col).sum()), atol=1e-13)


def test_lm_head_zero_hidden_is_uniform():
    V = 37
    lp, lse = oracle.lm_head_logprobs(np.zeros((1, 4), np.uint16), bf16_bits(rng0.normal(size=(V, 4))))
    assert np.allclose(lp, -math.log(V), atol=1e-14)


# ------------------------------------------------------------ Eq. 2 + Eq. 3
def log_softmax(z):
    m = z.max(axis=-1, keepdims=True)
    return z - (m + np.log(np.exp(z - m).sum(axis=-1, keepdims=True)))


def random_lp(B, N, V, scale=2.0):
    return log_softmax(rng0.normal(size=(B * (N + 1), V)) * scale)


def test_select_hand_worked_example():
    # V = 3, N = 2, beta = 0.5, gamma = 1, r = (0.5, 0.25)
    lp0 = np.log([0.7, 0.2, 0.1])
    lp1 = np.log([0.6, 0.3, 0.1])
    lp2 = np.log([0.2, 0.2, 0.6])
    lp = np.stack([lp0, lp1, lp2])
    beta = np.array([[0.5, 0.5]], np.float32)
    r = np.array([[0.5, 0.25]], np.float32)
    # shat_1 = 1.5 lp1 - 0.5 lp0 + log 0.5  -> (-1.28105, -1.69439, -2.99573)
    # shat_2 = 1.5 lp2 - 0.5 lp0 + log 0.25 -> (-3.62211, -2.99573, -1.00124)
    out = oracle.contrastive_select(lp, beta, r, 1.0, 1, 2)
    assert out["token"][0] == 2 and out["expert"][0] == 2
    expect = 1.5 * math.log(0.6) - 0.5 * math.log(0.1) + math.log(0.25)
    assert abs(out["score"][0] - (1.5 * math.log(0.6) - 0.5 * math.log(0.1) + math.log(0.25))) < 1e-12
    assert abs(out["token_gap"][0] - (expect - (1.5 * math.log(0.6) - 0.5 * math.log(0.7) + math.log(0.5)))) < 1e-12
    # a flipped amateur sign (+beta lp0) would pick token 0 of expert 1 instead:
    # 1.5 lp1 + 0.5 lp0 + log 0.5 = -1.63773 beats every other candidate then.


def test_select_prior_decides_between_equal_experts():
    # identical expert rows, identical beta: only gamma*log r differs, so the
    # expert with the larger relevance must win (a flipped prior sign picks the other)
    V = 10
    row = log_softmax(rng0.normal(size=V))
    lp = np.stack([log_softmax(rng0.normal(size=V)), row, row])
    beta = np.array([[0.5, 0.5]], np.float32)
    out = oracle.contrastive_select(lp, beta, np.array([[0.2, 0.9]], np.float32), 2.5, 1, 2)
    assert out["expert"][0] == 2
    out = oracle.contrastive_select(lp, beta, np.array([[0.9, 0.2]], np.float32), 2.5, 1, 2)
    assert out["expert"][0] == 1
    assert abs(out["expert_gap"][0] - 2.5 * math.log(0.9 / 0.2)) < 1e-6


def test_select_contrast_penalises_amateur_favourites():
    # expert prefers token 0 slightly over token 1; the amateur loves token 0.
    # beta = 0 keeps token 0, beta = 1 moves to token 1 (amateur enters with a minus sign)
    lp1 = np.log([0.5, 0.45, 0.05])
    lp0 = np.log([0.9, 0.05, 0.05])
    lp = np.stack([lp0, lp1])
    r = np.array([[0.5]], np.float32)
    assert oracle.contrastive_select(lp, np.array([[0.0]], np.float32), r, 2.5, 1, 1)["token"][0] == 0
    assert oracle.contrastive_select(lp, np.array([[1.0]], np.float32), r, 2.5, 1, 1)["token"][0] == 1


def test_select_single_expert_no_contrast_no_prior_is_greedy():
    for _ in range(20):
        V = 50
        z = rng0.normal(size=(2, V)) * 3
        lp = log_softmax(z)
        out = oracle.contrastive_select(lp, np.zeros((1, 1), np.float32), np.array([[0.3]], np.float32), 0.0, 1, 1)
        assert out["token"][0] == int(np.argmax(z[1])) and out["expert"][0] == 1


def test_select_beta_zero_is_retrieval_weighted_max():
    B, N, V = 3, 5, 30
    lp = random_lp(B, N, V)
    r = rng0.uniform(0.05, 1, size=(B, N)).astype(np.float32)
    g = 2.5
    out = oracle.contrastive_select(lp, np.zeros((B, N), np.float32), r, g, B, N)
    for b in range(B):
        cand = lp[b * (N + 1) + 1:(b + 1) * (N + 1)] + g * np.log(r[b].astype(np.float64))[:, None]
        k, v = np.unravel_index(np.argmax(cand), cand.shape)
        assert out["token"][b] == v and out["expert"][b] == k + 1


def test_select_flat_prior_equals_no_prior_and_scale_invariance():
    B, N, V = 4, 6, 40
    lp = random_lp(B, N, V)
    beta = rng0.uniform(0, 1, size=(B, N)).astype(np.float32)
    r = rng0.uniform(0.05, 1, size=(B, N)).astype(np.float32)
    base = oracle.contrastive_select(lp, beta, np.full((B, N), 0.37, np.float32), 2.5, B, N)
    nog = oracle.contrastive_select(lp, beta, r, 0.0, B, N)
    assert np.array_equal(base["token"], nog["token"]) and np.array_equal(base["expert"], nog["expert"])
    a = oracle.contrastive_select(lp, beta, r, 2.5, B, N)
    c = oracle.contrastive_select(lp, beta, (r * np.float32(0.25)).astype(np.float32), 2.5, B, N)
    assert np.array_equal(a["token"], c["token"]) and np.array_equal(a["expert"], c["expert"])


def test_select_expert_permutation_invariance():
    B, N, V = 2, 7, 64
    lp = random_lp(B, N, V)
    beta = rng0.uniform(0, 1, size=(B, N)).astype(np.float32)
    r = rng0.uniform(0.05, 1, size=(B, N)).astype(np.float32)
    a = oracle.contrastive_select(lp, beta, r, 2.5, B, N)
    perm = rng0.permutation(N)
    lp2 = lp.copy()
    for b in range(B):
        lp2[b * (N + 1) + 1:(b + 1) * (N + 1)] = lp[b * (N + 1) + 1 + perm]
    c = oracle.contrastive_select(lp2, beta[:, perm], r[:, perm], 2.5, B, N)
    assert np.array_equal(a["token"], c["token"])
    for b in range(B):
        assert perm[c["expert"][b] - 1] + 1 == a["expert"][b]


def test_select_never_returns_the_amateur_and_gaps_match_brute_force():
    B, N, V = 3, 4, 25
    lp = random_lp(B, N, V)
    for b in range(B):
        lp[b * (N + 1), 3] = 5.0  # amateur spike (not a valid log-prob; only enters with -beta)
    beta = np.full((B, N), 0.5, np.float32)
    r = rng0.uniform(0.05, 1, size=(B, N)).astype(np.float32)
    out = oracle.contrastive_select(lp, beta, r, 2.5, B, N)
    for b in range(B):
        assert 1 <= out["expert"][b] <= N
        shat = np.array([(1 + 0.5) * lp[b * (N + 1) + k] - 0.5 * lp[b * (N + 1)]
                         + 2.5 * math.log(float(r[b, k - 1])) for k in range(1, N + 1)])
        flat = sorted(((shat[k, v], v, k) for k in range(N) for v in range(V)), reverse=True)
        best = flat[0]
        assert out["token"][b] == best[1] and out["expert"][b] == best[2] + 1 and out["token"][b] != 3
        runner_tok = max(x[0] for x in flat if x[1] != best[1])
        runner_exp = max((x[0] for x in flat if x[1] == best[1] and x[2] != best[2]), default=-math.inf)
        assert abs(out["token_gap"][b] - (best[0] - runner_tok)) < 1e-12
        assert abs(out["expert_gap"][b] - (best[0] - runner_exp)) < 1e-12


def test_select_exact_tie_rules():
    V = 8
    row = np.full(V, -5.0)
    row[3] = row[5] = -0.1  # equal best tokens within an expert -> lower id
    lp = np.stack([np.full(V, -math.log(V)), row, row])  # equal experts -> lower index
    out = oracle.contrastive_select(lp, np.full((1, 2), 0.5, np.float32), np.full((1, 2), 0.5, np.float32),
                                    2.5, 1, 2)
    assert out["token"][0] == 3 and out["expert"][0] == 1
    assert out["token_gap"][0] == 0.0 and out["expert_gap"][0] == 0.0


def test_select_relevance_is_clipped_away_from_zero():
    lp = np.stack([np.log([0.5, 0.5]), np.log([0.9, 0.1]), np.log([0.1, 0.9])])
    out = oracle.contrastive_select(lp, np.zeros((1, 2), np.float32), np.array([[0.0, 1e-9]], np.float32),
                                    1.0, 1, 2)
    # both clip to 1e-8, so the prior is flat and expert 1 / token 0 wins the first tie by scan order
    assert math.isfinite(out["score"][0])
    assert abs(out["score"][0] - (math.log(0.9) + math.log(1e-8))) < 1e-9


# -------------------------------------------------------- composed decode step
def empty_prefix_case(L, Hq=4, Hkv=2, D=8, V=16, N=1, B=1, cap=4):
    S = B * (N + 1)
    d = Hq * D
    lay_elems = S * Hkv * cap * D
    kc = np.zeros(L * lay_elems, np.uint16)
    vc = np.zeros(L * lay_elems, np.uint16)
    off = np.arange(S, dtype=np.int64) * Hkv * cap * D
    capa = np.full(S, cap, np.int32)
    lens = np.zeros(S, np.int32)
    emb = bf16_bits(rng0.normal(size=(B, d)))
    w = bf16_bits(rng0.normal(size=(V, d)) * 0.1)
    dims = dict(B=B, N=N, L=L, Hq=Hq, Hkv=Hkv, D=D, V=V, gamma=2.5)
    return dims, kc, vc, lay_elems, off, capa, lens, emb, w


@pytest.mark.parametrize("L", [1, 3])
def test_step_with_empty_prefix_closed_form(L):
    # With empty caches, the only key of every layer is the token appended this
    # step, so attention returns its value row: query head hq gets the
    # normalised input's head Hkv + hq // G.  The residual stream then has a
    # closed form layer by layer.
    dims, kc, vc, lay, off, cap, lens, emb, w = empty_prefix_case(L)
    Hq, Hkv, D = dims["Hq"], dims["Hkv"], dims["D"]
    G = Hq // Hkv
    beta = np.full((1, 1), 0.5, np.float32)
    r = np.full((1, 1), 0.8, np.float32)
    out = oracle.decode_step(dims, kc, vc, lay, off, cap, lens, emb, w, beta, r)
    assert np.array_equal(lens, [1, 1])
    x = oracle.bf16_to_f64(emb[0])
    for l in range(L):
        xn = x / math.sqrt(np.mean(x * x) + oracle.RMS_EPS)
        u = oracle.bf16_to_f64(bf16_bits(xn)).reshape(Hq, D)
        for s in range(2):
            for h in range(Hkv):
                base = l * lay + off[s] + h * cap[s] * D
                assert np.array_equal(oracle.bf16_to_f64(kc[base:base + D]), u[h])
                assert np.array_equal(oracle.bf16_to_f64(vc[base:base + D]), u[Hkv + h])
        o = np.stack([u[Hkv + hq // G] for hq in range(Hq)]).ravel()
        x = x + o
    h = bf16_bits(x / math.sqrt(np.mean(x * x) + oracle.RMS_EPS))
    assert np.array_equal(out["h"][0], h) and np.array_equal(out["h"][1], h)
    z = oracle.bf16_to_f64(h) @ oracle.bf16_to_f64(w).T
    lse = z.max() + math.log(np.exp(z - z.max()).sum())
    assert np.allclose(out["lse"], lse, atol=1e-12)
    # expert and amateur see the same single token, so lp_1 == lp_0 and shat = lp + gamma log r
    assert out["token"][0] == int(np.argmax(z)) and out["expert"][0] == 1
    assert abs(out["score"][0] - (z.max() - lse + 2.5 * math.log(float(np.float32(0.8))))) < 1e-9


def test_step_appends_chosen_token_to_every_expert():
    w = synth.get("tiny", V=512, steps=2)
    from oracle.run import OracleRun
    run = OracleRun(w)
    o1 = run.step()
    lens1 = run.lens.copy()
    assert np.array_equal(lens1, synth.base_lengths(w) + 1)
    o2 = run.step()
    assert np.array_equal(run.lens, lens1 + 1)
    # the second step's appended key rows are the normalised embedding of the first step's token
    e = oracle.bf16_to_f64(synth.host_matrix(w, synth.T_EMBED, row0=int(o1["token"][0]), rows=1)[0])
    u = bf16_bits(e / math.sqrt(np.mean(e * e) + oracle.RMS_EPS))
    for s in range(w.S):
        pos = lens1[s]
        for h in range(w.Hkv):
            base = run.layout.kv_offset[s] + (h * run.layout.cap[s] + pos) * w.D
            assert np.array_equal(run.kc[base:base + w.D], u[h * w.D:(h + 1) * w.D])
            assert np.array_equal(run.vc[base:base + w.D], u[(w.Hkv + h) * w.D:(w.Hkv + h + 1) * w.D])
    assert 1 <= o2["expert"][0] <= w.N


# --------------------------------------------------- rotary position embedding
# The decoder LLMs the paper runs (Llama, Qwen) rotate queries and keys by
# position.  Reading: rotate-half pairing (f, f + D/2), inverse frequency
# theta^(-2f/D), angle pos * inv_freq in fp32 as the models compute it.
def test_rope_position_zero_is_identity():
    x = rng0.normal(size=64)
    assert np.array_equal(oracle.rope(x, 0, 5e5), x)


def test_rope_two_dims_is_a_plane_rotation_by_the_position():
    # D = 2: the only inverse frequency is theta^0 = 1, so the angle is pos
    x = np.array([0.75, -1.25])
    for pos in (1, 2, 7, 1000):
        c, s_ = math.cos(pos), math.sin(pos)
        want = np.array([x[0] * c - x[1] * s_, x[1] * c + x[0] * s_])
        assert np.allclose(oracle.rope(x, pos, 1e4), want, rtol=0, atol=1e-15)


def test_rope_frequencies_and_rotate_half_pairing():
    # theta = 2^16, D = 16: inverse frequencies 4^-f are exact in fp32, so the
    # angles are exactly pos * 4^-f; a unit vector on dimension f moves towards
    # f + D/2 (and f + D/2 towards f, with the opposite sign)
    D, theta, pos = 16, 65536.0, 37
    for f in range(D // 2):
        a = pos * 4.0 ** -f
        e = np.zeros(D); e[f] = 1.0
        y = oracle.rope(e, pos, theta)
        want = np.zeros(D); want[f] = math.cos(a); want[f + D // 2] = math.sin(a)
        assert np.allclose(y, want, rtol=0, atol=1e-15)
        e = np.zeros(D); e[f + D // 2] = 1.0
        y = oracle.rope(e, pos, theta)
        want = np.zeros(D); want[f] = -math.sin(a); want[f + D // 2] = math.cos(a)
        assert np.allclose(y, want, rtol=0, atol=1e-15)


def test_rope_scores_depend_on_relative_position_only():
    D, theta = 16, 65536.0  # exact angles, see above
    q, k = rng0.normal(size=D), rng0.normal(size=D)
    for m, n, t in ((5, 2, 11), (0, 9, 100), (300, 300, 7)):
        a = oracle.rope(q, m, theta) @ oracle.rope(k, n, theta)
        b = oracle.rope(q, m + t, theta) @ oracle.rope(k, n + t, theta)
        assert abs(a - b) < 1e-12
    # and it is a rotation: every (f, f + D/2) pair keeps its length
    y = oracle.rope(q, 12345, 5e5)
    assert np.allclose(np.hypot(y[:D // 2], y[D // 2:]), np.hypot(q[:D // 2], q[D // 2:]), rtol=1e-14)


def test_step_with_rope_rotates_queries_and_keys_at_the_token_position_not_values():
    # Two zero prefix rows, then this step's token at position 2.  The new K row
    # is bf16(rope(n[h], 2)), the V row bf16(n[Hkv + h]) unrotated; attention of
    # query head hq over keys (0, 0, k) gives e^s / (2 + e^s) * v with
    # s = scale * (rotated q) . (rotated k).
    dims, kc, vc, lay, off, cap, lens, emb, w = empty_prefix_case(1)
    dims["rope_theta"] = 1e4
    lens[:] = 2
    Hq, Hkv, D = dims["Hq"], dims["Hkv"], dims["D"]
    G = Hq // Hkv
    beta = np.full((1, 1), 0.5, np.float32)
    r = np.full((1, 1), 0.8, np.float32)
    out = oracle.decode_step(dims, kc, vc, lay, off, cap, lens, emb, w, beta, r)
    x = oracle.bf16_to_f64(emb[0])
    n = (x / math.sqrt(np.mean(x * x) + oracle.RMS_EPS)).reshape(Hq, D)
    q = np.stack([oracle.bf16_to_f64(bf16_bits(oracle.rope(n[hq], 2, 1e4))) for hq in range(Hq)])
    v = np.stack([oracle.bf16_to_f64(bf16_bits(n[Hkv + h])) for h in range(Hkv)])
    for s in range(2):
        for h in range(Hkv):
            base = off[s] + (h * cap[s] + 2) * D
            assert np.array_equal(oracle.bf16_to_f64(kc[base:base + D]), q[h])
            assert np.array_equal(oracle.bf16_to_f64(vc[base:base + D]), v[h])
    scale = 1.0 / math.sqrt(D)
    o = []
    for hq in range(Hq):
        sc = scale * (q[hq] @ q[hq // G])
        o.append(math.exp(sc) / (2.0 + math.exp(sc)) * v[hq // G])
    x1 = x + np.concatenate(o)
    h = bf16_bits(x1 / math.sqrt(np.mean(x1 * x1) + oracle.RMS_EPS))
    assert np.array_equal(out["h"][0], h) and np.array_equal(out["h"][1], h)


# ------------------------------------- relevance normalisation and fusion
# App. "Normalization of Retrieval and Reranker Scores", eps = 1e-8.
EPS = 1e-8


def test_relevance_dense_endpoints_and_midpoint():
    r = oracle.relevance([-1.0, 1.0, 0.0, -3.0, 2.0, 0.5], 0)
    assert list(r) == [0.0, 1.0 - EPS, 0.5, 0.0, 1.0 - EPS, 0.75]


def test_relevance_sparse_saturating_arctan():
    r = oracle.relevance([0.0, -5.0, 1.0, math.tan(math.pi / 8), 1e30], 1)
    assert r[0] == 0.0 and r[1] == 0.0           # max(s, 0) then atan(0) = 0
    assert abs(r[2] - 0.5) < 1e-15                # (2/pi) atan(1) = 1/2
    assert abs(r[3] - 0.25) < 1e-15               # (2/pi)(pi/8)
    assert r[4] == 1.0 - EPS                      # saturates below 1
    xs = np.linspace(0, 50, 101)
    assert np.all(np.diff(oracle.relevance(xs, 1)) > 0)  # monotone


def test_relevance_reranker_sigmoid_and_harmonic_mean():
    # dense s = 0 gives r_ret = 1/2; reranker z = 0 gives 1/2; HM(1/2, 1/2) = 1/(1 + eps)
    r = oracle.relevance([0.0], 0, z=[0.0])
    assert abs(r[0] - 0.5 / (1.0 + EPS)) < 1e-16
    # z = ln 3: sigmoid = 3/4; with r_ret = 1/2: HM = 2 (3/8) / (5/4 + eps)
    r = oracle.relevance([0.0], 0, z=[math.log(3.0)])
    assert abs(r[0] - 0.75 / (1.25 + EPS)) < 1e-15
    # a zero on either side gives zero; the fusion is symmetric
    assert oracle.relevance([-1.0], 0, z=[0.3])[0] == 0.0
    a = oracle.relevance([0.2], 0, z=[-0.7])[0]
    b = oracle.relevance([2 * (1 / (1 + math.exp(0.7))) - 1], 0, z=[math.log(0.6 / 0.4)])[0]
    assert abs(a - b) < 1e-15
    # between the smaller input and the geometric mean, in [0, 1)
    s = rng0.uniform(-1, 1, 50)
    z = rng0.normal(size=50) * 3
    r = oracle.relevance(s, 0, z=z)
    rr = (s + 1) / 2
    rz = 1 / (1 + np.exp(-z))
    assert np.all(r <= np.sqrt(rr * rz) + 1e-15) and np.all(r >= np.minimum(rr, rz) * (1 - 1e-7) - 1e-15)
    assert np.all((r >= 0) & (r < 1))


def test_relevance_without_reranker_is_the_retrieval_score():
    s = rng0.uniform(-1, 1, 20)
    assert np.array_equal(oracle.relevance(s, 0), np.clip((s + 1) / 2, 0, 1 - EPS))
    with pytest.raises(ValueError):
        oracle.relevance(s, 2)


# ------------------------------------------- aggregation variants (MoE / PoE)
# App. "Ablation of Expert Aggregation Rule".  Reading: p_k = softmax of the
# contrastive scores of Eq. 2 without the prior, weights r_k / sum r, MoE =
# weighted sum of the p_k, PoE = weighted product (sum of weighted logs).
def _lp(*rows):
    return np.log(np.array(rows, np.float64))


def test_aggregate_hand_worked_example_separates_max_moe_and_poe():
    u = [1 / 3] * 3
    lp = _lp(u, [0.7, 0.2, 0.1], [0.05, 0.35, 0.6])
    beta = np.zeros((1, 2), np.float32)
    r = np.full((1, 2), 0.5, np.float32)
    moe = oracle.aggregate_select(lp, beta, r, oracle.MOE)
    poe = oracle.aggregate_select(lp, beta, r, oracle.POE)
    # MoE: (0.375, 0.275, 0.35) -> token 0, carried by expert 1
    assert moe["token"][0] == 0 and moe["expert"][0] == 1
    assert abs(moe["score"][0] - math.log(0.375)) < 1e-12
    assert abs(moe["token_gap"][0] - math.log(0.375 / 0.35)) < 1e-12
    # PoE: sqrt of (0.035, 0.07, 0.06) -> token 1, where expert 2 puts more mass
    assert poe["token"][0] == 1 and poe["expert"][0] == 2
    assert abs(poe["score"][0] - 0.5 * math.log(0.07)) < 1e-12
    # attribution margins (log w p at the token): MoE 0.5*0.7 against 0.5*0.05,
    # PoE 0.5*0.35 against 0.5*0.2
    assert abs(moe["expert_gap"][0] - math.log(14.0)) < 1e-12
    assert abs(poe["expert_gap"][0] - math.log(1.75)) < 1e-12
    # Max (Eq. 3 with gamma = 0, beta = 0): the single most confident expert wins, token 0
    mx = oracle.contrastive_select(lp, beta, r, 0.0, 1, 2)
    assert mx["token"][0] == 0 and mx["expert"][0] == 1


def test_aggregate_weights_are_normalised_retrieval_scores():
    lp = _lp([0.25] * 4, [0.1, 0.6, 0.2, 0.1], [0.5, 0.1, 0.1, 0.3])
    beta = np.zeros((1, 2), np.float32)
    for scale in (1.0, 0.1):
        r = (np.array([[0.9, 0.1]]) * scale).astype(np.float32)
        moe = oracle.aggregate_select(lp, beta, r, oracle.MOE)
        w = r[0].astype(np.float64) / r[0].astype(np.float64).sum()
        mix = w[0] * np.array([0.1, 0.6, 0.2, 0.1]) + w[1] * np.array([0.5, 0.1, 0.1, 0.3])
        assert moe["token"][0] == 1 and abs(moe["score"][0] - math.log(mix[1])) < 1e-12
    # flipping the weights flips the winner
    r = np.array([[0.1, 0.9]], np.float32)
    assert oracle.aggregate_select(lp, beta, r, oracle.MOE)["token"][0] == 0


def test_aggregate_contrast_sharpens_against_a_flat_amateur():
    # uniform amateur: c_k = (1 + beta) log p_k + const, so p_k becomes p_k^(1+beta) renormalised
    p1 = np.array([0.7, 0.2, 0.1])
    lp = _lp([1 / 3] * 3, p1, [0.2, 0.5, 0.3])
    beta = np.ones((1, 2), np.float32)
    r = np.array([[1.0, 1e-30]], np.float32)  # clipped to 1e-8: expert 2 weighs ~1e-8
    moe = oracle.aggregate_select(lp, beta, r, oracle.MOE)
    sq = p1 ** 2 / (p1 ** 2).sum()
    assert moe["token"][0] == 0 and abs(moe["score"][0] - math.log(sq[0])) < 1e-6


def test_aggregate_single_expert_is_contrastive_greedy_and_permutation_invariant():
    rng = np.random.default_rng(3)
    V = 50
    z = rng.normal(size=(2, V)) * 3
    lp = z - np.log(np.exp(z).sum(1, keepdims=True))
    beta = np.full((1, 1), 0.5, np.float32)
    r = np.full((1, 1), 0.3, np.float32)
    tok = oracle.contrastive_select(lp, beta, r, 0.0, 1, 1)["token"]
    for rule in (oracle.MOE, oracle.POE):
        out = oracle.aggregate_select(lp, beta, r, rule)
        assert out["token"][0] == tok[0] and out["expert"][0] == 1
        assert out["expert_gap"][0] == math.inf  # no other expert to mistake it for
    # two copies of one expert with equal scores: an exact attribution tie,
    # margin 0, the lower index reported
    lp2 = lp[[0, 1, 1]]
    for rule in (oracle.MOE, oracle.POE):
        out = oracle.aggregate_select(lp2, np.full((1, 2), 0.5, np.float32), np.full((1, 2), 0.3, np.float32), rule)
        assert out["expert"][0] == 1 and out["expert_gap"][0] == 0.0
    z = rng.normal(size=(4, V)) * 2
    lp = z - np.log(np.exp(z).sum(1, keepdims=True))
    beta = np.array([[0.2, 0.7, 0.4]], np.float32)
    r = np.array([[0.5, 0.2, 0.9]], np.float32)
    perm = [2, 0, 1]
    for rule in (oracle.MOE, oracle.POE):
        a = oracle.aggregate_select(lp, beta, r, rule)
        b = oracle.aggregate_select(lp[[0] + [1 + p for p in perm]], beta[:, perm], r[:, perm], rule)
        assert a["token"][0] == b["token"][0] and abs(a["score"][0] - b["score"][0]) < 1e-12
        assert perm[b["expert"][0] - 1] + 1 == a["expert"][0]


def test_aggregate_depends_on_each_row_only_up_to_a_constant():
    # MoE and PoE take p_k as the softmax of the contrastive scores, so a
    # constant added to any row (raw logits z = lp + L instead of lp) shifts
    # each expert's scores by a constant that the softmax removes: the choice,
    # the aggregate and both margins stay the same
    rng = np.random.default_rng(11)
    B, N, V = 2, 3, 64
    z = rng.normal(size=(B * (N + 1), V)) * 2
    lp = z - np.log(np.exp(z).sum(1, keepdims=True))
    beta = rng.uniform(0.1, 0.9, (B, N)).astype(np.float32)
    r = rng.uniform(0.05, 0.95, (B, N)).astype(np.float32)
    shifted = lp + rng.normal(size=(B * (N + 1), 1)) * 7
    for rule in (oracle.MOE, oracle.POE):
        a = oracle.aggregate_select(lp, beta, r, rule)
        b = oracle.aggregate_select(shifted, beta, r, rule)
        assert np.array_equal(a["token"], b["token"]) and np.array_equal(a["expert"], b["expert"])
        for key in ("score", "token_gap", "expert_gap"):
            assert np.allclose(a[key], b[key], rtol=0, atol=1e-9), key
    # Eq. 3 itself is not invariant: its per-expert constants carry the L_k
    a = oracle.contrastive_select(lp, beta, r, 2.5, B, N)
    b = oracle.contrastive_select(shifted, beta, r, 2.5, B, N)
    assert not np.allclose(a["score"], b["score"])


def test_step_raw_logit_mode_and_moe_in_closed_form():
    # one expert over an empty prefix: expert and amateur see the same single
    # token, so lp_1 = lp_0 and (1 + beta) s_1 - beta s_0 = s_1.  Log-prob mode
    # scores z* - lse + gamma log r; raw-logit mode z* + gamma log r; MoE picks
    # the same token with score log p(token) and no prior.
    outs = {}
    case = empty_prefix_case(1)
    for key, extra in (("lp", {}), ("raw", dict(score_mode=1)), ("moe", dict(aggregation=1)),
                       ("poe", dict(aggregation=2))):
        dims, kc, vc, lay, off, cap, lens, emb, w = [x.copy() if hasattr(x, "copy") else x for x in case]
        dims.update(extra)
        beta = np.full((1, 1), 0.5, np.float32)
        r = np.full((1, 1), 0.8, np.float32)
        outs[key] = oracle.decode_step(dims, kc, vc, lay, off, cap, lens, emb, w, beta, r)
    lse = outs["lp"]["lse"][1]
    assert all(outs[k]["token"][0] == outs["lp"]["token"][0] for k in outs)
    assert abs(outs["raw"]["score"][0] - outs["lp"]["score"][0] - lse) < 1e-9
    prior = 2.5 * math.log(float(np.float32(0.8)))
    for k in ("moe", "poe"):
        assert abs(outs[k]["score"][0] - (outs["lp"]["score"][0] - prior)) < 1e-9
        assert outs[k]["expert"][0] == 1


# --------------------------------------------------------------- paper figures
def test_kv_storage_example_from_paper():
    import json, os
    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "kv_storage_example.json")))
    per_tok = synth.kv_bytes_per_token(g["layers"], g["kv_heads"], g["head_dim"], g["bytes_per_elem"])
    total = per_tok * g["passages"] * g["tokens_per_passage"]
    assert per_tok == 128 * 1024
    assert abs(total / 2 ** 30 - g["reported_gb"]) < 0.005


# ------------------------------------------ dynamic contrast strength (AdaCAD)
# beta_k = Jensen-Shannon divergence in bits between expert k's and the
# amateur's next-token distributions (the reading of "computed as in AdaCAD").
def _rows_from_probs(*rows):
    """log-probability rows (-inf where p = 0) of the given probability rows"""
    with np.errstate(divide="ignore"):
        return np.log(np.array(rows, np.float64))


def test_adacad_beta_identical_distributions_is_zero():
    p = rng0.dirichlet(np.ones(40))
    beta = oracle.adacad_beta(_rows_from_probs(p, p), 1, 1)
    assert abs(beta[0, 0]) < 1e-15


def test_adacad_beta_disjoint_supports_is_one_bit():
    amateur = np.zeros(6)
    amateur[1] = 1.0
    expert = np.zeros(6)
    expert[4] = 1.0
    beta = oracle.adacad_beta(_rows_from_probs(amateur, expert), 1, 1)
    assert beta[0, 0] == pytest.approx(1.0, abs=1e-15)


def test_adacad_beta_two_point_closed_form():
    # expert (1, 0) against amateur (1/2, 1/2): the midpoint is (3/4, 1/4), so
    # JSD = H(3/4, 1/4) - (H(expert) + H(amateur)) / 2 = (2 - 3/4 log2 3) - 1/2
    beta = oracle.adacad_beta(_rows_from_probs([0.5, 0.5], [1.0, 0.0]), 1, 1)
    assert beta[0, 0] == pytest.approx(1.5 - 0.75 * math.log2(3.0), abs=1e-14)


def test_adacad_beta_matches_entropy_form_is_symmetric_and_bounded():
    def H(p):
        p = p[p > 0]
        return float(-(p * np.log2(p)).sum())
    for trial in range(5):
        V = int(rng0.integers(2, 300))
        p = rng0.dirichlet(np.full(V, 0.3))
        q = rng0.dirichlet(np.full(V, 0.3))
        b_pq = oracle.adacad_beta(_rows_from_probs(q, p), 1, 1)[0, 0]
        b_qp = oracle.adacad_beta(_rows_from_probs(p, q), 1, 1)[0, 0]
        assert b_pq == pytest.approx(H(0.5 * (p + q)) - 0.5 * (H(p) + H(q)), abs=1e-12)
        assert b_pq == pytest.approx(b_qp, abs=1e-14)
        assert 0.0 <= b_pq <= 1.0


def test_adacad_beta_row_layout_per_query_and_expert():
    # query-major rows, the amateur first: beta[b][k-1] compares row b*(N+1)+k with row b*(N+1)
    B, N, V = 2, 3, 17
    probs = [rng0.dirichlet(np.ones(V)) for _ in range(B * (N + 1))]
    beta = oracle.adacad_beta(_rows_from_probs(*probs), B, N)
    for b in range(B):
        for k in range(1, N + 1):
            single = oracle.adacad_beta(_rows_from_probs(probs[b * (N + 1)], probs[b * (N + 1) + k]), 1, 1)
            assert beta[b, k - 1] == single[0, 0]


def test_step_with_dynamic_beta_uses_the_first_step_distributions():
    # the step's beta is the divergence of this step's own distributions, and
    # the selection of that step is Eq. 2 + Eq. 3 with it
    from oracle.run import OracleRun
    w = synth.get("tiny")
    run = OracleRun(w, dynamic_beta=True)
    out = run.step()
    lp, _ = oracle.lm_head_logprobs(out["h"], run.w_bits)
    want = oracle.adacad_beta(lp, w.B, w.N).astype(np.float32)
    assert np.array_equal(out["beta"], want)
    sel = oracle.contrastive_select(lp, want, run.r, w.gamma, w.B, w.N)
    assert np.array_equal(sel["token"], out["token"]) and np.array_equal(sel["expert"], out["expert"])
    # later steps keep it
    assert np.array_equal(run.beta, want)
    run.step()
    assert np.array_equal(run.beta, want)
