"""Pins of the CPU oracle to facts outside itself (CPU only).

Each check uses a closed form, an invariant, exact rational arithmetic, or a
published number, chosen so that a plausible slip in the oracle (a transposed
operand, a dropped term, a wrong sign, epsilon in the wrong place, the wrong
RoPE frequency or pairing, the SwiGLU gate on the wrong matrix, a missing KV
cache entry or residual, the wrong grouped-query head) makes one of them fail.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2601_03324_gb300 import synth

RNG = np.random.default_rng(12345)


# ---- GEMV (§3.1 data movement / §6.1 GEMV listing: one dot product per row) ----

def test_gemv_exact_rational_non_square():
    M, K = 5, 7
    W = RNG.standard_normal((M, K)).astype(np.float32)
    x = RNG.standard_normal(K)
    y = oracle.gemv(W, x)
    for i in range(M):
        exact = sum(Fraction(float(W[i, j])) * Fraction(float(x[j])) for j in range(K))
        bound = K * 2.0 ** -52 * sum(abs(float(W[i, j]) * x[j]) for j in range(K))
        assert abs(Fraction(y[i]) - exact) <= Fraction(bound)


def test_gemv_identity_and_one_hot_rows_are_exact():
    K = 37
    x = RNG.standard_normal(K)
    assert np.array_equal(oracle.gemv(np.eye(K, dtype=np.float32), x), x)
    perm = RNG.permutation(K)[:11]
    W = np.zeros((11, K), dtype=np.float32)
    W[np.arange(11), perm] = 1.0
    assert np.array_equal(oracle.gemv(W, x), x[perm])


def test_gemv_ones_gives_row_sums():
    W = RNG.standard_normal((9, 301)).astype(np.float32)
    y = oracle.gemv(W, np.ones(301))
    for i in range(9):
        exact = math.fsum(float(v) for v in W[i])
        assert abs(y[i] - exact) <= 301 * 2 ** -52 * float(np.abs(W[i]).sum())


def test_gemv_float_accumulator_within_recursive_sum_bound():
    W = RNG.standard_normal((6, 4096)).astype(np.float32)
    x = RNG.standard_normal(4096).astype(np.float32)
    y32 = oracle.gemv(W, x, acc_bits=32)
    for i in range(6):
        exact = math.fsum(float(W[i, j]) * float(x[j]) for j in range(4096))
        bound = 4096 * 2.0 ** -24 * float(np.abs(W[i].astype(np.float64) * x).sum())
        assert abs(float(y32[i]) - exact) <= bound


# ---- RMSNorm (§2.1, §11.2 listing: ss/n + 1e-5, 1/sqrt, then (x*g)*r) ----------

def test_rmsnorm_unit_gain_rms_closed_form():
    x = RNG.standard_normal(768) * 3.0
    out = oracle.rmsnorm(x, np.ones(768, np.float32), 1e-5)
    m = float(np.mean(x * x))
    assert abs(math.sqrt(float(np.mean(out * out))) - math.sqrt(m / (m + 1e-5))) < 1e-12


def test_rmsnorm_constant_vector_places_epsilon_inside_sqrt_after_mean():
    # x = c * 1 gives out = c * g / sqrt(c^2 + eps); with c^2 ~ eps every other
    # placement of eps (outside the sqrt, or added before dividing by n) differs.
    c, n, eps = 0.003, 64, 1e-5
    g = (1.0 + 0.5 * RNG.standard_normal(n)).astype(np.float32)
    out = oracle.rmsnorm(np.full(n, c), g, eps)
    expect = c * g.astype(np.float64) / math.sqrt(c * c + eps)
    assert np.allclose(out, expect, rtol=1e-13, atol=0)


def test_rmsnorm_linear_in_gain():
    x = RNG.standard_normal(100)
    g = RNG.standard_normal(100).astype(np.float32)
    a = oracle.rmsnorm(x, g)
    b = oracle.rmsnorm(x, (4 * g).astype(np.float32))
    assert np.allclose(b, 4 * a, rtol=1e-15, atol=0)


# ---- RoPE (§2.1: rotate q and k in the complex plane; Su et al.) --------------

def test_rope_position_zero_is_identity():
    v = RNG.standard_normal(96)
    assert np.array_equal(oracle.rope(v, 48, 0), v)


def test_rope_preserves_every_pair_norm():
    v = RNG.standard_normal(128)
    r = oracle.rope(v, 64, 517)
    assert np.allclose(np.hypot(r[0::2], r[1::2]), np.hypot(v[0::2], v[1::2]), rtol=1e-14)


def test_rope_first_pair_turns_by_pos_radians_counterclockwise():
    r = oracle.rope(np.array([1.0, 0.0]), 2, 3)
    assert abs(r[0] - math.cos(3.0)) < 1e-15 and abs(r[1] - math.sin(3.0)) < 1e-15


def test_rope_pair_frequency_is_theta_to_minus_2i_over_hd():
    # head_dim 4: pair 1 turns by pos * 10000^(-2/4) = pos / 100 radians
    v = np.array([0.0, 0.0, 1.0, 0.0])
    r = oracle.rope(v, 4, 250)
    assert abs(r[2] - math.cos(2.5)) < 1e-15 and abs(r[3] - math.sin(2.5)) < 1e-15
    assert r[0] == 0.0 and r[1] == 0.0


def test_rope_every_head_uses_the_same_frequencies():
    v = np.tile(RNG.standard_normal(16), 3)
    r = oracle.rope(v, 16, 77)
    assert np.array_equal(r[:16], r[16:32]) and np.array_equal(r[:16], r[32:])


def test_rope_scores_depend_on_relative_position_only():
    q, k = RNG.standard_normal(64), RNG.standard_normal(64)
    m, n = 900, 333
    lhs = float(np.dot(oracle.rope(q, 64, m), oracle.rope(k, 64, n)))
    rhs = float(np.dot(oracle.rope(q, 64, m - n), k))
    assert abs(lhs - rhs) < 1e-11 * float(np.abs(q).sum() * np.abs(k).sum())


# ---- softmax, SiLU, attention ---------------------------------------------------

def test_softmax_sums_to_one_and_matches_closed_form():
    s = oracle.softmax(RNG.standard_normal(1000) * 20)
    assert abs(s.sum() - 1.0) < 1e-12
    w = oracle.softmax(np.array([7.0, 7.0 + math.log(3.0)]))
    assert abs(w[0] - 0.25) < 1e-15 and abs(w[1] - 0.75) < 1e-15


def test_silu_closed_forms():
    assert oracle.silu(0.0) == 0.0
    assert abs(oracle.silu(40.0) - 40.0) < 1e-12
    assert abs(oracle.silu(-40.0)) < 1e-15
    for z in (0.3, 1.7, 5.0):  # z*s(z) - (-z)*s(-z) = z since s(z) + s(-z) = 1
        assert abs(oracle.silu(z) - oracle.silu(-z) - z) < 1e-15


def test_attention_single_position_returns_v():
    q = RNG.standard_normal(64)
    K = RNG.standard_normal((1, 64))
    V = RNG.standard_normal((1, 64))
    assert np.array_equal(oracle.attention_head(q, K, V), V[0])


def test_attention_equal_keys_average_values():
    q = RNG.standard_normal(32)
    K = np.tile(RNG.standard_normal(32), (9, 1))
    V = RNG.standard_normal((9, 32))
    assert np.allclose(oracle.attention_head(q, K, V), V.mean(axis=0), rtol=0, atol=1e-14)


def test_attention_scale_is_one_over_sqrt_head_dim():
    # hd = 4: q.k1 / sqrt(4) = ln 3, q.k0 = 0  ->  weights 1/4 and 3/4
    q = np.array([1.0, 0.0, 0.0, 0.0])
    K = np.array([[0.0, 0, 0, 0], [2 * math.log(3.0), 0, 0, 0]])
    V = RNG.standard_normal((2, 4))
    out = oracle.attention_head(q, K, V)
    assert np.allclose(out, 0.25 * V[0] + 0.75 * V[1], rtol=0, atol=1e-14)


# ---- layout and model ------------------------------------------------------------

def test_blob_sizes_match_published_parameter_counts():
    # 110M tied: 109,529,856 parameters; Llama-2-7B (untied): 6,738,415,616.
    assert oracle.blob_bytes(synth.model_config("110m"), True) == 4 * 109_529_856
    assert oracle.blob_bytes(synth.model_config("7b"), False) == 4 * 6_738_415_616
    for name in ("tiny", "110m", "7b"):
        cfg = synth.model_config(name)
        for tied in (False, True):
            assert oracle.blob_bytes(cfg, tied) == synth.blob_bytes(cfg, tied)


def test_layout_offsets_agree_with_generator_on_padded_shapes():
    cfg = dict(dim=12, hidden_dim=10, n_layers=2, n_heads=3, n_kv_heads=1, vocab_size=7,
               max_seq=5)
    names = ["E", "g_att", "Wq", "Wk", "Wv", "Wo", "g_ffn", "W1", "W3", "W2", "g_final",
             "Wcls"]
    ents, total = synth.layout(cfg, tied=False)
    assert total == oracle.blob_bytes(cfg, False)
    for (name, layer, off, shape, kind) in ents:
        assert off % 128 == 0
        assert oracle.tensor_offset(cfg, False, names.index(name), max(layer, 0)) == off


def _tiny_cfg(**kw):
    cfg = dict(dim=4, hidden_dim=1, n_layers=1, n_heads=1, n_kv_heads=1, vocab_size=4,
               max_seq=4, rope_theta=10000.0, norm_eps=1e-5, shared_classifier=0)
    cfg.update(kw)
    return cfg


def _blob(cfg, **tensors):
    """A blob of zeros with the named tensors set; gains default to 1."""
    ents, total = synth.layout(cfg)
    b = np.zeros(total // 4, dtype=np.float32)
    for (name, layer, off, shape, kind) in ents:
        n = int(np.prod(shape))
        if kind == "gain":
            b[off // 4: off // 4 + n] = 1.0
        key = name if layer < 0 else f"{name}{layer}"
        if key in tensors:
            b[off // 4: off // 4 + n] = np.asarray(tensors[key], np.float32).ravel()
    return b


def test_swiglu_gates_w1_and_scales_by_w3_then_w2_adds_to_residual():
    # d = 4, F = 1, attention output zero. x0 = c*1 so xb ~ g_ffn = (1,0,0,0)*2;
    # W1 picks 15 * xb0 = 30, W3 picks 0.25 * xb0 = 0.5: h = silu(30) * 0.5 = 15
    # (the swapped gate would give silu(0.5) * 30 = 9.3). W2 adds h to x[0];
    # with Wcls = I the logits are rmsnorm(x1) and logit0/logit1 = (c + h) / c.
    c = 10.0
    cfg = _tiny_cfg()
    E = np.full((4, 4), c, np.float32)
    blob = _blob(cfg, E=E, g_ffn0=[2.0, 0, 0, 0], W10=[[15.0, 0, 0, 0]], W30=[[0.25, 0, 0, 0]],
                 W20=[[1.0], [0], [0], [0]], Wcls=np.eye(4))
    lg = oracle.Model(cfg, blob).forward(2, 0)
    h = c * (lg[0] / lg[1] - 1.0)
    kappa = 2 * c / math.sqrt(c * c + 1e-5)  # xb0 = c * 2 / sqrt(c^2 + eps)
    assert abs(h - 15.0 * kappa * 0.25 * kappa) < 1e-9 * 15  # silu(30) = 30 to 1e-12
    assert abs(lg[2] - lg[1]) < 1e-15 and abs(lg[3] - lg[1]) < 1e-15


def test_kv_cache_attention_averages_all_positions_up_to_current():
    # Wq = Wk = 0: equal scores, so attention at pos 1 averages v0 and v1.
    # E[0] = (c,0,0,0), E[1] = (0,c,0,0): xb = 2*e_0 and 2*e_1; Wv = Wo = I.
    # x1 at pos 1 = (0,c,0,0) + (1,1,0,0), and Wcls = I shows its direction.
    c = 10.0
    cfg = _tiny_cfg()
    E = np.zeros((4, 4), np.float32)
    E[0, 0] = c
    E[1, 1] = c
    blob = _blob(cfg, E=E, Wv0=np.eye(4), Wo0=np.eye(4), Wcls=np.eye(4))
    m = oracle.Model(cfg, blob)
    lg0 = m.forward(0, 0)
    assert lg0[1] == 0.0 and lg0[0] > 0  # pos 0: x1 = (c+2, 0, 0, 0)
    lg1 = m.forward(1, 1)
    r = 2 * c / math.sqrt(c * c + 4e-5)  # 2 * rmsnorm scale of a one-hot of size c
    assert abs(lg1[0] / lg1[1] - (r / 2) / (c + r / 2)) < 1e-12
    # re-running position 1 with the same token gives the same logits
    assert np.array_equal(m.forward(1, 1), lg1)


def _unit_kappa(c: float, d: int, eps: float = 1e-5) -> float:
    """RMSNorm output of a one-hot row c * e_t with unit gain: kappa * e_t."""
    return c * (1.0 / math.sqrt(c * c / d + eps))


def test_rope_turns_q_and_k_at_their_own_positions_and_leaves_v_alone():
    # §2.1: RoPE rotates q and k (not v), and the cached key of position 0 keeps
    # the rotation of position 0. One head of width 4; pair (0, 1) turns by p
    # radians at position p. Token 2 at position 0, token 3 at position 1, each
    # embedding a one-hot row, so x_b = kappa * e_t:
    #   q(pos 1) = kappa*qa*e0, turned by 1 -> kappa*qa*(cos 1, sin 1)
    #   k(pos 0) = kappa*kb*e0 (angle 0),  k(pos 1) = kappa*kb*e1 turned by 1
    #   v(pos 0) = kappa*gv*e0,            v(pos 1) = kappa*gv*e1 (never turned)
    # Scores: s0 = kappa^2 qa kb cos(1) / 2 and s1 = 0 (q and k(pos 1) turn by
    # the same angle and start orthogonal). With Wo = I, zero FFN and Wcls = I,
    # the logits are proportional to x = (kappa gv w0, kappa gv w1, 0, c).
    # A key cached before its rotation, a key turned at the reader's position,
    # no rotation at all, or a rotated v each change lg0 / lg1 = w0 / w1.
    c, qa, kb, gv = 10.0, 0.5, 1.0, 1.0
    cfg = _tiny_cfg()
    E = np.zeros((4, 4), np.float32)
    E[2, 2] = c
    E[3, 3] = c
    Wq = np.zeros((4, 4), np.float32)
    Wq[0, 3] = qa
    Wk = np.zeros((4, 4), np.float32)
    Wk[0, 2] = kb
    Wk[1, 3] = kb
    Wv = np.zeros((4, 4), np.float32)
    Wv[0, 2] = gv
    Wv[1, 3] = gv
    blob = _blob(cfg, E=E, Wq0=Wq, Wk0=Wk, Wv0=Wv, Wo0=np.eye(4), Wcls=np.eye(4))
    m = oracle.Model(cfg, blob)
    kap = _unit_kappa(c, 4)
    lg0 = m.forward(2, 0)  # one position: the output is v(pos 0) itself
    assert abs(lg0[0] / lg0[2] - kap * gv / c) < 1e-12 and lg0[1] == 0.0 and lg0[3] == 0.0
    lg = m.forward(3, 1)
    s0 = (kap * qa) * (kap * kb) * math.cos(1.0) / 2.0
    w0 = 1.0 / (1.0 + math.exp(-s0))
    w1 = 1.0 - w0
    assert abs(lg[0] / lg[1] - w0 / w1) < 1e-12 * (w0 / w1)
    assert abs(lg[0] / lg[3] - kap * gv * w0 / c) < 1e-12
    assert lg[2] == 0.0


def test_each_head_reads_its_own_q_k_v_slices_and_writes_its_own_output():
    # Two heads of width 2 (H = Hkv = 2): head h reads q, k, v elements
    # [2h, 2h + 2) and writes o elements [2h, 2h + 2). Token 0 at position 0,
    # token 1 at position 1, one-hot embeddings (x_b = kappa * e_t).
    #   head 0: q = kappa*Qw*(1, 0), head 1: q = -0.75*kappa*Qw*(1, 0) (pos 1)
    #   both heads: k(pos 0) = kappa*kw*(1, 0), k(pos 1) = kappa*Kw*(1, 0)
    #   v(pos 0) = kappa*gw*e3 (head 1's slice), v(pos 1) = kappa*gw*e0 (head 0's)
    # Head 0 leans to position 1, head 1 to position 0 (its q points the other
    # way), so o = (kappa gw w1[0], 0, 0, kappa gw w0[1]) with w the softmax
    # weights of each head; q, k turn by the same angle at position 1 and k of
    # position 0 not at all, so s0 = a * kw * cos(1) / sqrt(2), s1 = a * Kw / sqrt(2)
    # with a = the head's q length times kappa. Heads reading head 0's q, one
    # kv head for all, or outputs written to the wrong slice break lg3/lg1 or lg2.
    c, Qw, kw, Kw, gw = 10.0, 1.0, 0.5, 1.0, 1.0
    cfg = _tiny_cfg(n_heads=2, n_kv_heads=2)
    E = np.zeros((4, 4), np.float32)
    E[0, 0] = c
    E[1, 1] = c
    Wq = np.zeros((4, 4), np.float32)
    Wq[0, 1] = Qw
    Wq[2, 1] = -0.75 * Qw
    Wk = np.zeros((4, 4), np.float32)
    Wk[0, 0] = kw
    Wk[2, 0] = kw
    Wk[0, 1] = Kw
    Wk[2, 1] = Kw
    Wv = np.zeros((4, 4), np.float32)
    Wv[3, 0] = gw
    Wv[0, 1] = gw
    blob = _blob(cfg, E=E, Wq0=Wq, Wk0=Wk, Wv0=Wv, Wo0=np.eye(4), Wcls=np.eye(4))
    m = oracle.Model(cfg, blob)
    kap = _unit_kappa(c, 4)
    lg0 = m.forward(0, 0)  # one position: head 1's output is its slice of v(pos 0)
    assert abs(lg0[3] / lg0[0] - kap * gw / c) < 1e-12 and lg0[1] == 0.0 and lg0[2] == 0.0
    lg = m.forward(1, 1)

    def weights(qlen):
        a = kap * qlen * kap
        s0 = a * kw * math.cos(1.0) / math.sqrt(2.0)
        s1 = a * Kw / math.sqrt(2.0)
        w1 = 1.0 / (1.0 + math.exp(s0 - s1))
        return 1.0 - w1, w1

    _, w1_h0 = weights(Qw)
    w0_h1, _ = weights(-0.75 * Qw)
    assert w1_h0 > 0.8 and w0_h1 > 0.7  # the heads lean to different positions
    assert abs(lg[0] / lg[1] - kap * gw * w1_h0 / c) < 1e-12
    assert abs(lg[3] / lg[1] - kap * gw * w0_h1 / c) < 1e-12
    assert lg[2] == 0.0


def test_zero_output_projections_make_the_layer_an_identity():
    cfg1 = dict(synth.model_config("tiny"), n_layers=1, vocab_size=512)
    blob1 = synth.make_blob(cfg1, seed=7)
    for nm in ("Wo", "W2"):
        synth.tensor(blob1, cfg1, nm, 0)[...] = 0.0
    cfg0 = dict(cfg1, n_layers=0)
    blob0 = np.zeros(synth.blob_bytes(cfg0) // 4, np.float32)
    for nm in ("E", "g_final", "Wcls"):
        synth.tensor(blob0, cfg0, nm)[...] = synth.tensor(blob1, cfg1, nm)
    a = oracle.Model(cfg1, blob1).forward(5, 0)
    b = oracle.Model(cfg0, blob0).forward(5, 0)
    assert np.array_equal(a, b)


def test_zero_layers_tied_unit_gain_logit_closed_form_and_argmax():
    cfg = dict(synth.model_config("tiny"), n_layers=0, vocab_size=2000, shared_classifier=1)
    blob = synth.make_blob(cfg, seed=11)
    synth.tensor(blob, cfg, "g_final")[...] = 1.0
    E = synth.tensor(blob, cfg, "E").astype(np.float64)
    m = oracle.Model(cfg, blob)
    for t in (0, 17, 1999):
        lg = m.forward(t, 0)
        n2 = math.fsum(E[t] * E[t])
        assert abs(lg[t] - n2 / math.sqrt(n2 / cfg["dim"] + 1e-5)) < 1e-12 * n2
        assert int(np.argmax(lg)) == t


def test_grouped_query_heads_equal_duplicated_multi_head_model():
    # Hkv = H/2: query head h reads kv head h // 2. The same model with Wk, Wv
    # rows duplicated per group and Hkv = H must give identical logits.
    cfg_g = dict(dim=32, hidden_dim=48, n_layers=2, n_heads=4, n_kv_heads=2, vocab_size=64,
                 max_seq=8, rope_theta=10000.0, norm_eps=1e-5, shared_classifier=0)
    cfg_m = dict(cfg_g, n_kv_heads=4)
    bg = synth.make_blob(cfg_g, seed=3)
    bm = np.zeros(synth.blob_bytes(cfg_m) // 4, np.float32)
    hd = 8
    for (name, layer, off, shape, kind) in synth.layout(cfg_m)[0]:
        src = synth.tensor(bg, cfg_g, name, layer)
        dst = synth.tensor(bm, cfg_m, name, layer)
        if name in ("Wk", "Wv"):
            for h in range(4):
                dst[h * hd:(h + 1) * hd] = src[(h // 2) * hd:(h // 2 + 1) * hd]
        else:
            dst[...] = src
    mg, mm = oracle.Model(cfg_g, bg), oracle.Model(cfg_m, bm)
    tok = [3, 9, 27, 50, 1]
    for p, t in enumerate(tok):
        assert np.array_equal(mg.forward(t, p), mm.forward(t, p))


def test_tying_heuristic_infers_from_blob_size():
    cfg = dict(synth.model_config("tiny"), n_layers=1, vocab_size=300, shared_classifier=-1)
    short = synth.make_blob(cfg, seed=1, tied=True)
    full = synth.make_blob(cfg, seed=1, tied=False)
    assert oracle.Model(cfg, short).tied is True
    assert oracle.Model(cfg, full).tied is False
    with pytest.raises(ValueError):
        oracle.Model(cfg, full[:-32])


def test_out_of_range_token_and_position_are_rejected():
    cfg = dict(synth.model_config("tiny"), n_layers=1, vocab_size=100, max_seq=4)
    m = oracle.Model(cfg, synth.make_blob(cfg, seed=1))
    for tok, pos in ((100, 0), (-1, 0), (0, 4), (0, -1)):
        with pytest.raises(ValueError):
            m.forward(tok, pos)


def test_float_and_double_oracles_agree_within_decode_tolerances():
    cfg = synth.model_config("tiny")
    blob = synth.make_blob(cfg)
    t64, l64 = oracle.Model(cfg, blob, 64).greedy(1, 24)
    m32 = oracle.Model(cfg, blob, 32)
    for p, (t, ref) in enumerate(zip(t64, l64)):
        got = m32.forward(t, p)  # teacher forcing with the double oracle's tokens
        assert np.abs(got - ref).max() <= 2e-3 * np.abs(ref).max()
        top2 = np.sort(ref)[-2:]
        if top2[1] - top2[0] > 1e-2:
            assert int(np.argmax(got)) == int(np.argmax(ref))


# ---- weight-only 8-bit codes (the paper's quantization future work, read as
# per-row symmetric 8-bit codes: s = max|w| / 127, q = nearest(w / s), ties to even) ----

def test_q8_integer_rows_with_max_127_keep_their_values_and_round_ties_to_even():
    W = np.array([[127, 0.5, 1.5, 2.5, -0.5, -1.5, 3.5, -2.5, -127, 64]], np.float32)
    q, s = oracle.quantize_rows_q8(W)
    assert s[0] == np.float32(1.0)
    assert q.tolist() == [[127, 0, 2, 2, 0, -2, 4, -2, -127, 64]]


def test_q8_zero_row_sign_symmetry_and_power_of_two_scaling():
    W = RNG.standard_normal((9, 33)).astype(np.float32)
    W[4] = 0.0
    q, s = oracle.quantize_rows_q8(W)
    assert s[4] == 0.0 and not q[4].any()
    qn, sn = oracle.quantize_rows_q8(-W)
    assert np.array_equal(qn, -q) and np.array_equal(sn, s)
    q8, s8 = oracle.quantize_rows_q8(W * np.float32(8.0))  # exact in float32
    assert np.array_equal(q8, q) and np.array_equal(s8, s * np.float32(8.0))


def test_q8_codes_reach_127_at_the_row_maximum_and_stay_within_half_a_step():
    W = (RNG.standard_normal((40, 200)) * 0.02).astype(np.float32)
    q, s = oracle.quantize_rows_q8(W)
    for i in range(40):
        j = int(np.argmax(np.abs(W[i])))
        assert abs(int(q[i, j])) == 127
        assert np.abs(q[i]).max() == 127
        err = np.abs(W[i].astype(np.float64) - float(s[i]) * q[i].astype(np.float64))
        assert err.max() <= 0.5 * float(s[i]) * (1 + 1e-6)  # nearest code, float32 division
    assert float(s[0]) == float(np.float32(np.abs(W[0]).max()) / np.float32(127.0))


def test_q8_gemv_is_the_gemv_of_the_weights_the_codes_stand_for():
    q = RNG.integers(-127, 128, size=(7, 13)).astype(np.int8)
    s = (RNG.random(7) * 0.01).astype(np.float32)
    x = RNG.standard_normal(13)
    y = oracle.gemv_q8(q, s, x)
    for i in range(7):
        exact = sum(Fraction(float(s[i])) * int(q[i, j]) * Fraction(float(x[j])) for j in range(13))
        bound = 13 * 2.0 ** -51 * sum(abs(float(s[i]) * int(q[i, j]) * x[j]) for j in range(13))
        assert abs(Fraction(y[i]) - exact) <= Fraction(bound)
    eye = np.eye(13, dtype=np.int8) * 127
    assert np.allclose(oracle.gemv_q8(eye, np.full(13, 1 / 127, np.float32), x),
                       x * 127 * float(np.float32(1 / 127)), rtol=0, atol=1e-15)


# ---- weight-only 4-bit codes (the same definition with 7 levels on each side
# of zero: s = max|w| / 7, q = nearest(w / s), ties to even, in [-7, 7]) ----

def test_q4_integer_rows_with_max_7_keep_their_values_and_round_ties_to_even():
    W = np.array([[7, 0.5, 1.5, 2.5, -0.5, -1.5, 3.5, -2.5, -7, 4, 6.5, -5.5]], np.float32)
    q, s = oracle.quantize_rows_q4(W)
    assert s[0] == np.float32(1.0)
    assert q.tolist() == [[7, 0, 2, 2, 0, -2, 4, -2, -7, 4, 6, -6]]


def test_q4_codes_reach_7_at_the_row_maximum_and_stay_within_half_a_step():
    W = (RNG.standard_normal((40, 256)) * 0.02).astype(np.float32)
    q, s = oracle.quantize_rows_q4(W)
    assert np.abs(q).max() == 7
    for i in range(40):
        j = int(np.argmax(np.abs(W[i])))
        assert abs(int(q[i, j])) == 7
        err = np.abs(W[i].astype(np.float64) - float(s[i]) * q[i].astype(np.float64))
        assert err.max() <= 0.5 * float(s[i]) * (1 + 1e-6)  # nearest level, float32 division
    assert float(s[0]) == float(np.float32(np.abs(W[0]).max()) / np.float32(7.0))


def test_q4_zero_row_sign_symmetry_and_power_of_two_scaling():
    W = RNG.standard_normal((9, 64)).astype(np.float32)
    W[4] = 0.0
    q, s = oracle.quantize_rows_q4(W)
    assert s[4] == 0.0 and not q[4].any()
    qn, sn = oracle.quantize_rows_q4(-W)
    assert np.array_equal(qn, -q) and np.array_equal(sn, s)
    q2, s2 = oracle.quantize_rows_q4(W * np.float32(8.0))  # exact in float32
    assert np.array_equal(q2, q) and np.array_equal(s2, s * np.float32(8.0))


def test_q4_code_is_the_nearest_of_the_15_levels_by_brute_force():
    W = (RNG.standard_normal((6, 50)) * 0.02).astype(np.float32)
    q, s = oracle.quantize_rows_q4(W)
    for i in range(6):
        levels = np.arange(-7, 8, dtype=np.float64) * float(s[i])
        for j in range(50):
            d = np.abs(levels - float(W[i, j]))
            assert d[int(q[i, j]) + 7] <= d.min() * (1 + 1e-6) + 1e-15


def _representable_blob(cfg, seed, kmax=127):
    """A blob whose every weight matrix row is k * 2^-12 with integer |k| <= kmax
    and some |k| == kmax: its codes with kmax levels and its scales are exact."""
    blob = synth.make_blob(cfg, seed=seed)
    names = ["Wq", "Wk", "Wv", "Wo", "W1", "W3", "W2"]
    mats = [("E", -1)] + [(n, l) for l in range(cfg["n_layers"]) for n in names]
    if not cfg["shared_classifier"]:
        mats.append(("Wcls", -1))
    for (n, l) in mats:
        T = synth.tensor(blob, cfg, n, l)
        k = np.clip(np.rint(T * 4096.0 * kmax / 127), -kmax, kmax)
        k[:, 0] = np.where(k[:, 0] < 0, -kmax, kmax)
        T[...] = (k / 4096.0).astype(np.float32)
    return blob


@pytest.mark.parametrize("tied", [1, 0])
def test_q8_model_equals_float_model_on_exactly_representable_weights(tied):
    cfg = dict(synth.model_config("tiny"), n_layers=2, vocab_size=500, max_seq=8,
               shared_classifier=tied)
    blob = _representable_blob(cfg, 5)
    mf = oracle.Model(cfg, blob)
    mq = oracle.Model(cfg, blob, weight_bits=8)
    for pos, tok in enumerate([3, 17, 499, 0, 250]):
        assert np.array_equal(mq.forward(tok, pos), mf.forward(tok, pos))


def test_q8_model_differs_from_float_model_by_quantization_only():
    cfg = dict(synth.model_config("tiny"), n_layers=2, vocab_size=500, max_seq=8)
    blob = synth.make_blob(cfg, seed=6)
    lf = oracle.Model(cfg, blob).forward(1, 0)
    lq = oracle.Model(cfg, blob, weight_bits=8).forward(1, 0)
    rel = np.abs(lq - lf).max() / np.abs(lf).max()
    assert 1e-5 < rel < 5e-2  # the codes change the result, by about the code step


@pytest.mark.parametrize("tied", [1, 0])
def test_q4_model_equals_float_model_on_exactly_representable_weights(tied):
    cfg = dict(synth.model_config("tiny"), n_layers=2, vocab_size=500, max_seq=8,
               shared_classifier=tied)
    blob = _representable_blob(cfg, 7, kmax=7)
    mf = oracle.Model(cfg, blob)
    mq = oracle.Model(cfg, blob, weight_bits=4)
    for pos, tok in enumerate([3, 17, 499, 0, 250]):
        assert np.array_equal(mq.forward(tok, pos), mf.forward(tok, pos))


def test_q4_model_is_coarser_than_q8_and_differs_by_quantization_only():
    cfg = dict(synth.model_config("tiny"), n_layers=2, vocab_size=500, max_seq=8)
    blob = synth.make_blob(cfg, seed=6)
    lf = oracle.Model(cfg, blob).forward(1, 0)
    l8 = oracle.Model(cfg, blob, weight_bits=8).forward(1, 0)
    l4 = oracle.Model(cfg, blob, weight_bits=4).forward(1, 0)
    r8 = np.abs(l8 - lf).max() / np.abs(lf).max()
    r4 = np.abs(l4 - lf).max() / np.abs(lf).max()
    assert 4 * r8 < r4 < 1.0  # 15 levels instead of 255: a far larger code step
    with pytest.raises(ValueError):
        oracle.Model(cfg, blob, weight_bits=5)
