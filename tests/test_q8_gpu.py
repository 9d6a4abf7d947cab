"""Weight-only 8-bit rows on the GPU: the codes against the oracle's (bit for
bit: every decision is taken in float32 on both sides), and tvl_gemv_q8
against the oracle's GEMV of the weights the codes stand for."""
import numpy as np
import pytest

import oracle
from helpers import gemv_bound
from paper_2601_03324_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def tvl():
    from paper_2601_03324_gb300 import tvl as t
    return t


def quantize_gpu(tvl, W):
    M, K = W.shape
    dW = torch.from_numpy(np.ascontiguousarray(W)).cuda()
    buf = torch.empty(tvl.tvl_q8_bytes(M, K), dtype=torch.uint8, device="cuda")
    tvl.tvl_quantize_q8(dW.data_ptr(), buf.data_ptr(), M, K)
    torch.cuda.synchronize()
    rows = buf.cpu().numpy().reshape(M, 16 + K)
    s = rows[:, :4].copy().view(np.float32).reshape(M)
    pad = rows[:, 4:16]
    q = rows[:, 16:].view(np.int8)
    return buf, q, s, pad


def tie_matrix():
    W = np.zeros((4, 32), np.float32)
    W[0, :8] = [127, 0.5, 1.5, 2.5, -0.5, -1.5, 3.5, -2.5]
    W[1] = np.arange(32, dtype=np.float32) - 15.5  # halves everywhere, max 16 -> scale 16/127
    W[2] = 0.0
    W[3, 5] = -3.0
    return W


SHAPES = [(768, 768), (2048, 768), (300, 288), (5, 4096), (4096, 11008), (32000, 768), (3, 16)]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"{s[0]}x{s[1]}")
def test_codes_and_scales_match_the_oracle_bit_for_bit(tvl, shape):
    W, _ = synth.gemv_operands(*shape, 4)
    _, q, s, pad = quantize_gpu(tvl, W)
    q_ref, s_ref = oracle.quantize_rows_q8(W)
    assert np.array_equal(s.view(np.uint32), s_ref.view(np.uint32))
    assert np.array_equal(q, q_ref)
    assert not pad.any()


def test_ties_and_zero_rows(tvl):
    W = tie_matrix()
    _, q, s, _ = quantize_gpu(tvl, W)
    q_ref, s_ref = oracle.quantize_rows_q8(W)
    assert np.array_equal(q, q_ref) and np.array_equal(s.view(np.uint32), s_ref.view(np.uint32))
    assert q[0, :8].tolist() == [127, 0, 2, 2, 0, -2, 4, -2]
    assert s[2] == 0.0 and not q[2].any()


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"{s[0]}x{s[1]}")
def test_gemv_q8_matches_the_oracle(tvl, shape):
    M, K = shape
    W, x = synth.gemv_operands(M, K, 5)
    buf, q, s, _ = quantize_gpu(tvl, W)
    dx = torch.from_numpy(x).cuda()
    y = torch.full((M,), float("nan"), device="cuda")
    tvl.tvl_gemv_q8(buf.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K)
    torch.cuda.synchronize()
    got = y.cpu().numpy()
    ref = oracle.gemv_q8(q, s, x)
    Wd = (s[:, None].astype(np.float64) * q.astype(np.float64))
    assert np.all(np.abs(got - ref) <= gemv_bound(Wd, x)), float(np.abs(got - ref).max())


def test_gemv_q8_rejects_bad_shapes(tvl):
    d = torch.zeros(4096, device="cuda")
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_q8(d.data_ptr(), d.data_ptr(), d.data_ptr(), 4, 24)   # 24 % 16 != 0
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_q8(d.data_ptr() + 4, d.data_ptr(), d.data_ptr(), 4, 32)  # misaligned
    with pytest.raises(tvl.TvlError):
        tvl.tvl_quantize_q8(d.data_ptr(), d.data_ptr(), 4, 8)


# ---- decode with 8-bit weight rows (tvl_config.weight_bits = 8) vs the oracle's
# model over the same codes; tolerances as for the float32 decode ----

from helpers import compare_greedy, lockstep_greedy, small_config  # noqa: E402


def check_q8_model(tvl, cfg, blob, n_steps, start=1, check_every=1, label=""):
    cfg = dict(cfg, weight_bits=8)
    ref = oracle.Model(cfg, blob, 64, weight_bits=8)
    with tvl.Model(cfg, blob) as m:
        toks, ref_logits, worst = lockstep_greedy(m, ref, start, n_steps,
                                                  check_every=check_every, label=label)
        gen = m.decode_greedy(start, 0, n_steps)
        compare_greedy(gen, toks[1:] + [int(np.argmax(ref_logits[-1]))], ref_logits)
    return worst


def test_q8_tiny_model_64_steps(tvl):
    cfg = synth.model_config("tiny")
    check_q8_model(tvl, cfg, synth.make_blob(cfg), cfg["steps"], label="tiny q8")


@pytest.mark.parametrize("kw", [
    dict(),
    dict(n_kv_heads=2),
    dict(n_layers=0, shared_classifier=1),
    dict(dim=128, n_heads=1, n_kv_heads=1, hidden_dim=256, shared_classifier=1),
], ids=["base", "gqa2", "L0_tied", "hd128_tied"])
def test_q8_small_shapes_match_oracle(tvl, kw):
    cfg = small_config(**kw)
    check_q8_model(tvl, cfg, synth.make_blob(cfg, seed=23), cfg["max_seq"], label=f"q8 {kw}")


def test_q8_110m_64_steps(tvl):
    cfg = synth.model_config("110m")
    check_q8_model(tvl, cfg, synth.make_blob(cfg), 64, check_every=8, label="110m q8")


def test_q8_streams_a_quarter_of_the_float_bytes(tvl):
    cfg = synth.model_config("110m")
    blob = synth.make_blob(cfg)
    with tvl.Model(cfg, blob) as mf, tvl.Model(dict(cfg, weight_bits=8), blob) as mq:
        sf, sq = mf.info().streamed_bytes, mq.info().streamed_bytes
    d, F, L, V = cfg["dim"], cfg["hidden_dim"], cfg["n_layers"], cfg["vocab_size"]
    expect = L * ((3 * d) * (16 + d) + d * (16 + d) + 2 * F * (16 + d) + d * (16 + F) + 8 * d) \
        + V * (16 + d) + (16 + d) + 4 * d
    assert sq == expect and 0.24 < sq / sf < 0.27
