"""Weight-only 4-bit rows on the GPU: the packed codes against the oracle's
(bit for bit: every decision is taken in float32 on both sides, and the
nibble order is the one include/tvl.h states), and tvl_gemv_q4 against the
oracle's GEMV of the weights the codes stand for."""
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
    """Packed rows from the GPU, unpacked: (device buffer, codes int8 [M, K], scales, pad)."""
    M, K = W.shape
    dW = torch.from_numpy(np.ascontiguousarray(W)).cuda()
    nbytes = tvl.tvl_q4_bytes(M, K)
    assert nbytes == M * (16 + K // 2)
    buf = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    tvl.tvl_quantize_q4(dW.data_ptr(), buf.data_ptr(), M, K)
    torch.cuda.synchronize()
    rows = buf.cpu().numpy().reshape(M, 16 + K // 2)
    s = rows[:, :4].copy().view(np.float32).reshape(M)
    pad = rows[:, 4:16]
    packed = rows[:, 16:]
    lo = (packed & 0xF).astype(np.int8)
    hi = (packed >> 4).astype(np.int8)
    q = np.empty((M, K), np.int8)
    q[:, 0::2] = np.where(lo > 7, lo - 16, lo)  # 4-bit two's complement, even column low
    q[:, 1::2] = np.where(hi > 7, hi - 16, hi)
    return buf, q, s, pad


SHAPES = [(768, 768), (2048, 768), (300, 288), (5, 4096), (4096, 11008), (32000, 768), (3, 32)]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"{s[0]}x{s[1]}")
def test_codes_and_scales_match_the_oracle_bit_for_bit(tvl, shape):
    W, _ = synth.gemv_operands(*shape, 6)
    _, q, s, pad = quantize_gpu(tvl, W)
    q_ref, s_ref = oracle.quantize_rows_q4(W)
    assert np.array_equal(s.view(np.uint32), s_ref.view(np.uint32))
    assert np.array_equal(q, q_ref)
    assert not pad.any()


def test_ties_zero_rows_and_nibble_order(tvl):
    W = np.zeros((4, 32), np.float32)
    W[0, :12] = [7, 0.5, 1.5, 2.5, -0.5, -1.5, 3.5, -2.5, -7, 4, 6.5, -5.5]
    W[1] = (np.arange(32, dtype=np.float32) - 15.5) / 4  # quarter steps, max 3.875
    W[3, 5] = -3.0
    buf, q, s, _ = quantize_gpu(tvl, W)
    q_ref, s_ref = oracle.quantize_rows_q4(W)
    assert np.array_equal(q, q_ref) and np.array_equal(s.view(np.uint32), s_ref.view(np.uint32))
    assert q[0, :12].tolist() == [7, 0, 2, 2, 0, -2, 4, -2, -7, 4, 6, -6]
    assert s[2] == 0.0 and not q[2].any()
    raw = buf.cpu().numpy().reshape(4, 32)[:, 16:]
    assert raw[0, 0] == 0x07 and raw[0, 1] == 0x22  # columns 0 (low nibble) and 1; 2 and 3
    assert raw[3, 2] == 0x90  # column 5 = -7 (the row maximum) in the high nibble of byte 2


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: f"{s[0]}x{s[1]}")
def test_gemv_q4_matches_the_oracle(tvl, shape):
    M, K = shape
    W, x = synth.gemv_operands(M, K, 7)
    buf, q, s, _ = quantize_gpu(tvl, W)
    dx = torch.from_numpy(x).cuda()
    y = torch.full((M,), float("nan"), device="cuda")
    for _ in range(2):
        tvl.tvl_gemv_q4(buf.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K)
        torch.cuda.synchronize()
        got = y.cpu().numpy()
        ref = oracle.gemv_q8(q, s, x)  # the GEMV of the codes' weights (any code range)
        Wd = s[:, None].astype(np.float64) * q.astype(np.float64)
        assert np.all(np.abs(got - ref) <= gemv_bound(Wd, x)), float(np.abs(got - ref).max())


def test_q4_rejects_bad_shapes(tvl):
    d = torch.zeros(8192, device="cuda")
    assert tvl.tvl_q4_bytes(4, 48) == 0 and tvl.tvl_q4_bytes(0, 32) == 0
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_q4(d.data_ptr(), d.data_ptr(), d.data_ptr(), 4, 48)   # 48 % 32 != 0
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_q4(d.data_ptr() + 4, d.data_ptr(), d.data_ptr(), 4, 32)  # misaligned
    with pytest.raises(tvl.TvlError):
        tvl.tvl_quantize_q4(d.data_ptr(), d.data_ptr(), 4, 16)
    with pytest.raises(tvl.TvlError):
        tvl.tvl_gemv_q4(d.data_ptr(), d.data_ptr(), d.data_ptr(), 1, 32768)  # row over a stage


# ---- decode with 4-bit weight rows (tvl_config.weight_bits = 4) vs the oracle's
# model over the same codes; tolerances as for the float32 decode ----

from helpers import compare_greedy, lockstep_greedy, small_config  # noqa: E402


def check_q4_model(tvl, cfg, blob, n_steps, start=1, check_every=1, label=""):
    cfg = dict(cfg, weight_bits=4)
    ref = oracle.Model(cfg, blob, 64, weight_bits=4)
    with tvl.Model(cfg, blob) as m:
        toks, ref_logits, worst = lockstep_greedy(m, ref, start, n_steps,
                                                  check_every=check_every, label=label)
        gen = m.decode_greedy(start, 0, n_steps)
        compare_greedy(gen, toks[1:] + [int(np.argmax(ref_logits[-1]))], ref_logits)
    return worst


def test_q4_tiny_model_64_steps(tvl):
    cfg = synth.model_config("tiny")
    check_q4_model(tvl, cfg, synth.make_blob(cfg), cfg["steps"], label="tiny q4")


@pytest.mark.parametrize("kw", [
    dict(),
    dict(n_kv_heads=2),
    dict(n_layers=0, shared_classifier=1),
    dict(dim=128, n_heads=1, n_kv_heads=1, hidden_dim=256, shared_classifier=1),
], ids=["base", "gqa2", "L0_tied", "hd128_tied"])
def test_q4_small_shapes_match_oracle(tvl, kw):
    cfg = small_config(**kw)
    check_q4_model(tvl, cfg, synth.make_blob(cfg, seed=29), cfg["max_seq"], label=f"q4 {kw}")


def test_q4_110m_64_steps(tvl):
    cfg = synth.model_config("110m")
    check_q4_model(tvl, cfg, synth.make_blob(cfg), 64, check_every=8, label="110m q4")


def test_q4_streams_an_eighth_of_the_float_bytes(tvl):
    cfg = synth.model_config("110m")
    blob = synth.make_blob(cfg)
    with tvl.Model(cfg, blob) as mf, tvl.Model(dict(cfg, weight_bits=4), blob) as mq:
        sf, sq = mf.info().streamed_bytes, mq.info().streamed_bytes
    d, F, L, V = cfg["dim"], cfg["hidden_dim"], cfg["n_layers"], cfg["vocab_size"]
    rq, rf = 16 + d // 2, 16 + F // 2
    expect = L * ((3 * d) * rq + d * rq + 2 * F * rq + d * rf + 8 * d) + V * rq + rq + 4 * d
    assert sq == expect and 0.12 < sq / sf < 0.14
