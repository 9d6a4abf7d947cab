"""Batched decode on the GPU (B sequences per launch) vs B independent oracles.

Each sequence of a batch is an independent decode: sequence b is compared
with its own oracle model fed the same tokens, step by step (max |d logit| <=
2e-3 * max |logit|), and the device greedy loop of the batch must produce
each oracle's greedy tokens wherever that oracle's top-2 margin exceeds 1e-2.
"""
import numpy as np
import pytest

import oracle
from helpers import assert_logits_close, compare_greedy, small_config
from paper_2601_03324_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def tvl():
    from paper_2601_03324_gb300 import tvl as t
    return t


def batch_teacher_forced(m, refs, toks, start_pos=0, check_every=1, label=""):
    """toks [n, B]: step i feeds toks[i, b] to sequence b at start_pos + i."""
    n, B = toks.shape
    V = refs[0].vocab
    out = np.empty(B * V, np.float32)
    for i in range(n):
        p = start_pos + i
        m.forward_batch(toks[i], p, out)
        for b in range(B):
            lg = refs[b].forward(int(toks[i, b]), p)
            if i % check_every == 0 or i == n - 1:
                assert_logits_close(out[b * V:(b + 1) * V], lg, f"{label} b{b} pos {p}")


def batch_greedy_check(m, refs, starts, n_steps, start_pos=0, label=""):
    gen = m.decode_greedy_batch(starts, start_pos, n_steps)
    assert gen.shape == (n_steps, len(starts))
    for b, ref in enumerate(refs):
        toks, lgs = ref.greedy(int(starts[b]), n_steps, start_pos=start_pos)
        compare_greedy(gen[:, b], toks[1:] + [int(np.argmax(lgs[-1]))], lgs)
    return gen


@pytest.mark.parametrize("B", [2, 3, 4])
@pytest.mark.parametrize("kw", [
    dict(),                                   # several layers, multi-chunk attention
    dict(n_kv_heads=2),                       # grouped query heads
    dict(dim=96, n_heads=2, n_kv_heads=2, hidden_dim=8200, vocab_size=333),  # W2 rows: 2 stages
    dict(n_layers=0),                         # embedding -> final norm -> classifier
    dict(dim=2080, n_heads=65, n_kv_heads=65, hidden_dim=64, vocab_size=100, n_layers=1,
         max_seq=24),                         # W1/W3 row pair wider than a stage
], ids=["base", "gqa2", "wide_ffn", "L0", "pair_defer"])
def test_batch_teacher_forced_and_greedy(tvl, B, kw):
    cfg = small_config(max_batch=4, **kw)
    blob = synth.make_blob(cfg, seed=31)
    n = cfg["max_seq"]
    V = cfg["vocab_size"]
    toks = synth.uniform_ints(n * B, 17, B, 0, V - 1).reshape(n, B)
    with tvl.Model(cfg, blob) as m:
        assert m.info().max_batch == 4
        refs = [oracle.Model(cfg, blob, 64) for _ in range(B)]
        batch_teacher_forced(m, refs, toks, label=f"B{B} {kw}")
        refs = [oracle.Model(cfg, blob, 64) for _ in range(B)]
        batch_greedy_check(m, refs, toks[0], n, label=f"B{B} greedy")


def test_equal_sequences_give_equal_bits(tvl):
    """Sequences are independent: equal inputs give bit-equal logits and tokens."""
    cfg = small_config(max_batch=4)
    blob = synth.make_blob(cfg, seed=3)
    V = cfg["vocab_size"]
    with tvl.Model(cfg, blob) as m:
        out = np.empty(4 * V, np.float32)
        for p in range(6):
            m.forward_batch([5, 9, 5, 9], p, out)
            assert np.array_equal(out[:V], out[2 * V:3 * V])
            assert np.array_equal(out[V:2 * V], out[3 * V:])
        gen = m.decode_greedy_batch([7, 7, 7, 7], 0, 40)
        assert (gen == gen[:, :1]).all()


def test_slot0_is_shared_with_batch1_calls(tvl):
    """A batch's sequence 0 uses the cache of tvl_forward: a batch-of-2 prefix
    continued by batch-1 steps is still sequence 0 of the oracle."""
    cfg = small_config(max_batch=2)
    blob = synth.make_blob(cfg, seed=6)
    toks = synth.uniform_ints(40, 9, 0, 0, cfg["vocab_size"] - 1).reshape(20, 2)
    ref0 = oracle.Model(cfg, blob, 64)
    out1 = np.empty(cfg["vocab_size"], np.float32)
    with tvl.Model(cfg, blob) as m:
        for p in range(10):
            m.forward_batch(toks[p], p)
            ref0.forward(int(toks[p, 0]), p)
        for p in range(10, 20):
            m.forward(int(toks[p, 0]), p, out1)
            assert_logits_close(out1, ref0.forward(int(toks[p, 0]), p), f"slot0 pos {p}")


def test_batch_arguments_are_checked(tvl):
    cfg = small_config(max_batch=2, max_seq=8)
    blob = synth.make_blob(cfg, seed=2)
    with tvl.Model(cfg, blob) as m:
        with pytest.raises(tvl.TvlError) as e:
            m.forward_batch([1, 2, 3], 0)
        assert e.value.status == tvl.E_INVAL
        with pytest.raises(tvl.TvlError) as e:
            m.forward_batch([1, cfg["vocab_size"]], 0)
        assert e.value.status == tvl.E_RANGE
        with pytest.raises(tvl.TvlError) as e:
            m.decode_greedy_batch([1, 2], 4, 5)
        assert e.value.status == tvl.E_RANGE
        m.decode_greedy_batch([1, 2], 4, 4)  # the boundary case fits
    one = small_config()
    with tvl.Model(one, synth.make_blob(one, seed=2)) as m:
        assert m.info().max_batch == 1
        with pytest.raises(tvl.TvlError) as e:
            m.forward_batch([1, 2], 0)
        assert e.value.status == tvl.E_INVAL
    with pytest.raises(tvl.TvlError) as e:
        tvl.Model(small_config(max_batch=2, weight_bits=8), synth.make_blob(one, seed=2))
    assert e.value.status == tvl.E_UNSUPPORTED


def test_110m_batch4_greedy(tvl):
    """The 110M shape, four sequences from different tokens, 64 greedy steps."""
    cfg = synth.model_config("110m", max_batch=4)
    blob = synth.make_blob(cfg)
    starts = [1, 100, 2000, 31999]
    with tvl.Model(cfg, blob) as m:
        refs = [oracle.Model(cfg, blob, 64) for _ in starts]
        batch_greedy_check(m, refs, starts, 64, label="110m B4")


def test_7b_batch2_teacher_forced(tvl):
    """7B shape with two sequences: W2 rows (11008) span three stages, so the
    per-sequence segment sums are exercised; two steps against the oracle."""
    cfg = synth.model_config("7b", max_batch=2)
    free, total = torch.cuda.mem_get_info()
    if free < 36e9:
        pytest.skip("needs ~36 GB of free device memory")
    blob = synth.make_blob(cfg)
    toks = np.array([[1, 29871], [450, 3444]], np.int32)
    with tvl.Model(cfg, blob) as m:
        refs = [oracle.Model(cfg, blob, 64) for _ in range(2)]
        batch_teacher_forced(m, refs, toks, label="7b B2")
        gen = m.decode_greedy_batch([1, 450], 2, 8)
        assert gen.min() >= 0 and gen.max() < cfg["vocab_size"]
