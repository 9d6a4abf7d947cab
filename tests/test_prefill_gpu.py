"""Multi-token prefill (tvl_prefill) on the GPU vs the CPU oracle fed the same
tokens one position at a time.

The logits of the last prefilled position must match the oracle's (max |d| <=
2e-3 * max |logit|), and the K/V rows it leaves behind must be the oracle's:
decoding after the prefill (teacher-forced logits, then the device greedy
loop) matches the oracle's continuation wherever its top-2 margin exceeds 1e-2.
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


def oracle_run(ref, toks, start=0):
    lg = None
    for i, t in enumerate(toks):
        lg = ref.forward(int(t), start + i)
    return lg


def check_prefill_then_decode(tvl, cfg, blob, n, n_decode=8, label=""):
    V = cfg["vocab_size"]
    toks = synth.uniform_ints(n, 23, 0, 0, V - 1)
    ref = oracle.Model(cfg, blob, 64)
    out = np.empty(V, np.float32)
    with tvl.Model(cfg, blob) as m:
        m.prefill(toks, 0, out)
        lg = oracle_run(ref, toks)
        assert_logits_close(out, lg, f"{label} prefill n={n}")
        if n + n_decode <= cfg["max_seq"]:
            # teacher-forced steps after the prefill read its K/V rows
            t = int(np.argmax(lg))
            for s in range(n_decode):
                m.forward(t, n + s, out)
                lg = ref.forward(t, n + s)
                assert_logits_close(out, lg, f"{label} decode pos {n + s}")
                t = int(np.argmax(lg))


@pytest.mark.parametrize("kw", [
    dict(),                                    # several layers
    dict(n_kv_heads=2),                        # grouped query heads
    dict(n_kv_heads=1, n_heads=8),             # one kv head, head_dim 8
    dict(n_layers=0),                          # embedding -> final norm -> classifier
    dict(dim=96, n_heads=2, n_kv_heads=2, hidden_dim=8200, vocab_size=333),  # wide FFN
    dict(dim=128, n_heads=1, n_kv_heads=1, hidden_dim=256),  # head_dim 128
    dict(n_heads=2, n_kv_heads=1),                           # head_dim 32, grouped
    dict(dim=192, n_heads=2, n_kv_heads=2, hidden_dim=128),  # head_dim 96
], ids=["base", "gqa2", "mqa", "L0", "wide_ffn", "hd128", "hd32_gqa", "hd96"])
def test_prefill_matches_oracle(tvl, kw):
    cfg = small_config(**kw)
    blob = synth.make_blob(cfg, seed=41)
    check_prefill_then_decode(tvl, cfg, blob, 40, label=str(kw))


@pytest.mark.parametrize("n", [1, 2, 31, 64])
def test_prefill_lengths(tvl, n):
    cfg = small_config()
    blob = synth.make_blob(cfg, seed=42)
    check_prefill_then_decode(tvl, cfg, blob, n, n_decode=0 if n == 64 else 4, label=f"n={n}")


def test_prefill_in_two_parts_and_greedy_after(tvl):
    cfg = small_config()
    V = cfg["vocab_size"]
    blob = synth.make_blob(cfg, seed=43)
    toks = synth.uniform_ints(36, 5, 0, 0, V - 1)
    ref = oracle.Model(cfg, blob, 64)
    out = np.empty(V, np.float32)
    with tvl.Model(cfg, blob) as m:
        m.prefill(toks[:20], 0)
        m.prefill(toks[20:], 20, out)
        lg = oracle_run(ref, toks)
        assert_logits_close(out, lg, "second part")
        start = int(np.argmax(lg))
        rtoks, rlg = ref.greedy(start, 20, start_pos=36)
        gen = m.decode_greedy(start, 36, 20)
        compare_greedy(gen, rtoks[1:] + [int(np.argmax(rlg[-1]))], rlg)


def test_prefill_device_logits_and_arguments(tvl):
    cfg = small_config(max_seq=16)
    blob = synth.make_blob(cfg, seed=44)
    V = cfg["vocab_size"]
    with tvl.Model(cfg, blob) as m:
        dl = torch.empty(V, device="cuda")
        host = np.empty(V, np.float32)
        m.prefill([3, 4, 5], 0, host)
        m.prefill([3, 4, 5], 0, dl.data_ptr())
        m.sync()
        assert np.array_equal(dl.cpu().numpy(), host)
        for toks, start in (([], 0), ([1] * 17, 0), ([1, 2], 15), ([V], 0), ([-1], 0), ([1], -1)):
            with pytest.raises(tvl.TvlError) as e:
                m.prefill(toks, start)
            assert e.value.status == tvl.E_RANGE
        m.prefill([1] * 16, 0)  # the whole cache fits
    with pytest.raises(tvl.TvlError) as e:
        with tvl.Model(dict(cfg, weight_bits=8), blob) as q:
            q.prefill([1, 2], 0)
    assert e.value.status == tvl.E_UNSUPPORTED


def test_110m_prefill_896_prompt_then_greedy(tvl):
    """The long-context workload's 896-token prompt in one prefill call."""
    cfg = synth.model_config("110m")
    blob = synth.make_blob(cfg)
    prompt = synth.long_context_tokens(896)
    ref = oracle.Model(cfg, blob, 64)
    out = np.empty(cfg["vocab_size"], np.float32)
    with tvl.Model(cfg, blob) as m:
        m.prefill(prompt, 0, out)
        lg = oracle_run(ref, prompt)
        assert_logits_close(out, lg, "110m prefill 896")
        start = int(np.argmax(lg))
        rtoks, rlg = ref.greedy(start, 32, start_pos=896)
        gen = m.decode_greedy(start, 896, 32)
        compare_greedy(gen, rtoks[1:] + [int(np.argmax(rlg[-1]))], rlg)


@pytest.mark.parametrize("parts,kw", [
    ((300, 140), dict()),                                     # 14 key tiles: 4 splits of 4
    ((1050,), dict(dim=128, n_heads=2, n_kv_heads=1)),        # 33 tiles: 7 splits of 5, hd 64
    ((129, 3, 700), dict(n_kv_heads=2)),                      # ragged parts, grouped heads
    ((65, 1, 300, 130), dict(dim=128, n_heads=2, n_kv_heads=1)),  # ragged, head_dim 64
], ids=["two_parts", "long_hd64", "ragged", "ragged_hd64"])
def test_prefill_long_key_ranges_split_across_ctas(tvl, parts, kw):
    """Rows that see more than 128 keys have their key range cut into up to
    eight parts, each a CTA of its own, whose partial sums are merged; the
    logits after each part and the continuation (which reads every row's K/V
    of the second layer, made from the first layer's merged attention) must
    match the oracle."""
    cfg = small_config(max_seq=1100, **kw)
    V = cfg["vocab_size"]
    blob = synth.make_blob(cfg, seed=45)
    toks = synth.uniform_ints(sum(parts), 7, 0, 0, V - 1)
    ref = oracle.Model(cfg, blob, 64)
    out = np.empty(V, np.float32)
    with tvl.Model(cfg, blob) as m:
        p0 = 0
        for n in parts:
            m.prefill(toks[p0:p0 + n], p0, out)
            lg = oracle_run(ref, toks[p0:p0 + n], p0)
            assert_logits_close(out, lg, f"prefill {p0}..{p0 + n - 1}")
            p0 += n
        t = int(np.argmax(lg))
        for s in range(4):
            m.forward(t, p0 + s, out)
            lg = ref.forward(t, p0 + s)
            assert_logits_close(out, lg, f"decode pos {p0 + s}")
            t = int(np.argmax(lg))
