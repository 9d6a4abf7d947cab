"""Failure handling on the GPU without a GPU fault: exchange tags across the
32-bit wrap, allocation failures at every point of the allocating calls, and a
standalone GEMV wait that runs out (a stage that is never copied)."""
import numpy as np
import pytest

import oracle
from helpers import assert_logits_close, compare_greedy, gemv_bound, small_config
from paper_2601_03324_gb300 import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def tvl():
    from paper_2601_03324_gb300 import tvl as t
    return t


def test_decode_across_the_exchange_tag_wrap(tvl):
    # Tags 1.. are used by the first steps; the next tag is then put just
    # before 2^32, so that the following launches would reuse tags those steps
    # left in the exchange words (and tag 0, which zeroed words carry). The
    # library must zero the words and restart at tag 1 instead: parity holds
    # and the model's next tag is small again.
    cfg = small_config(n_layers=2)
    blob = synth.make_blob(cfg, seed=21)
    ref = oracle.Model(cfg, blob)
    toks, logits = ref.greedy(1, 24)
    per_step = 5 * cfg["n_layers"] + 1
    with tvl.Model(cfg, blob) as m:
        out = np.empty(cfg["vocab_size"], np.float32)
        for p in range(6):
            m.forward(toks[p], p, out)
            assert_logits_close(out, logits[p], f"before the wrap, pos {p}")
        assert m.info().next_tag == 1 + 6 * per_step
        tvl._check(tvl.lib.tvl_debug_set_next_tag(m._h, 2 ** 32 - 1 - per_step // 2),
                   "tvl_debug_set_next_tag")
        m.forward(toks[6], 6, out)  # this launch's tags would pass 2^32 - 1
        assert_logits_close(out, logits[6], "across the wrap, pos 6")
        assert m.info().next_tag == 1 + per_step
        for p in range(7, 10):
            m.forward(toks[p], p, out)
            assert_logits_close(out, logits[p], f"after the wrap, pos {p}")
        # a greedy launch of several steps that starts right before the wrap
        tvl._check(tvl.lib.tvl_debug_set_next_tag(m._h, 2 ** 32 - 3 * per_step),
                   "tvl_debug_set_next_tag")
        gen = m.decode_greedy(toks[10], 10, 14)
        compare_greedy(gen, toks[11:], logits[10:])
        assert m.info().next_tag == 1 + 14 * per_step


def test_lowering_the_next_tag_clears_the_exchange_words(tvl):
    # Words are published as the unsigned maximum of the old and the new word,
    # so a tag below those the words hold would never show: lowering the tag
    # must zero the words first. Decode, go back to tag 1, decode on (the
    # teacher-forced logits and a greedy launch), parity throughout.
    cfg = small_config(n_layers=2)
    blob = synth.make_blob(cfg, seed=22)
    ref = oracle.Model(cfg, blob)
    toks, logits = ref.greedy(1, 20)
    per_step = 5 * cfg["n_layers"] + 1
    with tvl.Model(cfg, blob) as m:
        out = np.empty(cfg["vocab_size"], np.float32)
        for p in range(5):
            m.forward(toks[p], p, out)
            assert_logits_close(out, logits[p], f"pos {p}")
        assert m.info().next_tag == 1 + 5 * per_step
        tvl._check(tvl.lib.tvl_debug_set_next_tag(m._h, 1), "tvl_debug_set_next_tag")
        assert m.info().next_tag == 1
        for p in range(5, 8):
            m.forward(toks[p], p, out)
            assert_logits_close(out, logits[p], f"after lowering the tag, pos {p}")
        tvl._check(tvl.lib.tvl_debug_set_next_tag(m._h, 2), "tvl_debug_set_next_tag")
        gen = m.decode_greedy(toks[8], 8, 11)  # positions 8..18: oracle tokens 9..19
        compare_greedy(gen, toks[9:], logits[8:])
        assert m.info().next_tag == 2 + 11 * per_step


def test_set_next_tag_rejects_zero_and_values_beyond_32_bits(tvl):
    cfg = small_config(n_layers=1)
    with tvl.Model(cfg, synth.make_blob(cfg, seed=2)) as m:
        for bad in (0, 2 ** 32, 2 ** 40):
            assert tvl.lib.tvl_debug_set_next_tag(m._h, bad) == tvl.E_INVAL


def _load_status(tvl, cfg, blob):
    import ctypes
    c = tvl.make_config(cfg)
    h = ctypes.c_void_p()
    st = tvl.lib.tvl_load(ctypes.byref(c), ctypes.c_void_p(blob.ctypes.data), blob.nbytes, None,
                          ctypes.byref(h))
    return st, h


@pytest.mark.parametrize("weight_bits", [0, 8])
def test_every_allocation_failure_of_tvl_load_returns_nomem_and_holds_nothing(tvl, weight_bits):
    cfg = small_config(n_layers=2, weight_bits=weight_bits)
    blob = synth.make_blob(cfg, seed=3)
    st, h = _load_status(tvl, cfg, blob)  # warm the context up once
    assert st == tvl.OK
    tvl.lib.tvl_free(h)
    torch.cuda.synchronize()
    live0 = tvl.lib.tvl_debug_live_allocations()
    free0 = torch.cuda.mem_get_info()[0]
    k, failures = 0, 0
    try:
        while True:
            tvl.lib.tvl_debug_fail_allocation(k)
            st, h = _load_status(tvl, cfg, blob)
            if st == tvl.OK:
                break
            assert st == tvl.E_NOMEM, (k, tvl.status_string(st), tvl.last_error())
            assert not h.value
            assert tvl.lib.tvl_debug_live_allocations() == live0, k
            failures += 1
            k += 1
            assert k < 16
    finally:
        tvl.lib.tvl_debug_fail_allocation(-1)
    assert failures >= 3  # arena, mapped error word, W1/W3 scratch
    # freeing the load that finally succeeded returns everything
    tvl.lib.tvl_free(h)
    torch.cuda.synchronize()
    assert tvl.lib.tvl_debug_live_allocations() == live0
    assert abs(torch.cuda.mem_get_info()[0] - free0) < (4 << 20)


def test_prefill_allocation_failure_leaves_the_model_usable(tvl):
    cfg = small_config(n_layers=2)
    blob = synth.make_blob(cfg, seed=4)
    ref = oracle.Model(cfg, blob)
    toks, logits = ref.greedy(1, 6)
    with tvl.Model(cfg, blob) as m:
        live0 = tvl.lib.tvl_debug_live_allocations()
        tvl.lib.tvl_debug_fail_allocation(0)
        try:
            with pytest.raises(tvl.TvlError) as e:
                m.prefill(toks[:5], 0)
            assert e.value.status == tvl.E_NOMEM
        finally:
            tvl.lib.tvl_debug_fail_allocation(-1)
        assert tvl.lib.tvl_debug_live_allocations() == live0
        out = np.empty(cfg["vocab_size"], np.float32)
        m.prefill(toks[:5], 0, out)
        assert_logits_close(out, logits[4], "prefill after a failed first attempt")


def test_gemv_scratch_allocation_failure_returns_nomem_then_recovers(tvl):
    M, K = 64, 8192  # split along K: tvl_gemv needs its per-stream scratch
    W, x = synth.gemv_operands(M, K, 13)
    dW, dx = torch.from_numpy(W).cuda(), torch.from_numpy(x).cuda()
    y = torch.empty(M, device="cuda")
    s = torch.cuda.Stream()  # a fresh stream has no scratch yet
    live0 = tvl.lib.tvl_debug_live_allocations()
    for k in (0, 1):
        tvl.lib.tvl_debug_fail_allocation(k)
        try:
            with pytest.raises(tvl.TvlError) as e:
                tvl.tvl_gemv(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K, s.cuda_stream)
            assert e.value.status == tvl.E_NOMEM
        finally:
            tvl.lib.tvl_debug_fail_allocation(-1)
        assert tvl.lib.tvl_debug_live_allocations() == live0
    tvl.tvl_gemv(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K, s.cuda_stream)
    s.synchronize()
    assert np.all(np.abs(y.cpu().numpy() - oracle.gemv(W, x)) <= gemv_bound(W, x))


@pytest.mark.parametrize("shape", [(64, 8192), (100, 2048), (768, 768), (4096, 4096)],
                         ids=lambda s: f"{s[0]}x{s[1]}")
def test_gemv_wait_that_runs_out_is_reported_and_later_calls_are_right(tvl, shape):
    # CTA 0's last stage is never copied: its consumer gives up after the
    # one-second limit and raises TVL_E_TIMEOUT in the GEMV error word. Split
    # rows that other CTAs counted for that call must not disturb later calls
    # on the same counters (tvl_gemv_noalloc's static scratch).
    M, K = shape
    W, x = synth.gemv_operands(M, K, 14)
    dW, dx = torch.from_numpy(W).cuda(), torch.from_numpy(x).cuda()
    y = torch.empty(M, device="cuda")
    s = torch.cuda.Stream()
    ref = torch.empty(M, device="cuda")
    tvl.tvl_gemv(dW.data_ptr(), dx.data_ptr(), ref.data_ptr(), M, K, s.cuda_stream)
    s.synchronize()
    st = tvl.tvl_selftest_gemv_timeout(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K,
                                       s.cuda_stream)
    assert st == tvl.E_TIMEOUT, tvl.last_error()
    assert tvl.tvl_gemv_status(s.cuda_stream) == tvl.OK  # the query cleared it
    for _ in range(2):
        y.fill_(float("nan"))
        tvl.tvl_gemv_noalloc(dW.data_ptr(), dx.data_ptr(), y.data_ptr(), M, K, s.cuda_stream)
        s.synchronize()
        assert np.array_equal(y.cpu().numpy(), ref.cpu().numpy())
    assert tvl.tvl_gemv_status(s.cuda_stream) == tvl.OK
