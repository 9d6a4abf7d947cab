"""The C ABI without a GPU: the library loads, exports every declared entry
point, and rejects bad arguments on the host before touching the device."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_2601_03324_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def tvl():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2601_03324_gb300 import tvl as t
    return t


def declared_functions():
    text = open(os.path.join(ROOT, "include", "tvl.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tvl_\w+)\s*\(", text)))


def test_every_declared_entry_point_is_exported(tvl):
    names = declared_functions()
    assert len(names) >= 12
    lib = ctypes.CDLL(tvl.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(tvl.EXPORTED) == names


def test_blob_bytes_agree_with_generator_and_oracle(tvl):
    for name in ("tiny", "110m", "7b"):
        cfg = synth.model_config(name)
        for tied in (False, True):
            b = tvl.tvl_blob_bytes(cfg, tied)
            assert b == synth.blob_bytes(cfg, tied) == oracle.blob_bytes(cfg, tied)
    odd = dict(dim=12, hidden_dim=10, n_layers=2, n_heads=3, n_kv_heads=1, vocab_size=7,
               max_seq=5)
    assert tvl.tvl_blob_bytes(odd, False) == synth.blob_bytes(odd, False)
    assert tvl.tvl_blob_bytes(dict(odd, n_heads=5), False) == 0  # 12 % 5 != 0


@pytest.mark.parametrize("bad,status", [
    (dict(dim=0), "E_INVAL"),
    (dict(n_heads=3), "E_INVAL"),            # 64 % 3 != 0
    (dict(n_kv_heads=3), "E_INVAL"),         # 4 % 3 != 0
    (dict(max_seq=0), "E_INVAL"),
    (dict(shared_classifier=2), "E_INVAL"),
    (dict(dim=48, n_heads=4), "E_UNSUPPORTED"),   # dim % 32 != 0
    (dict(dim=64, n_heads=32), "E_UNSUPPORTED"),  # head_dim 2
    (dict(hidden_dim=98), "E_UNSUPPORTED"),
    (dict(dim=256, n_heads=1, n_kv_heads=1), "E_UNSUPPORTED"),  # head_dim 256 > 128
    (dict(weight_bits=5), "E_INVAL"),                           # 0, 8 or 4 only
    (dict(weight_bits=4, hidden_dim=112), "E_UNSUPPORTED"),     # 4-bit rows: 112 % 32 != 0
    (dict(weight_bits=8, hidden_dim=104), "E_UNSUPPORTED"),     # 8-bit rows: 104 % 16 != 0
    (dict(max_batch=5), "E_INVAL"),                             # 0 to 4 sequences
    (dict(max_batch=-1), "E_INVAL"),
    (dict(max_batch=2, weight_bits=8), "E_UNSUPPORTED"),        # batches need float32 rows
    (dict(max_batch=3, weight_bits=4), "E_UNSUPPORTED"),
])
def test_load_rejects_invalid_configs_on_the_host(tvl, bad, status):
    cfg = dict(dim=64, hidden_dim=96, n_layers=1, n_heads=4, n_kv_heads=4, vocab_size=100,
               max_seq=16, shared_classifier=0)
    cfg.update(bad)
    blob = np.zeros(64, np.float32)
    with pytest.raises(tvl.TvlError) as e:
        tvl.Model(cfg, blob)
    assert e.value.status == getattr(tvl, status)


def test_load_rejects_wrong_blob_size_before_any_device_work(tvl):
    cfg = dict(dim=64, hidden_dim=96, n_layers=1, n_heads=4, n_kv_heads=4, vocab_size=100,
               max_seq=16, shared_classifier=0)
    n = tvl.tvl_blob_bytes(cfg, False) // 4
    with pytest.raises(tvl.TvlError) as e:
        tvl.Model(cfg, np.zeros(n - 32, np.float32))
    assert e.value.status == tvl.E_SIZE
    # -1 infers tying from the size; neither size matches here
    with pytest.raises(tvl.TvlError) as e:
        tvl.Model(dict(cfg, shared_classifier=-1), np.zeros(n + 32, np.float32))
    assert e.value.status == tvl.E_SIZE


def test_null_and_bad_arguments(tvl):
    L = tvl.lib
    assert L.tvl_forward(None, 0, 0, None) == tvl.E_INVAL
    assert L.tvl_decode_greedy(None, 0, 0, 1, None) == tvl.E_INVAL
    assert L.tvl_sync(None) == tvl.E_INVAL
    L.tvl_free(None)
    assert L.tvl_gemv(None, None, None, 4, 4, None) == tvl.E_INVAL
    assert L.tvl_gemv(16, 16, 16, 0, 4, None) == tvl.E_INVAL
    assert L.tvl_selftest_barrier_timeout(0) == tvl.E_INVAL
    assert L.tvl_load(None, None, 0, None, None) == tvl.E_INVAL
    assert "range" in tvl.status_string(tvl.E_RANGE)
    assert tvl.status_string(99) == "unknown status"


def test_q8_row_bytes_on_the_host(tvl):
    assert tvl.tvl_q8_bytes(3, 32) == 3 * 48
    assert tvl.tvl_q8_bytes(32000, 768) == 32000 * 784
    for rows, cols in ((0, 32), (3, 8), (3, 24), (3, 0), (-1, 16)):
        assert tvl.tvl_q8_bytes(rows, cols) == 0


def test_q4_row_bytes_and_argument_checks_on_the_host(tvl):
    assert tvl.tvl_q4_bytes(3, 32) == 3 * 32
    assert tvl.tvl_q4_bytes(32000, 4096) == 32000 * (16 + 2048)
    for rows, cols in ((0, 32), (3, 16), (3, 48), (3, 0), (-1, 32)):
        assert tvl.tvl_q4_bytes(rows, cols) == 0
    L = tvl.lib
    # size, null and alignment checks come before any device call
    assert L.tvl_quantize_q4(None, None, 4, 32, None) == tvl.E_INVAL
    assert L.tvl_quantize_q4(16, 16, 4, 48, None) == tvl.E_INVAL
    assert L.tvl_quantize_q4(20, 16, 4, 32, None) == tvl.E_ALIGN
    assert L.tvl_gemv_q4(None, 16, 16, 4, 32, None) == tvl.E_INVAL
    assert L.tvl_gemv_q4(16, 16, 16, 4, 40, None) == tvl.E_INVAL
    assert L.tvl_gemv_q4(16, 24, 16, 4, 32, None) == tvl.E_ALIGN
    assert L.tvl_gemv_q4(16, 16, 16, 1, 32768, None) == tvl.E_UNSUPPORTED  # row over a stage
    assert "multiple of 32" in tvl.last_error() or "stage" in tvl.last_error()

