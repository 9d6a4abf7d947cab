"""ctypes binding of libtvl.so: the C ABI of include/tvl.h, same names.

Argument marshalling only: every step of the decode path runs in the
library's CUDA kernels. Device buffers are passed as integer addresses (for
example ``tensor.data_ptr()`` of a torch CUDA tensor), host buffers as numpy
arrays. If libtvl.so is missing the import of this module fails: there is no
CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libtvl.so")

OK, E_INVAL, E_SIZE, E_ALIGN, E_NOMEM, E_CUDA, E_RANGE, E_TIMEOUT, E_UNSUPPORTED = range(9)


class TvlError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({last_error()})")


class Config(ctypes.Structure):
    _fields_ = [
        ("dim", ctypes.c_int32), ("hidden_dim", ctypes.c_int32), ("n_layers", ctypes.c_int32),
        ("n_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
        ("vocab_size", ctypes.c_int32), ("max_seq", ctypes.c_int32),
        ("rope_theta", ctypes.c_double), ("norm_eps", ctypes.c_double),
        ("shared_classifier", ctypes.c_int32), ("weight_bits", ctypes.c_int32),
        ("max_batch", ctypes.c_int32),
    ]


class ModelInfo(ctypes.Structure):
    _fields_ = [
        ("arena_bytes", ctypes.c_int64), ("weight_bytes", ctypes.c_int64),
        ("streamed_bytes", ctypes.c_int64), ("grid", ctypes.c_int32),
        ("threads", ctypes.c_int32), ("smem_bytes", ctypes.c_int32),
        ("ring_stages", ctypes.c_int32), ("stage_bytes", ctypes.c_int32),
        ("tied", ctypes.c_int32), ("exchanges_per_step", ctypes.c_int32),
        ("max_batch", ctypes.c_int32), ("next_tag", ctypes.c_int64),
    ]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    P, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    st = ctypes.c_int
    L.tvl_blob_bytes.restype = sz
    L.tvl_blob_bytes.argtypes = [ctypes.POINTER(Config), i32]
    L.tvl_load.restype = st
    L.tvl_load.argtypes = [ctypes.POINTER(Config), P, sz, P, ctypes.POINTER(P)]
    L.tvl_load_file.restype = st
    L.tvl_load_file.argtypes = [ctypes.POINTER(Config), ctypes.c_char_p, P, ctypes.POINTER(P)]
    L.tvl_forward.restype = st
    L.tvl_forward.argtypes = [P, i32, i32, P]
    L.tvl_decode_greedy.restype = st
    L.tvl_decode_greedy.argtypes = [P, i32, i32, i32, P]
    L.tvl_prefill.restype = st
    L.tvl_prefill.argtypes = [P, P, i32, i32, P]
    L.tvl_forward_batch.restype = st
    L.tvl_forward_batch.argtypes = [P, i32, P, i32, P]
    L.tvl_decode_greedy_batch.restype = st
    L.tvl_decode_greedy_batch.argtypes = [P, i32, P, i32, i32, P]
    L.tvl_gemv.restype = st
    L.tvl_gemv.argtypes = [P, P, P, i32, i32, P]
    L.tvl_q8_bytes.restype = sz
    L.tvl_q8_bytes.argtypes = [i32, i32]
    L.tvl_quantize_q8.restype = st
    L.tvl_quantize_q8.argtypes = [P, P, i32, i32, P]
    L.tvl_gemv_q8.restype = st
    L.tvl_gemv_q8.argtypes = [P, P, P, i32, i32, P]
    L.tvl_q4_bytes.restype = sz
    L.tvl_q4_bytes.argtypes = [i32, i32]
    L.tvl_quantize_q4.restype = st
    L.tvl_quantize_q4.argtypes = [P, P, i32, i32, P]
    L.tvl_gemv_q4.restype = st
    L.tvl_gemv_q4.argtypes = [P, P, P, i32, i32, P]
    L.tvl_gemv_noalloc.restype = st
    L.tvl_gemv_noalloc.argtypes = [P, P, P, i32, i32, P]
    L.tvl_gemm.restype = st
    L.tvl_gemm.argtypes = [P, P, P, i32, i32, i32, P]
    L.tvl_gemm_status.restype = st
    L.tvl_gemm_status.argtypes = [P]
    L.tvl_gemv_status.restype = st
    L.tvl_gemv_status.argtypes = [P]
    L.tvl_selftest_gemv_timeout.restype = st
    L.tvl_selftest_gemv_timeout.argtypes = [P, P, P, i32, i32, P]
    L.tvl_sync.restype = st
    L.tvl_sync.argtypes = [P]
    L.tvl_free.restype = None
    L.tvl_free.argtypes = [P]
    L.tvl_status_string.restype = ctypes.c_char_p
    L.tvl_status_string.argtypes = [st]
    L.tvl_last_error.restype = ctypes.c_char_p
    L.tvl_last_error.argtypes = []
    L.tvl_get_info.restype = st
    L.tvl_get_info.argtypes = [P, ctypes.POINTER(ModelInfo)]
    L.tvl_step_times.restype = st
    L.tvl_step_times.argtypes = [P, P, i32]
    L.tvl_selftest_barrier_timeout.restype = st
    L.tvl_selftest_barrier_timeout.argtypes = [i32]
    L.tvl_debug_fail_allocation.restype = None
    L.tvl_debug_fail_allocation.argtypes = [i32]
    L.tvl_debug_live_allocations.restype = i64
    L.tvl_debug_live_allocations.argtypes = []
    L.tvl_debug_set_next_tag.restype = st
    L.tvl_debug_set_next_tag.argtypes = [P, ctypes.c_uint64]
    return L


lib = _load()

EXPORTED = ["tvl_blob_bytes", "tvl_load", "tvl_load_file", "tvl_forward", "tvl_decode_greedy",
            "tvl_forward_batch", "tvl_decode_greedy_batch", "tvl_prefill",
            "tvl_gemv", "tvl_gemv_noalloc", "tvl_gemv_status", "tvl_selftest_gemv_timeout",
            "tvl_gemm", "tvl_gemm_status",
            "tvl_q8_bytes", "tvl_quantize_q8", "tvl_gemv_q8",
            "tvl_q4_bytes", "tvl_quantize_q4", "tvl_gemv_q4",
            "tvl_sync", "tvl_free", "tvl_status_string", "tvl_last_error",
            "tvl_get_info", "tvl_step_times", "tvl_selftest_barrier_timeout",
            "tvl_debug_fail_allocation", "tvl_debug_live_allocations", "tvl_debug_set_next_tag"]


def status_string(s: int) -> str:
    return lib.tvl_status_string(int(s)).decode()


def last_error() -> str:
    return lib.tvl_last_error().decode()


def _check(s: int, where: str):
    if s != OK:
        raise TvlError(s, where)


def make_config(cfg: dict) -> Config:
    return Config(
        int(cfg["dim"]), int(cfg["hidden_dim"]), int(cfg["n_layers"]), int(cfg["n_heads"]),
        int(cfg["n_kv_heads"]), int(cfg["vocab_size"]), int(cfg["max_seq"]),
        float(cfg.get("rope_theta", 10000.0)), float(cfg.get("norm_eps", 1e-5)),
        int(cfg.get("shared_classifier", 0)), int(cfg.get("weight_bits", 0)),
        int(cfg.get("max_batch", 0)),
    )


def tvl_blob_bytes(cfg: dict, tied: bool) -> int:
    c = make_config(cfg)
    return int(lib.tvl_blob_bytes(ctypes.byref(c), int(tied)))


def _addr(buf) -> int:
    """Address of a numpy array (host) or an integer device address."""
    if isinstance(buf, np.ndarray):
        return buf.ctypes.data
    return int(buf)


def tvl_gemv(W, x, y, d_out: int, d_in: int, stream: int = 0):
    """y = W x on the device; W, x, y are device addresses."""
    _check(lib.tvl_gemv(ctypes.c_void_p(_addr(W)), ctypes.c_void_p(_addr(x)),
                        ctypes.c_void_p(_addr(y)), int(d_out), int(d_in),
                        ctypes.c_void_p(int(stream))), "tvl_gemv")


def tvl_gemv_noalloc(W, x, y, d_out: int, d_in: int, stream: int = 0):
    """tvl_gemv with its scratch in a static module array (nothing allocated)."""
    _check(lib.tvl_gemv_noalloc(ctypes.c_void_p(_addr(W)), ctypes.c_void_p(_addr(x)),
                                ctypes.c_void_p(_addr(y)), int(d_out), int(d_in),
                                ctypes.c_void_p(int(stream))), "tvl_gemv_noalloc")


def tvl_gemm(W, X, Y, n: int, M: int, K: int, stream: int = 0):
    """Y [n x M] = X [n x K] W^T on the tensor cores; device addresses."""
    _check(lib.tvl_gemm(ctypes.c_void_p(_addr(W)), ctypes.c_void_p(_addr(X)),
                        ctypes.c_void_p(_addr(Y)), int(n), int(M), int(K),
                        ctypes.c_void_p(int(stream))), "tvl_gemm")


def tvl_gemm_status(stream: int = 0) -> int:
    return lib.tvl_gemm_status(ctypes.c_void_p(stream))


def tvl_gemv_status(stream: int = 0) -> int:
    """Waits for `stream`; the standalone GEMV kernels' error since the last
    query (TVL_E_TIMEOUT) or OK. Returns the status, does not raise."""
    return lib.tvl_gemv_status(ctypes.c_void_p(stream))


def tvl_selftest_gemv_timeout(W, x, y, d_out: int, d_in: int, stream: int = 0) -> int:
    """Returns the status the self-test reports (TVL_E_TIMEOUT expected)."""
    return lib.tvl_selftest_gemv_timeout(ctypes.c_void_p(_addr(W)), ctypes.c_void_p(_addr(x)),
                                         ctypes.c_void_p(_addr(y)), int(d_out), int(d_in),
                                         ctypes.c_void_p(stream))


def tvl_q8_bytes(rows: int, cols: int) -> int:
    return int(lib.tvl_q8_bytes(int(rows), int(cols)))


def tvl_quantize_q8(W, Wq8, rows: int, cols: int, stream: int = 0):
    """Packed 8-bit rows of W (device addresses)."""
    _check(lib.tvl_quantize_q8(ctypes.c_void_p(_addr(W)), ctypes.c_void_p(_addr(Wq8)), int(rows),
                               int(cols), ctypes.c_void_p(int(stream))), "tvl_quantize_q8")


def tvl_gemv_q8(Wq8, x, y, d_out: int, d_in: int, stream: int = 0):
    """y = W' x over packed 8-bit rows (device addresses)."""
    _check(lib.tvl_gemv_q8(ctypes.c_void_p(_addr(Wq8)), ctypes.c_void_p(_addr(x)),
                           ctypes.c_void_p(_addr(y)), int(d_out), int(d_in),
                           ctypes.c_void_p(int(stream))), "tvl_gemv_q8")


def tvl_q4_bytes(rows: int, cols: int) -> int:
    return int(lib.tvl_q4_bytes(int(rows), int(cols)))


def tvl_quantize_q4(W, Wq4, rows: int, cols: int, stream: int = 0):
    """Packed 4-bit rows of W (device addresses)."""
    _check(lib.tvl_quantize_q4(ctypes.c_void_p(_addr(W)), ctypes.c_void_p(_addr(Wq4)), int(rows),
                               int(cols), ctypes.c_void_p(int(stream))), "tvl_quantize_q4")


def tvl_gemv_q4(Wq4, x, y, d_out: int, d_in: int, stream: int = 0):
    """y = W' x over packed 4-bit rows (device addresses)."""
    _check(lib.tvl_gemv_q4(ctypes.c_void_p(_addr(Wq4)), ctypes.c_void_p(_addr(x)),
                           ctypes.c_void_p(_addr(y)), int(d_out), int(d_in),
                           ctypes.c_void_p(int(stream))), "tvl_gemv_q4")


def tvl_selftest_barrier_timeout(limit_ms: int) -> int:
    """Returns the status the kernel reported (TVL_E_TIMEOUT expected)."""
    return int(lib.tvl_selftest_barrier_timeout(int(limit_ms)))


class Model:
    """A loaded model (tvl_load ... tvl_free)."""

    def __init__(self, cfg: dict, blob=None, path: str | None = None, stream: int = 0,
                 nbytes: int | None = None):
        self.cfg = dict(cfg)
        self._c = make_config(cfg)
        h = ctypes.c_void_p()
        if path is not None:
            s = lib.tvl_load_file(ctypes.byref(self._c), path.encode(),
                                  ctypes.c_void_p(int(stream)), ctypes.byref(h))
            where = "tvl_load_file"
        else:
            n = blob.nbytes if isinstance(blob, np.ndarray) else int(nbytes)
            s = lib.tvl_load(ctypes.byref(self._c), ctypes.c_void_p(_addr(blob)), n,
                             ctypes.c_void_p(int(stream)), ctypes.byref(h))
            where = "tvl_load"
        _check(s, where)
        self._h = h
        self.vocab = int(cfg["vocab_size"])

    def info(self) -> ModelInfo:
        out = ModelInfo()
        _check(lib.tvl_get_info(self._h, ctypes.byref(out)), "tvl_get_info")
        return out

    def forward(self, token: int, pos: int, logits=None):
        """One decode step. logits: None (stay on device), a float32 numpy array
        of V (host: the call waits), or an integer device address (async)."""
        if logits is None:
            ptr = None
        else:
            if isinstance(logits, np.ndarray):
                assert logits.dtype == np.float32 and logits.size >= self.vocab
            ptr = ctypes.c_void_p(_addr(logits))
        _check(lib.tvl_forward(self._h, int(token), int(pos), ptr), "tvl_forward")
        return logits

    def decode_greedy(self, start_token: int, start_pos: int, n_steps: int, tokens=True):
        """Greedy decoding on the device; returns the generated tokens (numpy
        int32 array) or None when tokens=False (no copy, no wait)."""
        out = np.empty(int(n_steps), dtype=np.int32) if tokens else None
        ptr = ctypes.c_void_p(out.ctypes.data) if tokens else None
        _check(lib.tvl_decode_greedy(self._h, int(start_token), int(start_pos), int(n_steps),
                                     ptr), "tvl_decode_greedy")
        return out

    def prefill(self, tokens, start_pos: int = 0, logits=None):
        """Prefill: len(tokens) positions from start_pos in one pass per layer;
        logits of the last position as for forward()."""
        toks = np.ascontiguousarray(tokens, dtype=np.int32)
        if logits is None:
            ptr = None
        else:
            if isinstance(logits, np.ndarray):
                assert logits.dtype == np.float32 and logits.size >= self.vocab
            ptr = ctypes.c_void_p(_addr(logits))
        _check(lib.tvl_prefill(self._h, ctypes.c_void_p(toks.ctypes.data), int(toks.size),
                               int(start_pos), ptr), "tvl_prefill")
        return logits

    def forward_batch(self, tokens, pos: int, logits=None):
        """One step of len(tokens) sequences at position pos. logits: None,
        a float32 numpy array of batch * V (host: the call waits), or an
        integer device address (async); laid out [batch][V]."""
        toks = np.ascontiguousarray(tokens, dtype=np.int32)
        if logits is None:
            ptr = None
        else:
            if isinstance(logits, np.ndarray):
                assert logits.dtype == np.float32 and logits.size >= toks.size * self.vocab
            ptr = ctypes.c_void_p(_addr(logits))
        _check(lib.tvl_forward_batch(self._h, int(toks.size), ctypes.c_void_p(toks.ctypes.data),
                                     int(pos), ptr), "tvl_forward_batch")
        return logits

    def decode_greedy_batch(self, start_tokens, start_pos: int, n_steps: int, tokens=True):
        """Greedy decoding of len(start_tokens) sequences in lockstep; returns
        int32 [n_steps, batch] (or None when tokens=False: no copy, no wait)."""
        toks = np.ascontiguousarray(start_tokens, dtype=np.int32)
        out = np.empty((int(n_steps), toks.size), dtype=np.int32) if tokens else None
        ptr = ctypes.c_void_p(out.ctypes.data) if tokens else None
        _check(lib.tvl_decode_greedy_batch(self._h, int(toks.size),
                                           ctypes.c_void_p(toks.ctypes.data), int(start_pos),
                                           int(n_steps), ptr), "tvl_decode_greedy_batch")
        return out

    def step_times(self, n: int) -> np.ndarray:
        out = np.empty(int(n), dtype=np.uint64)
        _check(lib.tvl_step_times(self._h, ctypes.c_void_p(out.ctypes.data), int(n)),
               "tvl_step_times")
        return out

    def sync(self):
        _check(lib.tvl_sync(self._h), "tvl_sync")

    def close(self):
        if getattr(self, "_h", None):
            lib.tvl_free(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
