"""CPU oracle of the batch-1 Llama-2 decode step (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference arms may import this package. It wraps ``liborc.so`` (built from
``orc.cpp`` by :func:`build`) with ctypes and numpy; it never imports the CUDA
package and the CUDA package never imports it.

The arithmetic lives in ``orc.cpp``: plain scalar loops, double accumulators
for the parity truth (``acc_bits=64``) or float ones (``acc_bits=32``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "orc.cpp")
_LIB = os.path.join(_HERE, "liborc.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile liborc.so with the host compiler (no SIMD flags, no FMA contraction)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "orc.h"))
    ):
        cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-ffp-contract=off",
               "-fno-fast-math", "-o", _LIB + ".tmp", _SRC]
        subprocess.run(cmd, check=True)
        os.replace(_LIB + ".tmp", _LIB)
    return _LIB


class Config(ctypes.Structure):
    _fields_ = [
        ("dim", ctypes.c_int32), ("hidden_dim", ctypes.c_int32), ("n_layers", ctypes.c_int32),
        ("n_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
        ("vocab_size", ctypes.c_int32), ("max_seq", ctypes.c_int32),
        ("rope_theta", ctypes.c_double), ("norm_eps", ctypes.c_double),
        ("shared_classifier", ctypes.c_int32),
    ]


def make_config(cfg: dict) -> Config:
    return Config(
        int(cfg["dim"]), int(cfg["hidden_dim"]), int(cfg["n_layers"]), int(cfg["n_heads"]),
        int(cfg["n_kv_heads"]), int(cfg["vocab_size"]), int(cfg["max_seq"]),
        float(cfg.get("rope_theta", 10000.0)), float(cfg.get("norm_eps", 1e-5)),
        int(cfg.get("shared_classifier", 0)),
    )


def lib():
    global _lib
    if _lib is None:
        path = build()
        L = ctypes.CDLL(path)
        P = ctypes.c_void_p
        i64, i32, dbl = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
        L.orc_blob_bytes.restype = i64
        L.orc_blob_bytes.argtypes = [ctypes.POINTER(Config), ctypes.c_int]
        L.orc_tensor_offset.restype = i64
        L.orc_tensor_offset.argtypes = [ctypes.POINTER(Config), ctypes.c_int, ctypes.c_int,
                                        ctypes.c_int]
        L.orc_model_new.restype = P
        L.orc_model_new.argtypes = [ctypes.POINTER(Config), P, ctypes.c_size_t, ctypes.c_int,
                                    ctypes.POINTER(ctypes.c_int)]
        L.orc_model_new_fmt.restype = P
        L.orc_model_new_fmt.argtypes = [ctypes.POINTER(Config), P, ctypes.c_size_t, ctypes.c_int,
                                        ctypes.c_int, ctypes.POINTER(ctypes.c_int)]
        L.orc_quantize_rows_q8.restype = None
        L.orc_quantize_rows_q8.argtypes = [P, i64, i64, P, P]
        L.orc_quantize_rows_q4.restype = None
        L.orc_quantize_rows_q4.argtypes = [P, i64, i64, P, P]
        L.orc_gemv_q8_f64.restype = None
        L.orc_gemv_q8_f64.argtypes = [P, P, P, P, i64, i64]
        L.orc_forward.restype = ctypes.c_int
        L.orc_forward.argtypes = [P, i32, i32, P]
        L.orc_model_tied.restype = ctypes.c_int
        L.orc_model_tied.argtypes = [P]
        L.orc_model_free.restype = None
        L.orc_model_free.argtypes = [P]
        L.orc_gemv_f64.argtypes = [P, P, P, i64, i64]
        L.orc_gemv_f32.argtypes = [P, P, P, i64, i64]
        L.orc_rmsnorm_f64.argtypes = [P, P, P, i64, dbl]
        L.orc_rope_f64.argtypes = [P, i64, i64, i32, dbl]
        L.orc_softmax_f64.argtypes = [P, i64]
        L.orc_silu_f64.restype = dbl
        L.orc_silu_f64.argtypes = [dbl]
        L.orc_attention_head_f64.argtypes = [P, P, P, i64, i64, i64, P]
        for name in ("orc_gemv_f64", "orc_gemv_f32", "orc_rmsnorm_f64", "orc_rope_f64",
                     "orc_softmax_f64", "orc_attention_head_f64"):
            getattr(L, name).restype = None
        _lib = L
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return ctypes.c_void_p(a.ctypes.data)


# ---- primitives ---------------------------------------------------------------

def gemv(W: np.ndarray, x: np.ndarray, acc_bits: int = 64) -> np.ndarray:
    """y = W x with W float32 [M, K] row-major."""
    W = np.ascontiguousarray(W, dtype=np.float32)
    M, K = W.shape
    if acc_bits == 64:
        x = np.ascontiguousarray(x, dtype=np.float64)
        y = np.empty(M, dtype=np.float64)
        lib().orc_gemv_f64(_ptr(W), _ptr(x), _ptr(y), M, K)
    else:
        x = np.ascontiguousarray(x, dtype=np.float32)
        y = np.empty(M, dtype=np.float32)
        lib().orc_gemv_f32(_ptr(W), _ptr(x), _ptr(y), M, K)
    return y


def quantize_rows_q8(W: np.ndarray):
    """8-bit codes and row scales of W float32 [M, K] (see orc_quantize_rows_q8)."""
    W = np.ascontiguousarray(W, dtype=np.float32)
    M, K = W.shape
    q = np.empty((M, K), dtype=np.int8)
    s = np.empty(M, dtype=np.float32)
    lib().orc_quantize_rows_q8(_ptr(W), M, K, _ptr(q), _ptr(s))
    return q, s


def quantize_rows_q4(W: np.ndarray):
    """4-bit codes (one per int8, in [-7, 7]) and row scales of W float32 [M, K]
    (see orc_quantize_rows_q4)."""
    W = np.ascontiguousarray(W, dtype=np.float32)
    M, K = W.shape
    q = np.empty((M, K), dtype=np.int8)
    s = np.empty(M, dtype=np.float32)
    lib().orc_quantize_rows_q4(_ptr(W), M, K, _ptr(q), _ptr(s))
    return q, s


def gemv_q8(q: np.ndarray, s: np.ndarray, x: np.ndarray) -> np.ndarray:
    """y = (s_i q_ij) x in double (the codes of quantize_rows_q8 or _q4)."""
    q = np.ascontiguousarray(q, dtype=np.int8)
    s = np.ascontiguousarray(s, dtype=np.float32)
    x = np.ascontiguousarray(x, dtype=np.float64)
    M, K = q.shape
    y = np.empty(M, dtype=np.float64)
    lib().orc_gemv_q8_f64(_ptr(q), _ptr(s), _ptr(x), _ptr(y), M, K)
    return y


def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float = 1e-5) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    g = np.ascontiguousarray(g, dtype=np.float32)
    out = np.empty_like(x)
    lib().orc_rmsnorm_f64(_ptr(x), _ptr(g), _ptr(out), x.size, eps)
    return out


def rope(v: np.ndarray, head_dim: int, pos: int, theta: float = 10000.0) -> np.ndarray:
    v = np.array(v, dtype=np.float64, copy=True)
    lib().orc_rope_f64(_ptr(v), v.size, head_dim, pos, theta)
    return v


def softmax(s: np.ndarray) -> np.ndarray:
    s = np.array(s, dtype=np.float64, copy=True)
    lib().orc_softmax_f64(_ptr(s), s.size)
    return s


def silu(z: float) -> float:
    return lib().orc_silu_f64(float(z))


def attention_head(q, K, V) -> np.ndarray:
    """q [hd]; K, V [npos, hd] (contiguous rows)."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    K = np.ascontiguousarray(K, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    npos, hd = K.shape
    out = np.empty(hd, dtype=np.float64)
    lib().orc_attention_head_f64(_ptr(q), _ptr(K), _ptr(V), npos, hd, hd, _ptr(out))
    return out


def blob_bytes(cfg: dict, tied: bool) -> int:
    c = make_config(cfg)
    return int(lib().orc_blob_bytes(ctypes.byref(c), int(tied)))


def tensor_offset(cfg: dict, tied: bool, which: int, layer: int = 0) -> int:
    c = make_config(cfg)
    return int(lib().orc_tensor_offset(ctypes.byref(c), int(tied), which, layer))


class Model:
    """One decode session of the oracle over a borrowed blob (numpy array kept alive)."""

    def __init__(self, cfg: dict, blob: np.ndarray, acc_bits: int = 64, weight_bits: int = 0):
        """weight_bits 8 or 4: every weight matrix as 8-bit or 4-bit codes with row scales."""
        self._blob = blob  # keep alive
        self.cfg = dict(cfg)
        c = make_config(cfg)
        err = ctypes.c_int(0)
        self._h = lib().orc_model_new_fmt(ctypes.byref(c), ctypes.c_void_p(blob.ctypes.data),
                                          blob.nbytes, acc_bits, int(weight_bits),
                                          ctypes.byref(err))
        if not self._h:
            raise ValueError(f"orc_model_new failed with code {err.value}")
        self.vocab = int(cfg["vocab_size"])

    @property
    def tied(self) -> bool:
        return bool(lib().orc_model_tied(self._h))

    def forward(self, token: int, pos: int) -> np.ndarray:
        out = np.empty(self.vocab, dtype=np.float64)
        rc = lib().orc_forward(self._h, int(token), int(pos), _ptr(out))
        if rc != 0:
            raise ValueError(f"orc_forward failed with code {rc}")
        return out

    def greedy(self, start_token: int, n_steps: int, start_pos: int = 0):
        """Greedy decode; returns (tokens fed, logits per step). Ties: lowest index."""
        toks, logits = [], []
        t = int(start_token)
        for s in range(n_steps):
            lg = self.forward(t, start_pos + s)
            toks.append(t)
            logits.append(lg)
            t = int(np.argmax(lg))  # numpy argmax returns the first maximum
        return toks, logits

    def close(self):
        if getattr(self, "_h", None):
            lib().orc_model_free(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
