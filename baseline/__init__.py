"""The paper's own method on one host core: a timing baseline for the benchmark.

``neon_decode.c`` runs the float32 decode step with the paper's NEON GEMV
(float32x4 lanes, four independent accumulators per row, §6.1 and §11.1) and
NEON RMSNorm (§11.2) on aarch64 hosts, plain C with the same four
accumulators elsewhere. It is neither the parity reference (``oracle/``) nor
part of the GPU library, and shares no code with either; only ``bench.py``
and ``tests/`` load it. Weights are borrowed from a blob laid out by
``paper_2601_03324_gb300.synth`` (the seeded input generator), one pointer per
tensor.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "neon_decode.c")
_LIB = os.path.join(_HERE, "libneon_decode.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile with the host compiler; NEON is part of every aarch64 target, so no
    machine-specific flag is needed."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        cmd = ["gcc", "-O3", "-std=c11", "-fPIC", "-shared", "-o", _LIB + ".tmp", _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(_LIB + ".tmp", _LIB)
    return _LIB


_PP = ctypes.POINTER(ctypes.c_void_p)


class _Weights(ctypes.Structure):
    _fields_ = [
        ("dim", ctypes.c_int), ("hidden", ctypes.c_int), ("n_layers", ctypes.c_int),
        ("n_heads", ctypes.c_int), ("n_kv_heads", ctypes.c_int), ("vocab", ctypes.c_int),
        ("max_seq", ctypes.c_int), ("rope_theta", ctypes.c_float), ("eps", ctypes.c_float),
        ("E", ctypes.c_void_p), ("g_final", ctypes.c_void_p), ("Wcls", ctypes.c_void_p),
        ("g_att", _PP), ("Wq", _PP), ("Wk", _PP), ("Wv", _PP), ("Wo", _PP), ("g_ffn", _PP),
        ("W1", _PP), ("W3", _PP), ("W2", _PP),
    ]


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        L.nb_new.restype = ctypes.c_void_p
        L.nb_new.argtypes = [ctypes.POINTER(_Weights)]
        L.nb_forward.restype = ctypes.c_int
        L.nb_forward.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p]
        L.nb_free.restype = None
        L.nb_free.argtypes = [ctypes.c_void_p]
        L.nb_has_neon.restype = ctypes.c_int
        _lib = L
    return _lib


def has_neon() -> bool:
    return bool(lib().nb_has_neon())


class Model:
    """One decode session of the host baseline over a borrowed blob."""

    def __init__(self, cfg: dict, blob: np.ndarray):
        from paper_2601_03324_gb300 import synth  # the input generator's layout only
        self._blob = blob
        tied = cfg.get("shared_classifier", 0) == 1
        L = int(cfg["n_layers"])

        def t(name, layer=-1):
            return ctypes.c_void_p(synth.tensor(blob, cfg, name, layer, tied).ctypes.data)

        self._arrays = {}
        for nm in ("g_att", "Wq", "Wk", "Wv", "Wo", "g_ffn", "W1", "W3", "W2"):
            arr = (ctypes.c_void_p * max(L, 1))()
            for l in range(L):
                arr[l] = t(nm, l).value
            self._arrays[nm] = arr
        w = _Weights(int(cfg["dim"]), int(cfg["hidden_dim"]), L, int(cfg["n_heads"]),
                     int(cfg["n_kv_heads"]), int(cfg["vocab_size"]), int(cfg["max_seq"]),
                     float(cfg.get("rope_theta", 10000.0)), float(cfg.get("norm_eps", 1e-5)),
                     t("E"), t("g_final"), t("Wcls"),
                     *[ctypes.cast(self._arrays[nm], _PP) for nm in
                       ("g_att", "Wq", "Wk", "Wv", "Wo", "g_ffn", "W1", "W3", "W2")])
        self._w = w
        self._h = lib().nb_new(ctypes.byref(w))
        if not self._h:
            raise MemoryError("nb_new failed")
        self.vocab = int(cfg["vocab_size"])

    def forward(self, token: int, pos: int) -> np.ndarray:
        out = np.empty(self.vocab, dtype=np.float32)
        rc = lib().nb_forward(self._h, int(token), int(pos), ctypes.c_void_p(out.ctypes.data))
        if rc != 0:
            raise ValueError(f"nb_forward failed with code {rc}")
        return out

    def close(self):
        if getattr(self, "_h", None):
            lib().nb_free(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
