"""Seeded synthetic inputs for the decode step: model blobs, GEMV operands, token ids.

This module draws random numbers and lays them out; it holds none of the
decode step's arithmetic. Tests of both the CPU oracle and the CUDA path, and
the benchmark, take their inputs from here, so both sides see the same bytes.

The random numbers come from ``rng.c`` (counter-based splitmix64 streams and
Box-Muller normals, one stream per tensor); the packed blob layout below is
this module's own statement of the format that the library loads: float32
row-major tensors, each starting at a 128-byte-aligned offset, in the order

    E[V x d]; per layer: g_att[d], Wq[d x d], Wk[kvd x d], Wv[kvd x d],
    Wo[d x d], g_ffn[d], W1[F x d], W3[F x d], W2[d x F]; g_final[d];
    Wcls[V x d] unless the classifier is tied to E.

Matrices are drawn N(0, 0.02^2) and RMSNorm gains 1 + N(0, 0.01^2); padding is
zero. Tensor k of the blob (in the order above, counting from 0) uses stream k.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rng.c")
_LIB = os.path.join(_HERE, "libtvl_synth.so")
_lib = None

# Named workloads: the shapes and seeds of the paper's model family.
WORKLOADS = {
    # ~15M-parameter tiny decoder, untied classifier, seed 0, 64 greedy steps
    "tiny": dict(dim=288, hidden_dim=768, n_layers=6, n_heads=6, n_kv_heads=6,
                 vocab_size=32000, max_seq=256, rope_theta=10000.0, norm_eps=1e-5,
                 shared_classifier=0, seed=0, steps=64),
    # the paper's 110M shape (tied classifier, like its stories110M model), seed 2
    "110m": dict(dim=768, hidden_dim=2048, n_layers=12, n_heads=12, n_kv_heads=12,
                 vocab_size=32000, max_seq=1024, rope_theta=10000.0, norm_eps=1e-5,
                 shared_classifier=1, seed=2, steps=256),
    # 7B shape, untied classifier, seed 4, 16 greedy steps (~27 GB of weights)
    "7b": dict(dim=4096, hidden_dim=11008, n_layers=32, n_heads=32, n_kv_heads=32,
               vocab_size=32000, max_seq=2048, rope_theta=10000.0, norm_eps=1e-5,
               shared_classifier=0, seed=4, steps=16),
}

# Standalone GEMV sweep shapes (d_out, d_in), seed 1.
GEMV_SHAPES = [(768, 768), (2048, 768), (768, 2048), (32000, 768), (11008, 4096),
               (4096, 11008), (32000, 4096)]
GEMV_SEED = 1
LONG_CONTEXT_SEED = 3  # token ids of the 110M long-context workload


def build(force: bool = False) -> str:
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-pthread",
               "-o", _LIB + ".tmp", _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(_LIB + ".tmp", _LIB)
    return _LIB


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        u64, i64, i32, dbl = ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32, ctypes.c_double
        L.tvl_synth_fill_normal.restype = None
        L.tvl_synth_fill_normal.argtypes = [ctypes.c_void_p, i64, u64, u64, dbl, dbl, ctypes.c_int]
        L.tvl_synth_uniform_ints.restype = None
        L.tvl_synth_uniform_ints.argtypes = [ctypes.c_void_p, i64, u64, u64, i32, i32]
        L.tvl_synth_draw.restype = u64
        L.tvl_synth_draw.argtypes = [u64, u64, u64]
        L.tvl_synth_normal_at.restype = dbl
        L.tvl_synth_normal_at.argtypes = [u64, u64, u64]
        L.tvl_synth_splitmix64.restype = u64
        L.tvl_synth_splitmix64.argtypes = [u64, u64]
        L.tvl_synth_key.restype = u64
        L.tvl_synth_key.argtypes = [u64, u64]
        _lib = L
    return _lib


def _threads() -> int:
    return max(1, min(64, os.cpu_count() or 1))


def fill_normal(out: np.ndarray, seed: int, stream: int, mean: float = 0.0,
                std: float = 1.0) -> np.ndarray:
    """Fill a contiguous float32 array in place from stream (seed, stream)."""
    assert out.dtype == np.float32 and out.flags["C_CONTIGUOUS"]
    lib().tvl_synth_fill_normal(ctypes.c_void_p(out.ctypes.data), out.size, seed, stream,
                                mean, std, _threads())
    return out


def normal(shape, seed: int, stream: int, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    return fill_normal(np.empty(shape, dtype=np.float32), seed, stream, mean, std)


def uniform_ints(n: int, seed: int, stream: int, lo: int, hi: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    lib().tvl_synth_uniform_ints(ctypes.c_void_p(out.ctypes.data), n, seed, stream, lo, hi)
    return out


# ---- blob layout ----------------------------------------------------------------

def _a128(b: int) -> int:
    return (b + 127) // 128 * 128


def layout(cfg: dict, tied: bool | None = None):
    """List of (name, layer, byte offset, shape, kind) in blob order, and total bytes.

    kind is "matrix" (N(0, 0.02^2)) or "gain" (1 + N(0, 0.01^2)).
    """
    if tied is None:
        tied = bool(cfg.get("shared_classifier", 0) == 1)
    d, F, V = cfg["dim"], cfg["hidden_dim"], cfg["vocab_size"]
    hd = d // cfg["n_heads"]
    kvd = cfg["n_kv_heads"] * hd
    ents = []
    off = 0

    def take(name, layer, shape, kind):
        nonlocal off
        n = int(np.prod(shape))
        ents.append((name, layer, off, tuple(shape), kind))
        off = _a128(off + 4 * n)

    take("E", -1, (V, d), "matrix")
    for l in range(cfg["n_layers"]):
        take("g_att", l, (d,), "gain")
        take("Wq", l, (d, d), "matrix")
        take("Wk", l, (kvd, d), "matrix")
        take("Wv", l, (kvd, d), "matrix")
        take("Wo", l, (d, d), "matrix")
        take("g_ffn", l, (d,), "gain")
        take("W1", l, (F, d), "matrix")
        take("W3", l, (F, d), "matrix")
        take("W2", l, (d, F), "matrix")
    take("g_final", -1, (d,), "gain")
    if not tied:
        take("Wcls", -1, (V, d), "matrix")
    return ents, off


def blob_bytes(cfg: dict, tied: bool | None = None) -> int:
    return layout(cfg, tied)[1]


def make_blob(cfg: dict, seed: int | None = None, tied: bool | None = None,
              out: np.ndarray | None = None) -> np.ndarray:
    """The packed weight blob of a synthetic model, as a float32 array.

    ``out`` may be a preallocated float32 buffer (e.g. pinned or mmap'd) of the
    right size; it is filled in place.
    """
    if seed is None:
        seed = int(cfg.get("seed", 0))
    ents, total = layout(cfg, tied)
    assert total % 4 == 0
    if out is None:
        out = np.empty(total // 4, dtype=np.float32)
    assert out.dtype == np.float32 and out.size == total // 4
    end_prev = 0
    for k, (name, layer, off, shape, kind) in enumerate(ents):
        if off > end_prev:
            out[end_prev // 4: off // 4] = 0.0
        n = int(np.prod(shape))
        view = out[off // 4: off // 4 + n]
        if kind == "gain":
            fill_normal(view, seed, k, 1.0, 0.01)
        else:
            fill_normal(view, seed, k, 0.0, 0.02)
        end_prev = off + 4 * n
    if total > end_prev:
        out[end_prev // 4:] = 0.0
    return out


def tensor(blob: np.ndarray, cfg: dict, name: str, layer: int = -1,
           tied: bool | None = None) -> np.ndarray:
    """A view of one tensor of a blob."""
    ents, _ = layout(cfg, tied)
    for (nm, l, off, shape, kind) in ents:
        if nm == name and l == layer:
            n = int(np.prod(shape))
            return blob[off // 4: off // 4 + n].reshape(shape)
    if name == "Wcls":
        return tensor(blob, cfg, "E", -1, tied)
    raise KeyError((name, layer))


def gemv_operands(d_out: int, d_in: int, index: int, seed: int = GEMV_SEED):
    """W ~ N(0, 0.02^2) [d_out x d_in] and x ~ N(0, 1) [d_in] for sweep shape `index`."""
    W = normal((d_out, d_in), seed, 2 * index, 0.0, 0.02)
    x = normal((d_in,), seed, 2 * index + 1, 0.0, 1.0)
    return W, x


def long_context_tokens(n: int = 896, seed: int = LONG_CONTEXT_SEED) -> np.ndarray:
    """Token ids uniform in [3, 31999] for the 110M long-context workload."""
    return uniform_ints(n, seed, 0, 3, 31999)


def model_config(name: str, **overrides) -> dict:
    cfg = dict(WORKLOADS[name])
    cfg.update(overrides)
    return cfg
