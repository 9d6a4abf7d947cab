"""Shared helpers of the GPU parity tests (oracle on the CPU vs libtvl on the GPU)."""
from __future__ import annotations

import numpy as np

import oracle
from paper_2601_03324_gb300 import synth

LOGIT_RTOL = 2e-3   # per step: max |d logit| <= 2e-3 * max |logit|
GEMV_RTOL = 1e-4    # per output: |d y_i| <= 1e-4 * sum_j |W_ij x_j|
MARGIN = 1e-2       # greedy tokens must agree where the top-2 margin exceeds this


def top2_margin(lg: np.ndarray) -> float:
    t = np.partition(lg, -2)[-2:]
    return float(t[1] - t[0])


def assert_logits_close(got: np.ndarray, ref: np.ndarray, where: str = ""):
    err = float(np.abs(got.astype(np.float64) - ref).max())
    tol = LOGIT_RTOL * float(np.abs(ref).max())
    assert err <= tol, f"{where}: max |d logit| {err:.3e} > {tol:.3e}"
    if top2_margin(ref) > MARGIN:
        assert int(np.argmax(got)) == int(np.argmax(ref)), f"{where}: argmax differs"


def teacher_forced(model, ref: "oracle.Model", tokens, start_pos: int = 0, check_every: int = 1,
                   label: str = ""):
    """Feed the same tokens to the GPU model and the oracle; compare logits."""
    out = np.empty(ref.vocab, dtype=np.float32)
    worst = 0.0
    for i, t in enumerate(tokens):
        p = start_pos + i
        lg = ref.forward(int(t), p)
        model.forward(int(t), p, out)
        if i % check_every == 0 or i == len(tokens) - 1:
            assert_logits_close(out, lg, f"{label} pos {p}")
            worst = max(worst, float(np.abs(out - lg).max() / np.abs(lg).max()))
    return worst


def lockstep_greedy(model, ref: "oracle.Model", start: int, n_steps: int, start_pos: int = 0,
                    check_every: int = 1, label: str = ""):
    """The oracle decodes greedily; the GPU model is fed the oracle's tokens
    (teacher forcing) and its logits are compared. Returns (tokens fed,
    oracle logits, worst relative error)."""
    out = np.empty(ref.vocab, dtype=np.float32)
    toks, logits, worst = [], [], 0.0
    t = int(start)
    for i in range(n_steps):
        p = start_pos + i
        lg = ref.forward(t, p)
        model.forward(t, p, out)
        if i % check_every == 0 or i == n_steps - 1:
            assert_logits_close(out, lg, f"{label} pos {p}")
            worst = max(worst, float(np.abs(out - lg).max() / np.abs(lg).max()))
        toks.append(t)
        logits.append(lg)
        t = int(np.argmax(lg))
    return toks, logits, worst


def compare_greedy(gen, ref_tokens, ref_logits):
    """Device greedy tokens vs the oracle's: equal until the first step whose
    oracle top-2 margin is within MARGIN (after that the paths may diverge)."""
    for s in range(len(gen)):
        if top2_margin(ref_logits[s]) <= MARGIN:
            return s
        assert int(gen[s]) == int(ref_tokens[s]), f"greedy step {s}: {gen[s]} != {ref_tokens[s]}"
    return len(gen)


def small_config(**kw) -> dict:
    cfg = dict(dim=64, hidden_dim=96, n_layers=2, n_heads=4, n_kv_heads=4, vocab_size=1000,
               max_seq=64, rope_theta=10000.0, norm_eps=1e-5, shared_classifier=0)
    cfg.update(kw)
    return cfg


def gemv_bound(W: np.ndarray, x: np.ndarray) -> np.ndarray:
    return GEMV_RTOL * (np.abs(W.astype(np.float64)) @ np.abs(x.astype(np.float64)))
