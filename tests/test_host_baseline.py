"""The host-side timing baseline (the paper's NEON method, or its plain-C form off
aarch64) computes the same decode step as the oracle, within the decode
tolerances, so that its tokens/s in the bench line time the same work."""
import numpy as np

import baseline
import oracle
from paper_2601_03324_gb300 import synth

from helpers import assert_logits_close


def test_host_baseline_matches_the_oracle_under_teacher_forcing():
    cfg = synth.model_config("tiny", n_layers=2, vocab_size=2000, max_seq=32)
    blob = synth.make_blob(cfg, seed=5)
    ref = oracle.Model(cfg, blob)
    toks, logits = ref.greedy(1, 12)
    nb = baseline.Model(cfg, blob)
    for p, (t, lg) in enumerate(zip(toks, logits)):
        assert_logits_close(nb.forward(t, p), lg, f"host baseline pos {p}")


def test_host_baseline_tied_classifier_and_grouped_heads():
    cfg = dict(dim=64, hidden_dim=96, n_layers=2, n_heads=4, n_kv_heads=2, vocab_size=500,
               max_seq=16, rope_theta=10000.0, norm_eps=1e-5, shared_classifier=1)
    blob = synth.make_blob(cfg, seed=9)
    ref = oracle.Model(cfg, blob)
    nb = baseline.Model(cfg, blob)
    for p, t in enumerate([3, 77, 12, 499, 0, 250]):
        assert_logits_close(nb.forward(t, p), ref.forward(t, p), f"tied/GQA pos {p}")


def test_host_baseline_odd_widths_take_the_tail_loops():
    # dim 36 (9 float4, not a multiple of 16) and hidden 70 (not a multiple of 4)
    cfg = dict(dim=36, hidden_dim=70, n_layers=1, n_heads=3, n_kv_heads=3, vocab_size=97,
               max_seq=8, rope_theta=10000.0, norm_eps=1e-5, shared_classifier=0)
    blob = synth.make_blob(cfg, seed=4)
    ref = oracle.Model(cfg, blob)
    nb = baseline.Model(cfg, blob)
    for p, t in enumerate([5, 6, 90]):
        got = nb.forward(t, p)
        assert np.isfinite(got).all()
        assert_logits_close(got, ref.forward(t, p), f"odd widths pos {p}")
