"""Host-side logic of bench.py on CPU: the multi-rank aggregation (gloo,
world size 2) and the reference arm's rank handling. Replicas only: every rank
decodes its own sequences, so the only collective is the timing reduction."""
import argparse
import json
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", init_method="env://")
    try:
        env = bench.dist_env()
        # rank r took (r + 1) * 100 ms for its steps
        ms = bench.max_over_ranks(100.0 * (rank + 1), world, "cpu")
        q.put((rank, env, ms, bench.job_tokens_per_s(world, 512, ms)))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, env, ms, val in out:
        assert env == (rank, rank, 2)
        assert ms == 200.0                      # the slowest rank's time, on every rank
        assert val == pytest.approx(2 * 512 / 0.2)  # all ranks' tokens / max time


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5
    assert bench.job_tokens_per_s(1, 100, 50.0) == pytest.approx(2000.0)


def _ref_args(**kw):
    a = dict(gpus=2, steps=1, warmup=0, impl="reference", workload="tiny", no_e2e=False,
             no_cpu_baseline=False, cpu_seconds=1.0, gemv_sweep=False, weights="f32", batch=1)
    a.update(kw)
    return argparse.Namespace(**a)


def test_reference_arm_other_ranks_exit_without_work(capsys):
    import bench
    from paper_2601_03324_gb300 import synth
    cfg = synth.model_config("tiny")
    assert bench.run_reference(_ref_args(), cfg, rank=1, world=2) == 0
    assert capsys.readouterr().out == ""


def test_reference_arm_rank0_line(capsys):
    import bench
    from paper_2601_03324_gb300 import synth
    cfg = synth.model_config("tiny")
    assert bench.run_reference(_ref_args(), cfg, rank=0, world=2) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["n_gpus"] == 2
    assert line["value"] > 0 and line["unit"] == "tokens/s" and line["higher_is_better"]
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]


def test_timed_windows_keep_the_sequence_mean_position():
    import bench
    # 20 steps of a 256-step sequence: positions 118..137, mean 127.5
    assert bench.timed_windows(256, 20, 0) == [(118, 20)]
    for seq, k, pos0 in ((256, 20, 0), (256, 600, 0), (64, 20, 0), (128, 20, 896), (16, 20, 0),
                         (256, 256, 0), (256, 1, 0), (256, 255, 0)):
        wins = bench.timed_windows(seq, k, pos0)
        assert sum(n for _, n in wins) == k
        steps = [p + i for (p, n) in wins for i in range(n)]
        assert all(pos0 <= q < pos0 + seq for q in steps)
        # every window is consecutive positions inside one sequence, and the
        # timed steps' mean position is the sequence's (up to half a step)
        assert abs(sum(steps) / k - (pos0 + (seq - 1) / 2)) <= 0.5


def test_window_start_tokens_come_from_the_fill_run():
    import numpy as np
    import bench
    fill = np.arange(1000, 1256)  # fill[s] = the greedy token after step s
    wins = [(0, 256), (118, 20)]
    assert bench.window_starts(wins, 0, [1], fill) == [[1], [1117]]
    fillb = np.stack([fill, fill + 5000], axis=1)  # two sequences
    assert bench.window_starts([(118, 20)], 0, [1, 100], fillb) == [[1117, 6117]]
    assert bench.positions_of([(0, 256), (0, 256), (118, 20)]) == [[0, 255], [118, 137]]


def test_reference_arm_config_equals_the_gpu_arms(capsys):
    import bench
    from paper_2601_03324_gb300 import synth
    cfg = synth.model_config("tiny")
    assert bench.run_reference(_ref_args(steps=3, gpus=1), cfg, rank=0, world=1) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    wins = bench.timed_windows(64, 3, 0)
    assert line["config"] == bench.workload_config("tiny", cfg, 1, "f32", bench.positions_of(wins))
    assert line["config"]["positions"] == [[30, 32]]


def test_streamed_bytes_per_step_by_weight_format():
    # The weights one decode step reads, worked out by hand for the 110M shape
    # (d 768, L 12, F 2048, V 32000, tied): float32 rows 4 bytes a value;
    # quantized rows 16 bytes of scale and padding plus the codes (K bytes for
    # 8-bit, K / 2 for 4-bit); the gains, one embedding row and the final gain
    # stay float32 (4-bit: (2304 + 768 + 4096) * 400 + 768 * 1040 + 8 * 768 =
    # 3,672,064 bytes per layer; 12 layers, then 32000 classifier rows of 400
    # bytes, one embedding row of 400 and the final gain's 3072).
    import bench
    from paper_2601_03324_gb300 import synth
    cfg = synth.model_config("110m")
    assert bench.streamed_bytes_of(cfg, 0) == 4 * (12 * (2304 * 768 + 768 * 768 + 3 * 2048 * 768
                                                        + 2 * 768) + 32000 * 768 + 2 * 768)
    assert bench.streamed_bytes_of(cfg, 0) == 438_122_496
    assert bench.streamed_bytes_of(cfg, 8) == 12 * ((2304 + 768 + 4096) * 784 + 768 * 2064
                                                    + 8 * 768) + 32000 * 784 + 784 + 3072
    assert bench.streamed_bytes_of(cfg, 4) == 12 * 3_672_064 + 32000 * 400 + 400 + 3072
    assert bench.streamed_bytes_of(cfg, 4) == 56_868_240
