#!/usr/bin/env python
"""Benchmark: batch-1 FP32 decode tokens/s of the 110M Llama-2-shape model.

A step is one decode step (all layers + classifier + greedy argmax) for one
token. The workload is greedy 256-step sequences from token 1 (the paper's
256-token run) with the weights resident in HBM. K timed steps are whole
sequences (one launch of the persistent decode kernel each) and, for the
K mod 256 steps left, one window of consecutive positions centred on the
sequence, so the timed steps have the sequence's mean KV length; an untimed
launch first decodes the whole sequence, which fills the KV cache and gives
the token each window starts from (greedy decoding is deterministic). The
positions timed are in config.positions; full_sequence times one whole
sequence on its own. Weights streamed per step (438 MB) exceed L2, so no L2
flush is needed between steps.

Printed JSON line (rank 0): value = tokens/s over all ranks; e2e = the same
metric through tvl_forward with host logits (token in, 128 KB of logits out,
host argmax, every step, the same positions); roofline of the decode kernel
against the measured HBM copy bandwidth; cpu_baseline = the CPU oracle with
float accumulators (the paper's scalar baseline) on one host core;
cpu_baseline_paper_method = the paper's NEON GEMV and RMSNorm on one host core.

--impl reference times the CPU oracle (the only reference this paper has; it
publishes no code) on the same workload and positions.

Multi-GPU (torchrun): replicas only — each rank decodes its own sequences; no
collective on the data path. value = all ranks' tokens / max rank time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import tempfile
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "batch-1 decode tokens/s (110M FP32); GEMV HBM GB/s vs ~8 TB/s peak"
METRIC_BATCH = "decode tokens/s, {b} sequences per step (110M FP32)"
BATCH_STARTS = [1, 100, 2000, 31999]  # first tokens of the sequences of a batched run
PAPER_TOKS = 61.3  # the paper's 110M FP32 decode on one M2 Pro core (Table 1)
SEQ = 256
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4096)
    ap.add_argument("--warmup", type=int, default=256)
    ap.add_argument("--impl", default="tvl", choices=["tvl", "reference"])
    ap.add_argument("--workload", default="110m", choices=["110m", "110m-long", "tiny", "7b"])
    ap.add_argument("--weights", default="f32", choices=["f32", "q8", "q4"],
                    help="q8 / q4: weight-only 8-bit / 4-bit rows (tvl_config.weight_bits)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--gemv-sweep", action="store_true", help="GEMV GB/s per shape instead")
    ap.add_argument("--hot", action="store_true",
                    help="with --gemv-sweep: one copy of W, so that W stays in L2 when it fits")
    ap.add_argument("--prefill", type=int, default=0,
                    help="time tvl_prefill of this many prompt tokens instead of decoding")
    ap.add_argument("--batch", type=int, default=1, choices=[1, 2, 3, 4],
                    help="sequences decoded together per launch (tvl_decode_greedy_batch)")
    return ap.parse_args()


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


# the sources the decode kernel is built from (a committed ncu capture of it
# stays valid while these are unchanged)
DECODE_SOURCES = ("decode_kernel.cuh", "stream_gemv.cuh", "ptx.cuh", "decode.cu",
                  "decode_batch.cu", "model.h", "host_common.h")


def kernel_hash() -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2601_03324_gb300", "csrc")
    for f in sorted(DECODE_SOURCES):
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(f.encode() + fh.read())
    return h.hexdigest()[:16]


def committed_traffic(workload: str, bytes_launch: int):
    """DRAM bytes of one launch of bytes_launch algorithmic bytes, from the
    committed ncu summary, if it was taken on the kernel sources as they are
    now. The capture covers a short launch; its read+write bytes are scaled by
    the ratio of algorithmic bytes (the traffic follows the bytes streamed)."""
    p = os.path.join(ROOT, "profiles", f"decode_kernel_{workload}.txt")
    if not os.path.exists(p):
        return None
    kv = {}
    for line in open(p):
        if ":" in line and not line.startswith("#"):
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    if kv.get("kernel_sources_sha256_16") != kernel_hash():
        return None
    try:
        dram = float(kv["dram_bytes_read"]) + float(kv["dram_bytes_write"])
        return dram * bytes_launch / float(kv["captured_algorithmic_bytes"])
    except (KeyError, ValueError, ZeroDivisionError):
        return None


def max_over_ranks(x: float, world: int, device: str) -> float:
    """The largest x over all ranks (the job's time is its slowest rank's)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(world: int, steps: int, max_ms: float) -> float:
    """Whole-job throughput: every rank decodes `steps` tokens of its own
    sequences (replicas), the job ends with its slowest rank."""
    return world * steps / (max_ms * 1e-3)


def step_bytes(cfg: dict, streamed: int, pos: int, batch: int = 1) -> int:
    """Algorithmic bytes of one step at position pos: every weight once (for
    all sequences of the batch), and per sequence the K/V cache rows of
    positions < pos, the new K/V row, the logits."""
    d, L, V = cfg["dim"], cfg["n_layers"], cfg["vocab_size"]
    kvd = cfg["n_kv_heads"] * (d // cfg["n_heads"])
    return streamed + batch * (2 * pos * kvd * 4 * L + 2 * kvd * 4 * L + 4 * V)


class Clocks:
    """nvidia-smi sampling during the timed region."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, dev_index: int, uuid: str | None):
        fd, self.path = tempfile.mkstemp(prefix="tvl_clocks_", suffix=".csv")
        self.f = os.fdopen(fd, "w")
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
               "-lms", "50"]
        cmd += ["-i", uuid] if uuid else ["-i", str(dev_index)]
        try:
            self.p = subprocess.Popen(cmd, stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None

    def _discard(self):
        self.f.close()
        try:
            os.remove(self.path)
        except OSError:
            pass

    def stop(self, t0: float, t1: float):
        if self.p is None:
            self._discard()
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.12)
        self.p.terminate()
        try:
            self.p.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.p.kill()
        self.f.close()
        with open(self.path) as fh:
            lines = fh.readlines()
        self._discard()
        rows = []
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                ts += float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                try:
                    pw = float(parts[3])
                except ValueError:
                    pw = None
                rows.append((ts, float(parts[1]), float(parts[2]), parts[5:9], pw))
            except (ValueError, IndexError):
                continue
        win = [r for r in rows if t0 - 0.06 <= r[0] <= t1 + 0.06] or rows[-3:]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in win for i, v in enumerate(r[3]) if v == "Active"})
        pws = [r[4] for r in win if r[4] is not None]
        return {"sm_mhz": statistics.median([r[1] for r in win]) if win else None,
                "sm_max_mhz": max(r[2] for r in win) if win else None,
                "reasons": reasons, "samples": len(win),
                "power_w": statistics.median(pws) if pws else None}


def timed_windows(seq: int, k: int, pos0: int):
    """(first position, steps) of each launch that times k steps of the
    workload's seq-step sequences from pos0: whole sequences, then the steps
    left as one window centred on the sequence, so that the timed steps have
    the sequence's mean KV length."""
    wins = [(pos0, seq)] * (k // seq)
    r = k % seq
    if r:
        wins.append((pos0 + (seq - r) // 2, r))
    return wins


def window_starts(wins, pos0: int, first, fill):
    """Start token(s) of each window: the sequence's first token(s) at pos0,
    else the greedy token(s) at that position from the fill run (fill[s] is
    the argmax after step s of the sequence)."""
    out = []
    for (p, n) in wins:
        out.append(list(first) if p == pos0 else [int(t) for t in np.atleast_1d(fill[p - pos0 - 1])])
    return out


def positions_of(wins):
    """config.positions: the distinct [first, last] position ranges timed."""
    seen = []
    for (p, n) in wins:
        r = [p, p + n - 1]
        if r not in seen:
            seen.append(r)
    return seen


def cpu_decode_rate(make, cfg, seconds: float):
    """A CPU decoder (make() -> object with forward(token, pos)) decoding
    greedily from token 1 for about `seconds`; tokens/s, steps, seconds."""
    m = make()
    t, n = 1, 0
    t0 = time.perf_counter()
    while True:
        lg = m.forward(t, n)
        t = int(np.argmax(lg))
        n += 1
        el = time.perf_counter() - t0
        if el >= seconds or n >= cfg["max_seq"]:
            break
    return n / el, n, el


WEIGHT_BITS = {"f32": 0, "q8": 8, "q4": 4}  # tvl_config.weight_bits of each --weights


def streamed_bytes_of(cfg: dict, weight_bits: int = 0) -> int:
    """Weight bytes one decode step reads: every matrix and gain of every
    layer, one embedding row, the final gain and the classifier (8-bit rows:
    16 + K bytes per row; 4-bit rows: 16 + K / 2)."""
    d, F, L, V = cfg["dim"], cfg["hidden_dim"], cfg["n_layers"], cfg["vocab_size"]
    kvd = cfg["n_kv_heads"] * (d // cfg["n_heads"])
    if weight_bits in (8, 4):
        rq = 16 + (d if weight_bits == 8 else d // 2)
        rf = 16 + (F if weight_bits == 8 else F // 2)
        return (L * ((d + 2 * kvd) * rq + d * rq + 2 * F * rq + d * rf + 8 * d) + V * rq + rq
                + 4 * d)
    return 4 * (L * ((d + 2 * kvd) * d + d * d + 3 * F * d + 2 * d) + V * d + 2 * d)


def l2_statement(streamed: int) -> str:
    """How the timed steps relate to L2 (the timing rule: inputs larger than L2,
    or say that they are not). GB300's L2 holds about 126 MB."""
    if streamed > 140e6:
        return (f"inputs larger than L2: every step streams {streamed / 1e6:.1f} MB of weights "
                f"(GB300 L2: about 126 MB), so no flush is needed between steps")
    return (f"weights fit in L2 ({streamed / 1e6:.1f} MB streamed per step; GB300 L2: about "
            f"126 MB) and are not flushed between the steps of a launch: the roofline against "
            f"HBM bandwidth understates this workload's bound (see roofline.l2)")


def workload_config(name, cfg, batch=1, weights="f32", positions=None):
    """The config object of the JSON line; both arms build it from the same
    arguments, so that the driver's same-config check holds."""
    desc = {"110m": "110M Llama-2-shape FP32 decoder (d768 L12 H12 F2048 V32000, tied), "
                    "batch 1, greedy 256-step sequences from token 1",
            "110m-long": "110M Llama-2-shape FP32 decoder (d768 L12 H12 F2048 V32000, tied), "
                         "batch 1, KV cache filled by one prefill of 896 prompt tokens "
                         "(uniform in [3, 31999], seed 3), greedy 128-step sequences at "
                         "positions 896..1023",
            "tiny": "tiny Llama-2-shape FP32 decoder (d288 L6 H6 F768 V32000, untied), batch 1, "
                    "greedy 64-step sequences from token 1",
            "7b": "7B Llama-2-shape FP32 decoder (d4096 L32 H32 F11008 V32000, untied), batch 1, "
                  "greedy 16-step sequences from token 1"}[name]
    seq = 128 if name == "110m-long" else min(cfg["steps"], cfg["max_seq"])
    if batch > 1:
        desc = desc.replace("batch 1, greedy", f"{batch} sequences per launch (first tokens "
                            f"{BATCH_STARTS[:batch]}), greedy").replace(" from token 1", "")
    return {"workload": desc, "seq_steps": seq, "batch": batch,
            "weights_seed": cfg["seed"], "parallelism": "replicas", "weights": weights,
            "positions": positions,
            "l2": l2_statement(streamed_bytes_of(cfg, 8 if weights == "q8" else 0))}


def run_reference(args, cfg, rank, world):
    """The CPU oracle (double accumulators, one host core) on the same
    positions as the GPU arm: an untimed greedy fill up to the last window's
    start, the warm-up steps, then the timed windows (or, when whole steps
    would take longer than about 150 s, the same fraction of every weight
    matrix's rows per step, scaled to whole steps)."""
    if rank != 0:
        return 0
    from paper_2601_03324_gb300 import synth
    import oracle
    blob = synth.make_blob(cfg)
    m = oracle.Model(cfg, blob, 64)
    seq, pos0 = min(cfg["steps"], cfg["max_seq"]), 0
    tok0 = 1
    if args.workload == "110m-long":
        prompt = synth.long_context_tokens()
        for p, t in enumerate(prompt):
            lg = m.forward(int(t), p)
        tok0, pos0, seq = int(np.argmax(lg)), len(prompt), cfg["max_seq"] - len(prompt)
    wins = timed_windows(seq, args.steps, pos0)
    fill, t = [], tok0
    for p in range(pos0, max(p for p, _ in wins)):
        t = int(np.argmax(m.forward(t, p)))
        fill.append(t)
    starts = window_starts(wins, pos0, [tok0], fill)
    wp, wn = wins[-1]
    for s in range(args.warmup):
        if s % wn == 0:
            t = starts[-1][0]
        t = int(np.argmax(m.forward(t, wp + s % wn)))
    t0 = time.perf_counter()
    m.forward(starts[0][0], wins[0][0])
    t_tok = time.perf_counter() - t0
    frac = min(1.0, 150.0 / max(1e-9, args.steps * t_tok))
    t0 = time.perf_counter()
    if frac >= 1.0:
        for (p, n), st in zip(wins, starts):
            t = st[0]
            for i in range(n):
                t = int(np.argmax(m.forward(t, p + i)))
        sample = (f"{args.steps} whole decode steps at the GPU arm's positions "
                  f"{positions_of(wins)} (greedy, after an untimed fill)")
    else:
        from paper_2601_03324_gb300 import synth as sy
        mats = [(n, l) for l in range(cfg["n_layers"])
                for n in ("Wq", "Wk", "Wv", "Wo", "W1", "W3", "W2")] + [("Wcls", -1)]
        xs = {}
        for s in range(args.steps):
            for (n, l) in mats:
                W = sy.tensor(blob, cfg, n, l)
                rows = max(1, int(math.ceil(frac * W.shape[0])))
                if W.shape[1] not in xs:
                    xs[W.shape[1]] = np.ones(W.shape[1])
                oracle.gemv(W[:rows], xs[W.shape[1]])
        sample = (f"each step: the oracle GEMV over {frac:.4f} of every weight matrix's rows "
                  f"(the GEMVs are the step's cost), scaled to whole steps")
    el = time.perf_counter() - t0
    val = args.steps * frac / el
    line = {"impl": "reference", "metric": METRIC, "value": val, "unit": "tokens/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * el / (args.steps * frac), "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": val / PAPER_TOKS if args.workload == "110m" else None, "dtype": "f64",
            "data": "synthetic (seeded N(0, 0.02) weights)",
            "config": workload_config(args.workload, cfg, 1, args.weights, positions_of(wins)),
            "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def gemv_sweep(args):
    import torch
    from paper_2601_03324_gb300 import synth, tvl
    torch.cuda.set_device(0)
    props = torch.cuda.get_device_properties(0)
    l2 = props.L2_cache_size
    s = torch.cuda.Stream()
    out = []
    uuid = getattr(props, "uuid", None)
    uuid = f"GPU-{uuid}" if uuid and not str(uuid).startswith("GPU-") else (str(uuid) if uuid else None)
    clocks = Clocks(0, uuid)
    t_wall0 = time.time()
    for i, (M, K) in enumerate(synth.GEMV_SHAPES):
        W, x = synth.gemv_operands(M, K, i)
        packed = {"q8": (tvl.tvl_q8_bytes, tvl.tvl_quantize_q8, tvl.tvl_gemv_q8),
                  "q4": (tvl.tvl_q4_bytes, tvl.tvl_quantize_q4, tvl.tvl_gemv_q4)}.get(args.weights)
        wbytes = packed[0](M, K) if packed else 4 * M * K
        nbytes = wbytes + 4 * (M + K)
        copies = 1 if args.hot else max(1, math.ceil(3 * l2 / wbytes))
        if packed:  # packed 8-bit or 4-bit rows of W, one copy per rotation slot
            dW1 = torch.from_numpy(W).cuda()
            dW = torch.empty((copies, wbytes), dtype=torch.uint8, device="cuda")
            for c in range(copies):
                packed[1](dW1.data_ptr(), dW[c].data_ptr(), M, K)
            torch.cuda.synchronize()
            del dW1
            call = packed[2]
        else:
            dW = torch.from_numpy(W).cuda().repeat(copies, 1).reshape(copies, M, K)
            call = tvl.tvl_gemv
        dx = torch.from_numpy(x).cuda()
        dy = torch.empty(M, device="cuda")
        reps = 200
        with torch.cuda.stream(s):
            for r in range(10):
                call(dW[r % copies].data_ptr(), dx.data_ptr(), dy.data_ptr(), M, K, s.cuda_stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                for r in range(reps):
                    call(dW[r % copies].data_ptr(), dx.data_ptr(), dy.data_ptr(), M, K,
                         s.cuda_stream)
            g.replay()
            s.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s)
            g.replay()
            e1.record(s)
        e1.synchronize()
        us = e0.elapsed_time(e1) * 1000.0 / reps
        out.append({"shape": [M, K], "us": us, "GB/s": nbytes / us / 1e3,
                    "copies": copies, "fits_l2": wbytes <= l2})
        del dW, g
    clk = clocks.stop(t_wall0, time.time())
    peak, src = measured_peaks()
    for o in out:
        o["frac_of_" + src + "_hbm"] = o["GB/s"] / peak
    mode = ("hot: one copy of W, resident in L2 when it fits (its GB/s is then an L2 figure, "
            "not an HBM one)" if args.hot else
            "cold: W rotated over copies totalling 3x L2, so every call reads it from HBM")
    print(json.dumps({"gemv_sweep": out, "weights": args.weights, "mode": mode,
                      "peak_gbs": peak, "peak_source": src, "reps_per_shape": 200,
                      "timing": "200 calls captured in one CUDA graph, CUDA events around "
                                "one replay, divided by 200",
                      "clocks": dict(clk, window="the whole sweep, set-up included")}),
          flush=True)


def prefill_bench(args, cfg):
    """tokens/s of tvl_prefill: a prompt of args.prefill seeded token ids
    (uniform in [3, 31999]) from position 0, one call per step, K calls timed
    with CUDA events after W warm-up calls. The products run on the tensor
    cores; the roofline is theirs: algorithmic FLOPs (2 per weight per
    position, plus the causal attention's 4 hd per query-key pair) per second,
    and the tensor pipe's share of the measured bf16 peak for the three bf16
    products each float32 product takes."""
    import torch
    from paper_2601_03324_gb300 import synth, tvl
    torch.cuda.set_device(0)
    n = int(args.prefill)
    blob = synth.make_blob(cfg)
    stream = torch.cuda.Stream()
    model = tvl.Model(cfg, blob, stream=stream.cuda_stream)
    info = model.info()
    prompt = synth.uniform_ints(n, synth.LONG_CONTEXT_SEED, 1, 3, 31999)
    host = np.empty(cfg["vocab_size"], dtype=np.float32)
    model.prefill(prompt, 0, host)  # first call: allocations, bf16 parts of the weights
    for _ in range(max(3, args.warmup)):
        model.prefill(prompt, 0)
    model.sync()
    props = torch.cuda.get_device_properties(0)
    uuid = getattr(props, "uuid", None)
    uuid = f"GPU-{uuid}" if uuid and not str(uuid).startswith("GPU-") else (str(uuid) if uuid else None)
    clocks = Clocks(0, uuid)
    time.sleep(0.15)
    t0 = time.time()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        model.prefill(prompt, 0)
    e1.record(stream)
    model.sync()
    clk = clocks.stop(t0, time.time())
    ms = e0.elapsed_time(e1) / args.steps
    d, F, L = cfg["dim"], cfg["hidden_dim"], cfg["n_layers"]
    kvd = cfg["n_kv_heads"] * (d // cfg["n_heads"])
    hd = d // cfg["n_heads"]
    w_layers = L * ((d + 2 * kvd) * d + d * d + 3 * F * d)
    flops = 2.0 * n * w_layers + 4.0 * hd * cfg["n_heads"] * L * n * (n + 1) / 2 + 2.0 * cfg["vocab_size"] * d
    achieved = flops / (ms * 1e-3) / 1e12
    pk = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))) if os.path.exists(
        os.path.join(ROOT, "MEASURED_PEAKS.json")) else {}
    bf16 = float(pk.get("bf16_tflops", 1900.0))
    line = {"metric": f"prefill tokens/s ({args.workload}, {n}-token prompt, FP32 accuracy)",
            "value": n / (ms * 1e-3), "unit": "tokens/s", "n_gpus": 1, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True,
            "dtype": "f32 (bf16 parts, fp32 accumulation)", "data": "synthetic (seeded N(0, 0.02) weights)",
            "config": {"workload": args.workload, "prompt_tokens": n, "weights_seed": cfg["seed"],
                       "l2": l2_statement(streamed_bytes_of(cfg))},
            "roofline": {"bound": "tensor", "achieved": achieved, "unit": "TFLOP/s",
                         "algorithmic_flops_per_call": flops,
                         "tensor_pipe_frac": 3 * 2.0 * n * w_layers / (ms * 1e-3) / 1e12 / bf16,
                         "peak_bf16": bf16,
                         "note": "achieved = float32-equivalent FLOPs per second; the tensor "
                                 "pipe runs three bf16 products for each (tensor_pipe_frac: "
                                 "their share of the measured bf16 peak)"},
            "clocks": clk, "grid": info.grid}
    print(json.dumps(line), flush=True)
    model.close()
    return 0


def main():
    args = parse()
    rank, local_rank, world = dist_env()
    from paper_2601_03324_gb300 import synth
    cfg = synth.model_config("110m" if args.workload == "110m-long" else args.workload)
    if args.impl == "reference":
        return run_reference(args, cfg, rank, world)
    import torch
    import torch.distributed as dist
    if args.gemv_sweep:
        return gemv_sweep(args)
    if args.prefill:
        return prefill_bench(args, cfg)
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local_rank)
    from paper_2601_03324_gb300 import tvl

    B = args.batch
    if B > 1 and (args.weights != "f32" or args.workload == "110m-long"):
        print(json.dumps({"error": "--batch > 1 needs --weights f32 and a workload other than "
                                   "110m-long"}))
        return 2
    blob = synth.make_blob(cfg)
    if args.weights in ("q8", "q4"):
        cfg = dict(cfg, weight_bits=WEIGHT_BITS[args.weights])
    if B > 1:
        cfg = dict(cfg, max_batch=B)
    stream = torch.cuda.Stream()
    model = tvl.Model(cfg, blob, stream=stream.cuda_stream)
    info = model.info()
    seq = min(cfg["steps"], cfg["max_seq"])  # the workload's greedy sequence length
    tok0, pos0 = 1, 0
    prefill = None
    if args.workload == "110m-long":
        # fill the KV cache with the 896-token prompt in one prefill call
        # (tvl_prefill; timed on its own, not part of the decode figure);
        # every timed sequence then decodes positions 896..1023 greedily
        prompt = synth.long_context_tokens()
        host = np.empty(cfg["vocab_size"], dtype=np.float32)
        model.prefill(prompt, 0, host)
        pe0, pe1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        pe0.record(stream)
        for _ in range(3):
            model.prefill(prompt, 0)
        pe1.record(stream)
        model.sync()
        pms = pe0.elapsed_time(pe1) / 3
        prefill = {"tokens": len(prompt), "ms": pms, "tokens_per_s": len(prompt) / pms * 1e3,
                   "note": "tvl_prefill of the prompt (tensor-core GEMMs in float32 accuracy "
                           "per layer), "
                           "mean of 3 calls"}
        tok0, pos0 = int(np.argmax(host)), len(prompt)
        seq = cfg["max_seq"] - pos0

    first = [tok0] if B == 1 else BATCH_STARTS[:B]

    def launch(starts, p, n):
        if B == 1:
            return model.decode_greedy(starts[0], p, n, tokens=False)
        return model.decode_greedy_batch(starts, p, n, tokens=False)

    def run_windows(wins, starts, events=None):
        """One launch per window; CUDA events around each when asked."""
        for (p, n), st in zip(wins, starts):
            if events is not None:
                e0 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
            launch(st, p, n)
            if events is not None:
                e1 = torch.cuda.Event(enable_timing=True)
                e1.record(stream)
                events.append((e0, e1, p, n))
        return len(wins)

    # untimed: the whole sequence once (fills the KV cache, gives the greedy
    # tokens the windows start from), then the warm-up steps
    fill = (model.decode_greedy(tok0, pos0, seq) if B == 1 else
            model.decode_greedy_batch(first, pos0, seq))
    wins = timed_windows(seq, args.steps, pos0)
    starts = window_starts(wins, pos0, first, fill)
    wwins = timed_windows(seq, max(3, args.warmup), pos0)
    run_windows(wwins, window_starts(wwins, pos0, first, fill))
    model.sync()
    props = torch.cuda.get_device_properties(local_rank)
    uuid = getattr(props, "uuid", None)
    uuid = f"GPU-{uuid}" if uuid and not str(uuid).startswith("GPU-") else (str(uuid) if uuid else None)
    clocks = Clocks(local_rank, uuid)
    time.sleep(0.15)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    ev = []
    t_wall0 = time.time()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    launches = run_windows(wins, starts, ev)
    end.record(stream)
    model.sync()
    torch.cuda.synchronize()
    t_wall1 = time.time()
    if world > 1:
        dist.barrier()
    el_ms = start.elapsed_time(end)
    clk = clocks.stop(t_wall0, t_wall1)
    el_ms = max_over_ranks(el_ms, world, "cuda")

    # roofline of the decode kernel: algorithmic bytes of every timed launch
    # over the sum of their CUDA-event durations
    per = [(a.elapsed_time(b), p, n) for (a, b, p, n) in ev]
    kern_ms = sum(t for t, p, n in per)
    bytes_timed = sum(step_bytes(cfg, info.streamed_bytes, p + i, B)
                      for (t, p, n) in per for i in range(n))
    bytes_launch = bytes_timed / len(per)
    peak, peak_src = measured_peaks()
    achieved = bytes_timed / (kern_ms * 1e-3) / 1e9
    traffic = committed_traffic(args.workload + ("" if args.weights == "f32" else "_" + args.weights) +
                                (f"_b{B}" if B > 1 else ""), bytes_launch)

    # one whole sequence on its own (not part of the timed region)
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(stream)
    launch(first, pos0, seq)
    f1.record(stream)
    model.sync()
    full_ms = f0.elapsed_time(f1)
    full_seq = {"positions": [pos0, pos0 + seq - 1], "ms_per_step": full_ms / seq,
                "tokens_per_s": B * seq / (full_ms * 1e-3),
                "roofline_frac": sum(step_bytes(cfg, info.streamed_bytes, pos0 + i, B)
                                     for i in range(seq)) / (full_ms * 1e-3) / 1e9 / peak,
                "note": "one launch of the whole greedy sequence after the timed region "
                        "(CUDA events on the model's stream)"}
    steps_ns = model.step_times(seq).astype(np.float64)
    dts = np.diff(steps_ns) / 1e3 if seq > 1 else np.array([full_ms * 1e3])

    # L2 roofline where the streamed weights fit in L2: the bandwidth of an
    # L2-resident buffer of the same size, measured on the spot. (Of the probes
    # tried — sum, row and column sums, amax, a copy, an in-place add — the
    # in-place add, reads and writes counted, gave the highest figure.)
    l2_roof = None
    if info.streamed_bytes <= 0.6 * props.L2_cache_size:
        buf = torch.empty(info.streamed_bytes // 4, dtype=torch.float32, device="cuda")
        buf.normal_()
        with torch.cuda.stream(stream):
            for _ in range(20):
                buf.add_(0.0)
            q0, q1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            q0.record(stream)
            reps = 200
            for _ in range(reps):
                buf.add_(0.0)
            q1.record(stream)
        stream.synchronize()
        l2_gbs = 2 * 4 * (info.streamed_bytes // 4) * reps / (q0.elapsed_time(q1) * 1e-3) / 1e9
        del buf
        l2_roof = {"peak": l2_gbs, "unit": "GB/s", "frac": achieved / l2_gbs,
                   "probe": f"in-place add over one {info.streamed_bytes / 1e6:.1f} MB float32 "
                            f"buffer kept in L2 ({reps} back-to-back passes, reads and writes "
                            f"counted, CUDA events)"}

    # end to end through the public API: token(s) in, host logits out, host
    # argmax, at the same positions as the timed launches
    e2e = None
    if not args.no_e2e:
        import torch as _t
        host_logits = _t.empty(B * cfg["vocab_size"], dtype=_t.float32, pin_memory=True).numpy()
        V = cfg["vocab_size"]
        k_e2e = min(args.steps, 2048)
        ewins = timed_windows(seq, k_e2e, pos0)
        estarts = window_starts(ewins, pos0, first, fill)

        def api_step(toks, p):
            if B == 1:
                model.forward(toks[0], p, host_logits)
            else:
                model.forward_batch(toks, p, host_logits)
            return [int(np.argmax(host_logits[b * V:(b + 1) * V])) for b in range(B)]

        toks = list(estarts[-1])
        for i in range(min(8, ewins[-1][1])):
            toks = api_step(toks, ewins[-1][0] + i)
        t0 = time.perf_counter()
        for (p, n), st in zip(ewins, estarts):
            toks = list(st)
            for i in range(n):
                toks = api_step(toks, p + i)
        e2e_s = time.perf_counter() - t0
        e2e = {"value": world * B * k_e2e / e2e_s, "unit": "tokens/s",
               "h2d_bytes_per_step": 4 * B, "d2h_bytes_per_step": 4 * B * V,
               "positions": positions_of(ewins),
               "note": ("tvl_forward" if B == 1 else "tvl_forward_batch") +
                       " per step: token(s) as launch arguments, logits to pinned host "
                       "memory, argmax on the host"}

    cpu = cpu_pm = None
    if rank == 0 and not args.no_cpu_baseline and args.workload in ("110m", "tiny"):
        import oracle
        wb = WEIGHT_BITS[args.weights]
        rate, n, el = cpu_decode_rate(lambda: oracle.Model(cfg, blob, 32, weight_bits=wb), cfg,
                                      args.cpu_seconds)
        cpu = {"value": rate, "unit": "tokens/s", "cores": 1, "kind": "oracle",
               "sample": f"first {n} greedy steps of the workload from token 1 ({el:.1f} s, "
                         f"float accumulators: the paper's scalar baseline, one thread)"}
        if wb == 0:
            import baseline
            rate, n, el = cpu_decode_rate(lambda: baseline.Model(cfg, blob), cfg,
                                          args.cpu_seconds / 2)
            cpu_pm = {"value": rate, "unit": "tokens/s", "cores": 1,
                      "kind": ("paper method: NEON float32x4 GEMV with four accumulators and "
                               "NEON RMSNorm" if baseline.has_neon() else
                               "paper method in plain C (this host has no NEON)"),
                      "sample": f"first {n} greedy steps of the workload from token 1 "
                                f"({el:.1f} s, one thread)"}

    value = job_tokens_per_s(world, args.steps, el_ms) * B
    # board energy per token (paper's energy section reports mJ/token): the
    # median board power sampled during the timed region times its duration
    energy = None
    if clk.get("power_w"):
        energy = {"power_w": clk["power_w"],
                  "mj_per_token": 1e3 * clk["power_w"] * (el_ms * 1e-3) / (args.steps * B),
                  "note": "nvidia-smi power.draw (board), median over the timed region"}
    streamed_cfg = streamed_bytes_of(cfg, WEIGHT_BITS[args.weights])
    assert streamed_cfg == info.streamed_bytes, (streamed_cfg, info.streamed_bytes)
    line = {
        "metric": METRIC if B == 1 else METRIC_BATCH.format(b=B), "value": value,
        "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": el_ms / args.steps,
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": (value / PAPER_TOKS
                        if args.workload == "110m" and args.weights == "f32" and B == 1 else None),
        "dtype": {"f32": "f32", "q8": "f32 activations, int8 weight rows",
                  "q4": "f32 activations, int4 weight rows"}[args.weights],
        "data": "synthetic (seeded N(0, 0.02) weights)",
        "config": workload_config(args.workload, cfg, B, args.weights, positions_of(wins)),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "kernel": "decode_kernel", "peak_source": peak_src,
                     "bytes_per_launch": bytes_launch, "bytes_timed": bytes_timed,
                     "launches": len(per), "kernel_ms": kern_ms, "l2": l2_roof},
        "full_sequence": full_seq,
        "cpu_baseline": cpu,
        "cpu_baseline_paper_method": cpu_pm,
        "e2e": e2e,
        "gpu_launches": launches,
        "clocks": clk,
        "step_latency_us": {"p50": float(np.percentile(dts, 50)),
                            "p90": float(np.percentile(dts, 90)),
                            "p99": float(np.percentile(dts, 99)),
                            "max": float(np.max(dts)), "std": float(np.std(dts)),
                            "source": "device timestamps at the end of each step of the "
                                      "whole-sequence launch (tvl_step_times)"},
        "energy": energy,
        "grid": info.grid, "ring_stages": info.ring_stages,
        "prefill": prefill,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    model.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main() or 0)
