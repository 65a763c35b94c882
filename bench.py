#!/usr/bin/env python3
"""Benchmark of the rollout hot path on GB300: a Qwen3-8B-shaped bf16 decoder
(random init) decoding a teacher-forced batch of 16 rollouts, prompt 512 tokens
then 1024 decode steps with per-token log-probs.

One step = one whole rollout (prefill of 16 x 512 tokens + 1024 decode steps of
16 tokens each).  `value` = decoded tokens per second over all ranks (replicas:
every rank runs its own rollout batch; no collective on the data path).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

`--impl reference` times the fp64 CPU oracle on a bounded sample of the same
workload (the only comparison program this method has).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode tokens/s and prefill/score tokens/s on 1 GB300; % HBM / bf16 roofline"
UNIT = "tokens/s"
B, P, N = 16, 512, 1024
WORKLOAD = ("qwen3-8b-shaped bf16 rollout decode: batch 16, prompt 512 random tokens, "
            "1024 teacher-forced decode steps, per-token log-probs")
ORACLE_TOKENS = 32  # tokens of rollout row 0 the CPU oracle scores per sample
# Scoring 32 x 4096 (all 36 layers): linear layers 2 * 131072 * 6.946e9 params, lm_head over
# 4095 scored positions per row (the kernel evaluates all 4096), causal attention.
SCORE_FLOPS = (2 * 32 * 4096 * (36 * 192937984) + 2 * 32 * 4096 * 151936 * 4096
               + 36 * 32 * 32 * 2 * 2 * 128 * (4096 * 4097 // 2))


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    return ap.parse_args()


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(v: float, world: int) -> float:
    """Largest value over the ranks (the job's time is its slowest replica's)."""
    if world == 1:
        return v
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_tokens(vocab: int, rank: int):
    """Rollout batch of replica `rank`: its own seeded token stream (weights are shared)."""
    import synth
    return synth.tokens((B, P + N + 1), vocab, stream=rank)


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms while running."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.path = tempfile.mktemp(suffix=".csv")
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(device_index)],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) >= 9:
                rows.append(f)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        load = [v for v in sm if mx and v > 0.5 * max(mx)] or sm
        return {"sm_mhz": statistics.median(load) if load else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows),
                "power_w_max": max((num(r[3]) or 0.0) for r in rows)}


def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        return None


def source_sha(paths):
    h = hashlib.sha256()
    for p in paths:
        h.update(open(os.path.join(ROOT, p), "rb").read())
    return h.hexdigest()[:16]


def recorded_traffic(key: str):
    """DRAM bytes per launch from a committed ncu summary, if the kernel source is unchanged."""
    try:
        t = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))[key]
    except (OSError, ValueError, KeyError):
        return None
    if source_sha(t["sources"]) != t["source_sha"]:
        return None
    return t["dram_bytes_per_launch"]


# --------------------------------------------------------------------------- CPU oracle sample
def oracle_sample(s, W, seq_row):
    """fp64 oracle: full causal forward + log-probs over the first ORACLE_TOKENS tokens."""
    import oracle
    t0 = time.perf_counter()
    lp, _, _ = oracle.score_sequence(s, W, seq_row[:ORACLE_TOKENS + 1])
    dt = time.perf_counter() - t0
    return ORACLE_TOKENS / dt, dt, lp


def cpu_cores():
    n = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return int(os.environ.get("OPENBLAS_NUM_THREADS", n))


def cpu_baseline_entry(value, dt):
    return {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
            "sample": (f"fp64 oracle: causal forward and per-token log-probs of the first "
                       f"{ORACLE_TOKENS} tokens of rollout row 0 (all 36 layers + lm_head; "
                       f"weights widened from bf16 layer by layer), {dt:.1f} s")}


# --------------------------------------------------------------------------- arms
def run_reference(args, world, rank):
    if rank != 0:
        return
    import synth
    s = synth.shape("q8b")
    W = synth.LazyWeights(s, cache=True)
    seq = synth.tokens((B, P + N + 1), s.vocab)
    times = []
    for i in range(args.warmup + args.steps):
        _, dt, _ = oracle_sample(s, W, seq[0])
        if i >= args.warmup:
            times.append(dt)
    dt = statistics.mean(times)
    value = ORACLE_TOKENS / dt
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": WORKLOAD, "sample_tokens": ORACLE_TOKENS},
            "cpu_baseline": cpu_baseline_entry(value, dt),
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_ours(args, world, rank, local):
    import numpy as np
    import torch

    import synth
    from paper_2609_12471_gb300 import build as qkbuild
    qkbuild.build()
    import paper_2609_12471_gb300 as qk
    from paper_2609_12471_gb300.runtime import Decoder

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    s = synth.shape("q8b")
    want_cpu = rank == 0 and world == 1 and not args.no_cpu_baseline
    W = synth.LazyWeights(s, cache=want_cpu)
    names = [t[0] for t in synth.tensor_list(s)]
    dec = Decoder(qk.qk_config_preset("q8b"), (W[n] for n in names), device=dev)
    seq = replica_tokens(s.vocab, rank)
    seq_d = torch.tensor(seq, dtype=torch.int32, device=dev)
    kv = dec.new_kv(B, P + N)
    lp = torch.empty(B, N + 1, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        dec.rollout(kv, B, P + N, seq_d, P, logprobs=lp)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    if dec.check_status() != 0:
        raise RuntimeError("device status flags set during warm-up")

    # ---- timed region: K whole rollouts, device-resident inputs
    n_layers = s.n_layers
    qk.qk_profile_begin(dec.handle, qk.QK_PROF_GATE_UP, args.steps * N * n_layers)
    clocks = ClockSampler(local)
    barrier(world)
    torch.cuda.synchronize(dev)
    launches0 = qk.qk_launch_count()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    launches = qk.qk_launch_count() - launches0
    barrier(world)
    clk = clocks.stop()
    ms = e0.elapsed_time(e1)
    ms_step = max_over_ranks(ms / args.steps, world)
    prof_ms, prof_n = qk.qk_profile_end(dec.handle)
    if dec.check_status() != 0:
        raise RuntimeError("device status flags set during the timed region")
    value = world * B * N / (ms_step / 1e3)

    # ---- prefill alone (for the prefill tokens/s figure), warmed up first: its workspace
    # kind differs from the rollout's
    pz = torch.empty(B, dtype=torch.float32, device=dev)

    def prefill():
        dec.prefill(kv, B, P + N, seq_d[:, :P].contiguous(), 0, None, seq_d[:, P].contiguous(), pz)

    for _ in range(2):
        prefill()
    torch.cuda.synchronize(dev)
    p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    p0.record(stream)
    for _ in range(args.steps):
        prefill()
    p1.record(stream)
    torch.cuda.synchronize(dev)
    prefill_ms = p0.elapsed_time(p1) / args.steps

    # ---- end to end through the public API with host buffers
    seq_h = torch.from_numpy(seq).pin_memory()
    lp_h = torch.empty(B, N + 1, dtype=torch.float32).pin_memory()
    seq_dev = torch.empty_like(seq_d)
    torch.cuda.synchronize(dev)
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        seq_dev.copy_(seq_h, non_blocking=True)
        dec.rollout(kv, B, P + N, seq_dev, P, logprobs=lp)
        lp_h.copy_(lp, non_blocking=True)
        torch.cuda.synchronize(dev)
    e2e_s = max_over_ranks((time.perf_counter() - t0) / args.steps, world)
    e2e_value = world * B * N / e2e_s
    lp_np = lp_h.numpy()
    if not (np.all(np.isfinite(lp_np)) and np.all(lp_np <= 1e-4)):
        raise RuntimeError("log-probs out of range")

    # ---- scoring pass (teacher-forced log-probs of 32 x 4096 tokens): secondary figure
    SB, ST = 32, 4096
    score_tok = torch.tensor(synth.tokens((SB, ST), s.vocab, stream=100 + rank), dtype=torch.int32,
                             device=dev)
    score_lp = torch.empty(SB, ST - 1, dtype=torch.float32, device=dev)
    dec.score(score_tok, logprobs=score_lp)  # warm-up
    torch.cuda.synchronize(dev)
    s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n_score = 2
    s0.record(stream)
    for _ in range(n_score):
        dec.score(score_tok, logprobs=score_lp)
    s1.record(stream)
    torch.cuda.synchronize(dev)
    score_s = max_over_ranks(s0.elapsed_time(s1) / n_score / 1e3, world)
    if dec.check_status() != 0 or not torch.isfinite(score_lp).all():
        raise RuntimeError("scoring produced invalid output")
    del score_tok, score_lp
    dec._ws.clear()
    torch.cuda.empty_cache()
    decode_configs = other_decode_configs(dec, dev, stream, rank)
    backward = backward_config(dec, dev, stream, rank, world)

    if rank != 0:
        return
    peaks = measured_peaks()
    hbm_peak = peaks["hbm_gbs"] if peaks else 6800.0
    bf16_peak = peaks["bf16_tflops"] if peaks else 1900.0
    c = dec.cfg
    if prof_n < 1:
        raise RuntimeError("no gate/up launch was bracketed")
    gu_bytes = 2 * c.intermediate * c.hidden * 2 + B * c.hidden * 2 + B * c.intermediate * 2
    avg_launch_s = (prof_ms / prof_n) / 1e3
    achieved = gu_bytes / avg_launch_s / 1e9
    roofline = {"bound": "hbm", "kernel": "decode gate/up linear (tcgen05 stream-K GEMM, 16 token rows)",
                "timed_launches": "the gate/up launches of each timed rollout's first decode step "
                                  "(later steps replay a captured CUDA graph without event nodes)",
                "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                "frac": achieved / hbm_peak,
                "peak_source": "measured" if peaks else "fallback",
                "algorithmic_bytes_per_launch": gu_bytes, "launches_timed": prof_n,
                "avg_launch_us": avg_launch_s * 1e6,
                "traffic": recorded_traffic("gate_up_decode_b16")}
    step_bytes = 15136811008 + B * sum(P + j + 1 for j in range(N)) * 147456 / N
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD, "batch": B, "prompt_tokens": P, "decode_steps": N,
                       "l2": "inputs larger than L2: 15.1 GB of weights streamed per decode step",
                       "replicas": world},
            "prefill_tokens_per_s": world * B * P / (prefill_ms / 1e3),
            "score_tokens_per_s": world * SB * ST / score_s,
            "score_roofline": {"bound": "tensor", "workload": "scoring 32 x 4096 tokens",
                               "flops_per_call": SCORE_FLOPS,
                               "achieved": SCORE_FLOPS / score_s / 1e12,
                               "peak": bf16_peak, "unit": "TFLOP/s",
                               "frac": SCORE_FLOPS / score_s / 1e12 / bf16_peak,
                               "peak_source": "measured (burst)" if peaks else "fallback"},
            "decode_hbm_fraction_of_8tbs": (step_bytes * N / 1e9) / ((ms_step - prefill_ms) / 1e3) / 8000.0,
            "decode_configs": decode_configs,
            "backward": backward,
            "roofline": roofline, "clocks": clk, "gpu_launches": int(launches),
            "launches_before_timed": int(launches0),
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(seq.nbytes),
                    "d2h_bytes_per_step": int(lp_h.numel() * 4)}}
    if want_cpu:
        v, dt, _ = oracle_sample(s, W, seq[0])
        line["cpu_baseline"] = cpu_baseline_entry(v, dt)
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- other decode configs
LAYER_WEIGHT_BYTES = 385875968        # one Qwen3-8B layer: qkv, o, gate/up, down (bf16)
STEP_WEIGHT_BYTES = 15136811008       # 36 layers + lm_head + norms
KV_BYTES_PER_TOKEN_LAYER = 4096       # K and V of 8 kv heads x 128 dims, bf16
KV_BYTES_PER_TOKEN = 36 * KV_BYTES_PER_TOKEN_LAYER


def _hbm_entry(bytes_per_step, step_s, hbm_peak, tokens_per_step):
    gbs = bytes_per_step / step_s / 1e9
    return {"tokens_per_s": tokens_per_step / step_s, "us_per_step": step_s * 1e6,
            "bytes_per_step": int(bytes_per_step), "achieved_gbs": gbs,
            "frac_of_measured_hbm": gbs / hbm_peak, "frac_of_8tbs": gbs / 8000.0}


def _event_time(fn, reps, stream):
    import torch
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        fn()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / 1e3 / reps


def other_decode_configs(dec, dev, stream, rank):
    """Decode throughput of the other decode workloads, each against its HBM roofline
    (weight + KV bytes per step):
      * batch-1 rollout decode of the 36-layer model (prompt 512, 256 teacher-forced steps);
      * one 8B layer's decode step at batch 1 / 8 / 32 / 64 over a 2048-entry N(0, 1) cache
        (new token at position 2048; layer 0 of the loaded model);
      * the 36-layer model at batch 64 over a long cache (N(0, 1) entries), decode steps at
        positions 4096, 6144 and 8191 (KV context 4097 .. 8192)."""
    import torch
    import synth
    from paper_2609_12471_gb300 import _binding as qkb
    peaks = measured_peaks()
    hbm = peaks["hbm_gbs"] if peaks else 6800.0
    gen = torch.Generator(device=dev)
    gen.manual_seed(2)
    out = {}
    c = dec.cfg
    # -- batch-1 rollout
    P1, N1 = 512, 256
    seq1 = torch.tensor(synth.tokens((1, P1 + N1 + 1), c.vocab, stream=300 + rank), dtype=torch.int32,
                        device=dev)
    kv1 = dec.new_kv(1, P1 + N1)
    lp1 = torch.empty(1, N1 + 1, dtype=torch.float32, device=dev)
    pz1 = torch.empty(1, dtype=torch.float32, device=dev)
    roll = lambda: dec.rollout(kv1, 1, P1 + N1, seq1, P1, logprobs=lp1)
    pre = lambda: dec.prefill(kv1, 1, P1 + N1, seq1[:, :P1].contiguous(), 0, None,
                              seq1[:, P1].contiguous(), pz1)
    for _ in range(2):
        roll()
        pre()
    t_roll = _event_time(roll, 2, stream)
    t_pre = _event_time(pre, 3, stream)
    step_s = (t_roll - t_pre) / N1
    kv_mean = sum(P1 + j + 1 for j in range(N1)) / N1 * KV_BYTES_PER_TOKEN
    out["batch1_rollout"] = dict(_hbm_entry(STEP_WEIGHT_BYTES + kv_mean, step_s, hbm, 1),
                                 workload="36 layers, batch 1, prompt 512, 256 teacher-forced steps")
    del kv1
    # -- one layer, KV 2048, batch 1 / 8 / 32 / 64
    S = 2048
    layer = {}
    for Bn in (1, 8, 32, 64):
        half = Bn * c.n_kv_heads * (S + 1) * c.head_dim
        kvl = torch.empty(2 * half, dtype=torch.bfloat16, device=dev)
        kvl.normal_(generator=gen)
        x = torch.randn(Bn, c.hidden, generator=gen, device=dev)
        pos = torch.full((Bn,), S, dtype=torch.int32, device=dev)
        ws = dec.workspace(qkb.QK_CALL_DECODE, Bn, 1, S + 1)
        f = lambda: qkb.qk_decode_layer(dec.handle, 0, kvl, Bn, S + 1, x, pos, Bn, ws)
        for _ in range(5):
            f()
        t = _event_time(f, 50, stream)
        layer[str(Bn)] = _hbm_entry(LAYER_WEIGHT_BYTES + Bn * S * KV_BYTES_PER_TOKEN_LAYER, t, hbm, Bn)
        del kvl
    out["one_layer_kv2048"] = layer
    if dec.check_status() != 0:
        raise RuntimeError("device status flags set in the one-layer decode configs")
    # -- 36 layers, batch 64, long cache
    Bn, Smax = 64, 8192
    kvb = dec.new_kv(Bn, Smax)
    kvb.view(torch.bfloat16).normal_(generator=gen)
    tok = torch.tensor(synth.tokens((Bn,), c.vocab, stream=400 + rank), dtype=torch.int32, device=dev)
    tgt = torch.tensor(synth.tokens((Bn,), c.vocab, stream=401 + rank), dtype=torch.int32, device=dev)
    lpb = torch.empty(Bn, dtype=torch.float32, device=dev)
    long = {}
    for p in (4096, 6144, 8191):
        pos = torch.full((Bn,), p, dtype=torch.int32, device=dev)
        f = lambda: dec.decode_step(kvb, Bn, Smax, tok, pos, None, tgt, lpb)
        for _ in range(2):
            f()
        t = _event_time(f, 5, stream)
        long[str(p + 1)] = _hbm_entry(STEP_WEIGHT_BYTES + Bn * (p + 1) * KV_BYTES_PER_TOKEN, t, hbm, Bn)
    out["batch64_long_context"] = {"workload": "36 layers, batch 64, KV context 4097 / 6145 / 8192",
                                   "by_context": long}
    if dec.check_status() != 0 or not torch.isfinite(lpb).all():
        raise RuntimeError("the batch-64 long-context decode produced invalid output")
    del kvb
    dec._ws.clear()
    torch.cuda.empty_cache()
    return out


# --------------------------------------------------------------------------- backward
BWD_B, BWD_T = 2, 4096


def backward_flops(B, T):
    """Algorithmic FLOPs of one gradient of the token log-likelihood of the 36-layer model over
    B x T tokens: 6 flops per (token, weight) for the linear layers and the lm_head (forward 2,
    backward 4), and 3 x the causal attention forward (QK^T and PV over the T (T + 1) / 2
    query-key pairs of each row and head; the backward is twice the forward).  The kernels
    also run the attention probabilities and the lm_head logits a second time (not counted)."""
    M = B * T
    linear = 6 * M * (36 * 192937984 + 151936 * 4096)
    attn = 36 * 3 * 2 * 2 * 128 * 32 * B * (T * (T + 1) // 2)
    return linear + attn


def backward_config(dec, dev, stream, rank, world):
    """Backward pass (qk_backward_logprob, the gradient of Eq. sft; Eq. ppo through its
    coefficients) of the 36-layer model over 2 x 4096 tokens, token-mean coefficients:
    device-resident inputs, then end to end from pinned host buffers (tokens and
    coefficients in, the loss out)."""
    import torch
    import synth
    peaks = measured_peaks()
    sustained = peaks["bf16_tflops_sustained"] if peaks and "bf16_tflops_sustained" in peaks else 1700.0
    B_, T_ = BWD_B, BWD_T
    tok_h = torch.tensor(synth.tokens((B_, T_), dec.cfg.vocab, stream=500 + rank), dtype=torch.int32)
    coef_h = torch.full((B_, T_ - 1), 1.0 / (B_ * (T_ - 1)), dtype=torch.float32)
    tok = tok_h.to(dev)
    coef = coef_h.to(dev)
    grads = dec.new_grads()
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    f = lambda: dec.backward(tok, coef, grads, loss=loss)
    f()
    torch.cuda.synchronize(dev)
    if dec.check_status() != 0 or not torch.isfinite(loss).all():
        raise RuntimeError("the backward pass produced invalid output")
    t = max_over_ranks(_event_time(f, 2, stream), world)
    # end to end: pinned host tokens / coefficients in, loss out, every call
    tok_p, coef_p = tok_h.pin_memory(), coef_h.pin_memory()
    loss_h = torch.empty(1, dtype=torch.float32).pin_memory()
    tok_d, coef_d = torch.empty_like(tok), torch.empty_like(coef)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    for _ in range(2):
        tok_d.copy_(tok_p, non_blocking=True)
        coef_d.copy_(coef_p, non_blocking=True)
        dec.backward(tok_d, coef_d, grads, loss=loss)
        loss_h.copy_(loss, non_blocking=True)
        torch.cuda.synchronize(dev)
    e2e = max_over_ranks((time.perf_counter() - t0) / 2, world)
    fl = backward_flops(B_, T_)
    out = {"workload": f"gradient of the token-mean log-likelihood, 36-layer Qwen3-8B-shaped bf16, "
                       f"{B_} x {T_} tokens (weights, fp32 gradients and the kept activations resident)",
           "tokens_per_s": world * B_ * T_ / t, "ms_per_call": t * 1e3,
           "roofline": {"bound": "tensor", "flops_per_call": fl, "achieved": fl / t / 1e12,
                        "peak": sustained, "unit": "TFLOP/s", "frac": fl / t / 1e12 / sustained,
                        "peak_source": "measured (sustained)" if peaks else "fallback",
                        "dominant_kernel": "gemm_bwd_tc_kernel<256, 256, 1, 1, E_F32> (weight gradients dW = dY^T X)"},
           "e2e": {"tokens_per_s": world * B_ * T_ / e2e, "h2d_bytes_per_call": int(tok_h.nbytes + coef_h.nbytes),
                   "d2h_bytes_per_call": 4},
           "loss": float(loss_h.item())}
    del grads
    dec._ws.clear()
    torch.cuda.empty_cache()
    return out


def main():
    args = parse()
    world, rank, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
