#!/usr/bin/env python3
"""Benchmark of the Domino draft-side block step on GB300; prints ONE JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config NAME]

Workload: the Qwen3-8B-shaped batch-1 K=16 draft step (H=4096, V=151936, d_s=1024, r=256,
k=8, N=16), the configuration the metric's target is stated on; synthetic seeded inputs
(paper_2605_29707_gb300/inputs.py).  A step is one domino_draft_step call: embedding gather,
GRU input projection, W1 hidden projection, GRU recurrence + low-rank code, fused vocabulary
GEMM with online softmax/top-k, merge + tree.

value   draft blocks/s over all ranks (B blocks per step per rank), device-timed with CUDA
        events around exactly K steps, inputs resident in HBM; the weights (1.4 GB) exceed
        the 129 MB L2, so no flush is needed between steps.
e2e     the same metric through domino_draft_step_host: per step, hidden + prefix ids are
        copied from pinned host memory and the top-k lists and tree are copied back.
roofline  the dominant kernel (vocabulary GEMM + softmax/top-k): algorithmic bytes (or
        FLOPs) per launch / its mean CUDA-event duration in the timed region.
configs the other Qwen3-shaped workloads (1.7B B=1, 8B B=32, 32B B=64) timed the same way in
        the same run: us per step, blocks/s, the vocabulary kernel's roofline (HBM-bound at
        B=1, tensor-bound against the sustained bf16 peak at B=32/64), the step roofline and
        the per-kernel breakdown.
One GPU only: the library is a single-GPU library (its vocabulary GEMM shares weight tiles
between the CTAs of a cluster by TMA multicast, which only 1-GPU runs may use), so a launch
with WORLD_SIZE > 1 or --gpus > 1 prints a line saying so and runs nothing.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "µs per draft step & draft blocks/s (1 GB300); LM-head HBM GB/s / roofline %"
UNIT = "draft blocks/s"
DEFAULT_CONFIG = "qwen3-8b"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
VOCAB_SOURCES = ["paper_2605_29707_gb300/csrc/tc_gemm.cuh", "paper_2605_29707_gb300/csrc/tc_pair.cuh",
                 "paper_2605_29707_gb300/csrc/tc_softmax.cu", "paper_2605_29707_gb300/csrc/tc_softmax_k8.cu",
                 "paper_2605_29707_gb300/csrc/ptx.cuh", "paper_2605_29707_gb300/csrc/topk.cuh"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "vocab_gemm_traffic.json")


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


EXTRA_CONFIGS = ("qwen3-1.7b", "qwen3-8b-b32", "qwen3-32b-b64")
SINGLE_GPU = ("one GPU only: the library's vocabulary GEMM shares weight tiles within a CTA cluster by TMA "
              "multicast, which only 1-GPU runs may use; run bench.py without torchrun and --gpus 1")


def single_gpu_refusal(world: int, gpus: int):
    """The line a multi-GPU launch prints instead of running (None for a 1-GPU launch)."""
    if world <= 1 and gpus <= 1:
        return None
    return {"metric": METRIC, "unit": UNIT, "n_gpus": max(world, gpus), "unavailable": SINGLE_GPU}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        p["source"] = "measured"
        return p
    p = dict(FALLBACK_PEAKS)
    p["source"] = "fallback"
    return p


def source_sha(paths):
    h = hashlib.sha256()
    for p in paths:
        with open(os.path.join(ROOT, p), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 100 ms while running."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}", "--format=csv,noheader",
                 "-lms", "100", "-f", self.path], stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        time.sleep(0.15)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons, n = [], None, set(), 0
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1].split()[0]))
                    smax = float(parts[2].split()[0])
                except ValueError:
                    continue
                n += 1
                for name, val in zip(self.NAMES, parts[5:9]):
                    if val.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": n}


def vocab_plan(cfg, num_sms):
    """Tile plan of the vocabulary GEMM (mirrors the library's host plan) for byte counting."""
    M = cfg.M
    if M <= 128:
        swap, bn = True, max(16, 1 << (M - 1).bit_length())
        tok_tiles, w_tiles = -(-M // bn), -(-cfg.V // 128)
    else:
        swap, bn = False, 256
        tok_tiles, w_tiles = -(-M // 128), -(-cfg.V // 256)
    per_tok = max(1, num_sms // tok_tiles)
    wpc = -(-w_tiles // per_tok)
    nchunks = -(-w_tiles // wpc)
    kmax = 8 if cfg.k <= 8 else (16 if cfg.k <= 16 else 32)
    return dict(swap=swap, bn=bn, nchunks=nchunks, rec_words=2 + 2 * kmax, grid=tok_tiles * nchunks)


def vocab_work(cfg, num_sms, has_b2=False):
    """Algorithmic bytes and FLOPs of one vocabulary-GEMM launch: every W_lm and W2 row once,
    the activations once, the per-chunk partial records written once (logits never stored)."""
    M, V, H, R = cfg.M, cfg.V, cfg.H, cfg.R
    plan = vocab_plan(cfg, num_sms)
    weights = V * (H + R) * 2 + (V * 2 if has_b2 else 0)
    acts = M * (H + R) * 2
    partials = M * plan["nchunks"] * plan["rec_words"] * 4
    return {"bytes": weights + acts + partials, "flops": 2.0 * M * V * (H + R), "per_unit_bytes": (H + R) * 2,
            "units": V, "plan": plan}


def step_work(cfg):
    """Whole-step algorithmic bytes (every weight once + activations) and FLOPs."""
    M, V, H, R, Ds = cfg.M, cfg.V, cfg.H, cfg.R, cfg.Ds
    weights = (V * H + V * R + 3 * Ds * H + 3 * Ds * Ds + R * (H + Ds)) * 2
    acts = M * H * 2 * 2 + M * 4  # hidden, gathered embedding rows, ids
    flops = 2.0 * M * (H * V + R * V + 3 * Ds * H + 3 * Ds * Ds + (H + Ds) * R)
    return {"bytes": weights + acts, "flops": flops}


def roofline_entry(kind_bytes, kind_flops, ms, peaks, sustained):
    hbm = peaks["hbm_gbs"]
    tens = peaks["bf16_tflops_sustained" if sustained else "bf16_tflops"]
    t_mem = kind_bytes / (hbm * 1e9)
    t_flop = kind_flops / (tens * 1e12)
    if t_mem >= t_flop:
        achieved = kind_bytes / (ms * 1e-3) / 1e9
        return {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(achieved / hbm, 4), "peak_source": peaks["source"]}
    achieved = kind_flops / (ms * 1e-3) / 1e12
    return {"bound": "tensor", "achieved": round(achieved, 1), "peak": tens, "unit": "TFLOP/s",
            "frac": round(achieved / tens, 4),
            "peak_source": peaks["source"] + (" sustained" if sustained else " burst")}


def traffic_for(cfg_name):
    if not os.path.exists(TRAFFIC_FILE):
        return None, "no ncu record"
    with open(TRAFFIC_FILE) as f:
        rec = json.load(f)
    if rec.get("source_sha") != source_sha(VOCAB_SOURCES):
        return None, "kernel changed since the ncu capture"
    ent = rec.get("configs", {}).get(cfg_name)
    if not ent:
        return None, "no capture for this workload"
    return ent["traffic_bytes_per_launch"], ent.get("note", "")


def dev_bf16(a, device):
    import numpy as np
    import torch
    return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(device)


# ---------------------------------------------------------------------------- CPU oracle legs
def oracle_full_step_seconds(wl, budget_s, max_steps=1000):
    """Times whole oracle steps (all positions, all vocabulary rows) for about budget_s."""
    import oracle
    c = wl.cfg
    times = []
    t_end = time.perf_counter() + budget_s
    while len(times) < max_steps and (not times or time.perf_counter() < t_end):
        t0 = time.perf_counter()
        oracle.draft_step(wl.weights, wl.hidden, wl.prefix_ids, c.k, c.N, seqs=[0])
        times.append(time.perf_counter() - t0)
    return statistics.mean(times), len(times)


def cpu_baseline(wl, budget_s=12.0):
    import oracle
    sec, n = oracle_full_step_seconds(wl, budget_s)
    c = wl.cfg
    return {"value": round(1.0 / sec, 4), "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
            "sample": f"{n} whole oracle steps of one sequence ({c.K} positions x {c.V} vocabulary rows, fp64, "
                      f"OpenMP), {sec:.3f} s each; blocks/s = 1/seconds per step"}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0  # under torchrun the oracle runs on rank 0 alone
    import numpy as np
    import oracle
    from paper_2605_29707_gb300 import inputs
    oracle.build()
    wl = inputs.make_workload(args.config)
    c, w = wl.cfg, wl.weights
    hid = (wl.hidden[0].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    ids = wl.prefix_ids[0]
    # the correction branch's state (GRU + low-rank code) once per block, timed
    t0 = time.perf_counter()
    E = oracle.embed(w["emb"], ids)
    S = oracle.gru(E, w["w_ih"], w["w_hh"], w["b_ih"], w["b_hh"])
    u = oracle.lowrank(hid, S, w["w1"], w["b1"])
    t_head = time.perf_counter() - t0
    # calibrate one vocabulary slice, then size the per-step sample to the time budget
    probe = 2048
    t0 = time.perf_counter()
    z = oracle.logits(hid, u, w["w_lm"][:probe], w["w2"][:probe], None if w["b2"] is None else w["b2"][:probe])
    oracle.topk(oracle.log_softmax(z)[0], c.k)
    t_probe = time.perf_counter() - t0
    budget = float(os.environ.get("DOMINO_REF_BUDGET_S", "90"))
    per_step = budget / max(1, args.steps + args.warmup)
    Vs = int(min(c.V, max(128, probe * per_step / max(t_probe, 1e-6))))
    times = []
    for i in range(args.warmup + args.steps):
        v0 = (i * Vs) % max(1, c.V - Vs + 1)
        t0 = time.perf_counter()
        z = oracle.logits(hid, u, w["w_lm"][v0:v0 + Vs], w["w2"][v0:v0 + Vs],
                          None if w["b2"] is None else w["b2"][v0:v0 + Vs])
        lp, _ = oracle.log_softmax(z)
        oracle.topk(lp, min(c.k, Vs))
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    t_tree0 = time.perf_counter()
    oracle.tree(np.zeros((c.K, c.k), np.int32) + np.arange(c.k, dtype=np.int32), -np.tile(np.arange(c.k, dtype=np.float64), (c.K, 1)) - 1.0, c.N)
    t_tree = time.perf_counter() - t_tree0
    sec_step = t_head + statistics.mean(times) * (c.V / Vs) + t_tree
    value = c.B / sec_step
    cores = oracle.max_threads()
    sample = (f"{args.steps} timed samples, each the fp64 oracle's logits, log-softmax and top-k for all {c.K} "
              f"positions over a {Vs}-row vocabulary slice ({Vs / c.V:.4f} of the step); the GRU + low-rank code "
              f"({t_head:.3f} s) and the tree are timed once per block; seconds per block = head + mean slice "
              f"time x V/slice + tree = {sec_step:.3f} s")
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(sec_step * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_dict(c),
            "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def config_dict(c):
    return {"workload": f"{c.name}: B={c.B} K={c.K} H={c.H} V={c.V} d_s={c.Ds} r={c.R} k={c.k} N={c.N}",
            "B": c.B, "K": c.K, "H": c.H, "V": c.V, "d_s": c.Ds, "r": c.R, "k": c.k, "N": c.N,
            "parallelism": "one GPU",
            "l2": f"no flush: the weights ({c.V * c.H * 2 / 1e9:.2f} GB of W_lm alone) exceed the 129 MB L2"}


# ---------------------------------------------------------------------------- our arm
def time_steps(st, hidden, ids, stream, n, warmup):
    """Mean device time (us) of n back-to-back steps on `stream` after `warmup` untimed ones."""
    import torch
    for _ in range(max(3, warmup)):
        st.enqueue(hidden, ids, stream)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(n):
        rc = st.enqueue(hidden, ids, stream)
        if rc != 0:
            raise RuntimeError(f"step returned {rc}")
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / n * 1e3


def verify_timing(st, c, device, stream, reps=200):
    import torch
    from paper_2605_29707_gb300 import binding, inputs
    torch.cuda.synchronize()
    trees = [(st.tree_parent.view(c.B, c.N)[b].cpu().numpy(), st.tree_token.view(c.B, c.N)[b].cpu().numpy())
             for b in range(c.B)]
    case = inputs.make_verify_case(c.B, c.N, c.V, 97, p_plant=0.8, trees=trees)
    t = torch.from_numpy(case.target).to(device)
    par = st.tree_parent.view(c.B, c.N)
    tok = st.tree_token.view(c.B, c.N)
    ra = torch.empty((c.B, c.N + 1), dtype=torch.int32, device=device)
    nodes = torch.empty((c.B, c.N), dtype=torch.int32, device=device)
    cnt = torch.empty(c.B, dtype=torch.int32, device=device)
    bon = torch.empty(c.B, dtype=torch.int32, device=device)

    def run():
        rc = binding.domino_verify_tree_greedy(t, par, tok, c.B, c.N, c.V, ra, nodes, cnt, bon, stream)
        if rc != 0:
            raise RuntimeError(f"domino_verify_tree_greedy returned {rc}")
    for _ in range(3):
        run()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    us = e0.elapsed_time(e1) / reps * 1e3
    nbytes = c.B * (c.N + 1) * c.V * 4
    greedy_tau = round(float(cnt.float().mean().item()) + 1.0, 3)

    # the same trees at temperature 1 (domino_verify_tree_sample): planted tokens raised by 9 so
    # that they carry about two thirds of a row's mass, one seeded uniform per row
    T = 1.0
    case_s = inputs.make_verify_case(c.B, c.N, c.V, 98, p_plant=0.8, trees=trees, margin=9.0)
    t_s = torch.from_numpy(case_s.target).to(device)
    uu = torch.from_numpy(inputs.uniform01(c.B * (c.N + 1), (98, "verify-sample-u")).astype("float32")).to(device)

    def run_s():
        rc = binding.domino_verify_tree_sample(t_s, par, tok, uu, T, c.B, c.N, c.V, ra, nodes, cnt, bon, stream)
        if rc != 0:
            raise RuntimeError(f"domino_verify_tree_sample returned {rc}")
    for _ in range(3):
        run_s()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(reps):
        run_s()
    e1.record(stream)
    torch.cuda.synchronize()
    us_s = e0.elapsed_time(e1) / reps * 1e3
    return {"us": round(us, 2), "logits_bytes": nbytes, "GB_per_s": round(nbytes / (us * 1e-6) / 1e9, 1),
            "tau_mean": greedy_tau,
            "sampled": {"temperature": T, "us": round(us_s, 2), "GB_per_s": round(nbytes / (us_s * 1e-6) / 1e9, 1),
                        "tau_mean": round(float(cnt.float().mean().item()) + 1.0, 3)},
            "note": "synthetic target logits (planted tokens); tau is a mechanics check, not a quality number"}


def rollout_timing(st, wl, c, hidden, device, stream, reps=50):
    """The sequential draft loop (domino_rollout_greedy / _sample / _sample_gumbel) on this workload's weights and
    hidden states: device time per block of K tokens, split into the kernels by the library's
    per-kernel CUDA events.  Timed with the input-projection table emb . W_ih^T (built once,
    outside the timed region) and, for comparison, without it."""
    import numpy as np
    import torch
    from paper_2605_29707_gb300 import binding
    if c.B > 8 or not st.head_on:
        return None
    anchors = torch.from_numpy(np.ascontiguousarray(wl.prefix_ids[:, 0])).to(device)
    nb = binding.domino_rollout_workspace_bytes(c.B, c.K, c.H, c.V, c.Ds, c.R)
    ws = torch.empty(nb, dtype=torch.uint8, device=device)
    tok = torch.empty((c.B, c.K), dtype=torch.int32, device=device)
    lp = torch.empty((c.B, c.K), dtype=torch.float32, device=device)
    uni = torch.rand((c.B, c.K), generator=torch.Generator().manual_seed(11)).to(device)
    table = torch.empty(binding.domino_input_table_bytes(c.V, c.Ds) // 4, dtype=torch.float32, device=device)
    t0 = time.perf_counter()
    rc = binding.domino_build_input_table(st.w["emb"], st.w["w_ih"], c.V, c.H, c.Ds, table, stream)
    build_s = time.perf_counter() - t0
    if rc != 0:
        raise RuntimeError(f"domino_build_input_table returned {rc}")
    w = st.w
    head_t = binding.make_head(w.get("emb"), w.get("w_ih"), w.get("w_hh"), w.get("b_ih"), w.get("b_hh"),
                               w.get("w1"), w.get("b1"), w.get("w2"), w.get("b2"), c.Ds, c.R, table)

    def timed(head, sampled, split=False):
        def run():
            if sampled == "race":
                rc = binding.domino_rollout_sample_gumbel(hidden, anchors, 0x5EED, w["w_lm"], head, c.B, c.K, c.H,
                                                          c.V, tok, lp, ws, nb, stream)
            elif sampled:
                rc = binding.domino_rollout_sample(hidden, anchors, uni, w["w_lm"], head, c.B, c.K, c.H, c.V, tok,
                                                   lp, ws, nb, stream)
            else:
                rc = binding.domino_rollout_greedy(hidden, anchors, w["w_lm"], head, c.B, c.K, c.H, c.V, tok, lp,
                                                   ws, nb, stream)
            if rc != 0:
                raise RuntimeError(f"rollout returned {rc}")
        for _ in range(3):
            run()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            run()
        e1.record(stream)
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) / reps * 1e3
        kern = None
        if split:
            binding.domino_timing_begin(4 * reps)
            for _ in range(reps):
                run()
            torch.cuda.synchronize()
            kern = {n: round(v[0] / max(1, v[1]) * 1e3, 2) for n, v in binding.domino_timing_end().items()
                    if v[1] > 0}
        return us, kern, binding.domino_check_status(ws, stream)

    us, split, status = timed(head_t, False, split=True)
    us_s, _, status_s = timed(head_t, True)
    us_g, split_g, status_g = timed(head_t, "race", split=True)
    us_nt, split_nt, status_nt = timed(st.head, False, split=True)
    # every byte the loop needs once: W_lm (base GEMM), W1[:, :H] (its GEMM), W2, W_hh and
    # W1[:, H:] (step kernel: W2 on chip, the rest in L2 across steps), one table row per token
    # fed back, and the fp32 base logits written and read back once
    unique = (2 * c.V * c.H + 2 * c.R * c.H + 2 * c.V * c.R + 2 * 3 * c.Ds * c.Ds + 2 * c.R * c.Ds
              + 4 * 3 * c.Ds * c.B * c.K + 2 * 4 * c.B * c.K * c.V)
    peaks = load_peaks()
    roof_us = unique / (peaks["hbm_gbs"] * 1e9) * 1e6
    return {"us_per_block": round(us, 2), "draft_tokens_per_s": round(c.B * c.K / (us * 1e-6), 1),
            "us_per_kernel": split, "status": status, "unique_bytes_per_block": unique,
            "sampled": {"us_per_block": round(us_s, 2), "draft_tokens_per_s": round(c.B * c.K / (us_s * 1e-6), 1),
                        "status": status_s, "rule": "inverse CDF of the caller's uniforms (domino_rollout_sample)"},
            "sampled_race": {"us_per_block": round(us_g, 2), "draft_tokens_per_s": round(c.B * c.K / (us_g * 1e-6), 1),
                             "us_per_kernel": split_g, "status": status_g,
                             "frac_of_hbm_roofline": round(roof_us / us_g, 4),
                             "rule": "exponential race / Gumbel-max under a 64-bit seed (domino_rollout_sample_gumbel)"},
            "input_table": {"bytes": table.numel() * 4, "build_s": round(build_s, 4),
                            "note": "emb . W_ih^T [V, 3 d_s] fp32, built once per set of weights (tensor cores)"},
            "without_table": {"us_per_block": round(us_nt, 2), "us_per_kernel": split_nt, "status": status_nt},
            "hbm_roofline_us": round(roof_us, 2), "frac_of_hbm_roofline": round(roof_us / us, 4),
            "note": "B sequences x K draft tokens, each fed back; timing only (parity is in the tests)"}


def torch_unfused_timing(st, c, hidden, stream, reps=50):
    """Context only, not the library: the vocabulary GEMM of the step done the unfused way in
    PyTorch -- cuBLAS bf16 matmuls of hidden with W_lm and of u with W2 writing full logits to
    HBM, then log_softmax and topk -- on the same weights and hidden states (u is a zero tensor
    of the right shape: the GRU and W1 are left out, so this times S5 + S6 only)."""
    import torch
    h = hidden.view(c.M, c.H)
    w_lm, w2 = st.w["w_lm"], (st.w.get("w2") if st.head_on else None)
    u = torch.zeros(c.M, c.R, dtype=torch.bfloat16, device=h.device) if w2 is not None else None

    def run():
        z = torch.matmul(h, w_lm.t())
        if w2 is not None:
            z = z + torch.matmul(u, w2.t())
        return torch.topk(torch.log_softmax(z.float(), dim=-1), c.k, dim=-1)
    with torch.cuda.stream(stream):
        for _ in range(3):
            run()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            run()
        e1.record(stream)
        torch.cuda.synchronize()
    return {"us": round(e0.elapsed_time(e1) / reps * 1e3, 2),
            "note": "context only: torch matmul (cuBLAS) for W_lm and W2 with full logits in HBM, then "
                    "log_softmax + topk (S5 + S6 of the step, the GRU and W1 left out); not part of the library"}


def graph_replay(st, hidden, ids, device, n, blocks_per_step):
    """Capture one step in a CUDA graph and time n replays; on a capture failure, say why."""
    import torch
    try:
        s = torch.cuda.Stream(device)
        g = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(g, stream=s):
            rc = st.enqueue(hidden, ids, s)
        if rc != 0:
            return {"error": f"capture: step returned {rc}"}
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        cur = torch.cuda.current_stream(device)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(cur)
        for _ in range(n):
            g.replay()
        e1.record(cur)
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) / n * 1e3
        return {"us_per_step": round(us, 2), "value": round(blocks_per_step * 1e6 / us, 3), "replays": n}
    except Exception as e:  # noqa: BLE001 -- reported, not fatal
        torch.cuda.synchronize()
        return {"error": str(e).splitlines()[0][:200]}


def per_kernel(st, hidden, ids, stream, n, launches):
    """Per-kernel device time of n steps, each kernel bracketed by an event pair (the library's
    timing hooks): {kind: (total ms, launches)}.  Events between launches serialise the
    GRU / vocabulary-GEMM overlap, so step times come from time_steps, not from this."""
    import torch
    from paper_2605_29707_gb300 import binding
    torch.cuda.synchronize()
    binding.domino_timing_begin(n * launches)
    bad = False
    for _ in range(n):
        bad |= st.enqueue(hidden, ids, stream) != 0
    torch.cuda.synchronize()
    kern = binding.domino_timing_end()
    if bad:
        raise RuntimeError("a step of the per-kernel region returned an error")
    return kern


def vocab_roofline(c, kern, num_sms, peaks, has_b2, n):
    """Roofline entry of the vocabulary kernel from its mean event-timed launch."""
    vw = vocab_work(c, num_sms, has_b2=has_b2)
    vk_ms, vk_n = kern["vocab_gemm_softmax_topk"]
    vk_mean = vk_ms / max(1, vk_n)
    roof = roofline_entry(vw["bytes"], vw["flops"], vk_mean, peaks, sustained=True)
    traffic, traffic_note = traffic_for(c.name)
    roof.update({"kernel": "vocab_gemm_softmax_topk", "traffic": traffic,
                 "algorithmic_bytes_per_launch": vw["bytes"], "algorithmic_flops_per_launch": vw["flops"],
                 "mean_launch_us": round(vk_mean * 1e3, 2), "launches": vk_n, "traffic_note": traffic_note,
                 "timing": f"CUDA events around each launch, {n} steps right after the timed region",
                 "share_of_step": round(vk_ms / max(1e-9, sum(v[0] for v in kern.values())), 4)})
    return roof


def step_roofline(c, peaks, us):
    sw = step_work(c)
    t = max(sw["bytes"] / (peaks["hbm_gbs"] * 1e9), sw["flops"] / (peaks["bf16_tflops_sustained"] * 1e12))
    return {"us": round(t * 1e6, 2), "frac": round(t / (us * 1e-6), 4), "bytes": sw["bytes"], "flops": sw["flops"],
            "note": "max(every weight once / HBM peak, FLOPs / sustained bf16 peak)"}


def measure_config(name, device, stream, steps, warmup, num_sms, peaks):
    """One more workload in the same run: µs per step (CUDA events around `steps` back-to-back
    steps, clocks sampled meanwhile), the per-kernel breakdown, the vocabulary kernel's roofline,
    the step roofline and the step with the correction branch off."""
    import torch
    from paper_2605_29707_gb300 import binding, inputs
    from paper_2605_29707_gb300.step import DraftStep
    wl = inputs.make_workload(name)
    c = wl.cfg
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=device)
    hidden = dev_bf16(wl.hidden, device)
    ids = torch.from_numpy(wl.prefix_ids).to(device)
    sampler = ClockSampler(device.index or 0)
    sampler.start()
    us = time_steps(st, hidden, ids, stream, steps, warmup)
    clocks = sampler.stop()
    rc = binding.domino_check_status(st.workspace, stream)
    if rc != 0:
        raise binding.DominoError(rc, f"{name}: device status")
    n = min(steps, 200)
    kern = per_kernel(st, hidden, ids, stream, n, st.launches_per_step())
    st_off = DraftStep(st.w, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=device, head_on=False)
    us_off = time_steps(st_off, hidden, ids, stream, steps, warmup)
    del st_off
    # the same step with the input-projection table (built once per set of weights, outside the
    # timed region): the GRU reads a table row per position instead of the E . W_ih^T GEMM
    st_tab = DraftStep(st.w, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=device, input_table=True)
    us_tab = time_steps(st_tab, hidden, ids, stream, steps, warmup)
    input_table = {"us_per_step": round(us_tab, 2), "value": round(c.B * 1e6 / us_tab, 3),
                   "launches_per_step": st_tab.launches_per_step(),
                   "step_roofline_frac": step_roofline(c, peaks, us_tab)["frac"],
                   "note": "us_per_step here: the same step reading the GRU's input-gate sums from the table; "
                           "the config's own us_per_step is the step without it"}
    del st_tab
    out = {"config": config_dict(c), "us_per_step": round(us, 2), "value": round(c.B * 1e6 / us, 3), "unit": UNIT,
           "steps": steps, "warmup": max(3, warmup), "gpu_launches": steps * st.launches_per_step(),
           "roofline": vocab_roofline(c, kern, num_sms, peaks, wl.weights.get("b2") is not None, n),
           "step_roofline": step_roofline(c, peaks, us),
           "kernel_breakdown": {k: {"us_per_step": round(v[0] / n * 1e3, 2), "launches": v[1]}
                                for k, v in kern.items() if v[1] > 0},
           "head_overhead": {"us_head_off": round(us_off, 2), "overhead_us": round(us - us_off, 2),
                             "overhead_pct": round(100.0 * (us / us_off - 1.0), 2)},
           "input_table_step": input_table,
           "clocks": clocks}
    del st, hidden, ids, wl
    torch.cuda.empty_cache()
    return out


def run_step_only(args):
    """Only the draft step of one workload (W warm-up + K timed steps, then one greedy tree
    verification when B <= 4): a short, fixed launch sequence for profiler captures.  Prints one
    JSON line with the step time; not a benchmark line."""
    import torch
    from paper_2605_29707_gb300 import binding, inputs
    from paper_2605_29707_gb300.step import DraftStep
    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    wl = inputs.make_workload(args.config)
    c = wl.cfg
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=device)
    hidden = dev_bf16(wl.hidden, device)
    ids = torch.from_numpy(wl.prefix_ids).to(device)
    stream = torch.cuda.current_stream(device)
    us = time_steps(st, hidden, ids, stream, args.steps, args.warmup)
    rc = binding.domino_check_status(st.workspace, stream)
    if rc != 0:
        raise binding.DominoError(rc, "device status")
    verify = verify_timing(st, c, device, stream, reps=3) if c.B <= 4 else None
    kern = per_kernel(st, hidden, ids, stream, args.steps, st.launches_per_step())
    print(json.dumps({"step_only": c.name, "us_per_step": round(us, 2), "launches_per_step": st.launches_per_step(),
                      "steps": args.steps, "warmup": max(3, args.warmup),
                      "verify_us": verify["us"] if verify else None,
                      "us_per_kernel": {k: round(v[0] / max(1, v[1]) * 1e3, 2) for k, v in kern.items() if v[1]}}),
          flush=True)
    return 0


def run_ours(args):
    import numpy as np
    import torch

    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)

    from paper_2605_29707_gb300 import binding, inputs
    from paper_2605_29707_gb300.step import DraftStep

    wl = inputs.make_workload(args.config)
    c = wl.cfg
    st = DraftStep(wl.weights, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=device)
    hidden = dev_bf16(wl.hidden, device)
    ids = torch.from_numpy(wl.prefix_ids).to(device)
    stream = torch.cuda.current_stream(device)
    launches = st.launches_per_step()
    num_sms = torch.cuda.get_device_properties(device).multi_processor_count

    for _ in range(args.warmup):
        rc = st.enqueue(hidden, ids, stream)
        if rc != 0:
            raise binding.DominoError(rc, "warm-up step")
    rc = binding.domino_check_status(st.workspace, stream)
    if rc != 0:
        raise binding.DominoError(rc, "warm-up device status")

    # ---- timed region: exactly K steps, CUDA events on the launching stream
    sampler = ClockSampler(0)
    sampler.start()
    torch.cuda.synchronize(device)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    bad = 0
    for _ in range(args.steps):
        bad |= st.enqueue(hidden, ids, stream) != 0
    ev1.record(stream)
    torch.cuda.synchronize(device)
    clocks = sampler.stop()
    if bad:
        raise RuntimeError("a timed step returned an error")
    rc = binding.domino_check_status(st.workspace, stream)
    if rc != 0:
        raise binding.DominoError(rc, "timed device status")
    ms = ev0.elapsed_time(ev1)

    # ---- second timed region: the same steps with an event pair around every kernel (the
    #      per-kernel breakdown and the roofline)
    k_steps = min(args.steps, 1000)
    kern = per_kernel(st, hidden, ids, stream, k_steps, launches)
    ms_step = ms / args.steps
    value = c.B * args.steps / (ms / 1e3)

    # ---- e2e through the host-buffer entry point (pinned inputs and outputs)
    M = c.M
    h_hidden = torch.from_numpy(wl.hidden.view(np.int16)).pin_memory()
    h_ids = torch.from_numpy(wl.prefix_ids).pin_memory()
    host = {"topk_ids": torch.empty(M * c.k, dtype=torch.int32).pin_memory(),
            "topk_logp": torch.empty(M * c.k, dtype=torch.float32).pin_memory(),
            "tree_parent": torch.empty(c.B * c.N, dtype=torch.int32).pin_memory(),
            "tree_token": torch.empty(c.B * c.N, dtype=torch.int32).pin_memory(),
            "tree_depth": torch.empty(c.B * c.N, dtype=torch.int32).pin_memory(),
            "tree_score": torch.empty(c.B * c.N, dtype=torch.float32).pin_memory()}
    n_e2e = max(3, min(args.steps, 1000))
    for _ in range(3):
        st.run_host(h_hidden, h_ids, host, stream)
    t0 = time.perf_counter()
    for _ in range(n_e2e):
        rc = st.run_host(h_hidden, h_ids, host, stream)
        if rc != 0:
            raise binding.DominoError(rc, "host-buffer step")
    t_e2e = time.perf_counter() - t0
    e2e_value = c.B * n_e2e / t_e2e
    h2d = M * c.H * 2 + M * 4
    # the host entry point reads its outputs (top-k ids and log-probs, the four tree arrays) and a
    # copy of the status in one copy of the workspace region that holds them (256-byte aligned)
    al = lambda n: (n + 255) // 256 * 256
    d2h = 2 * al(M * c.k * 4) + 4 * al(c.B * c.N * 4) + 4

    # ---- Domino-head overhead: the same workload with the correction branch off (R = 0, the
    #      paper's "w/o Domino head" base distribution), same device weights
    head_overhead = None
    if st.head_on:
        st_off = DraftStep(st.w, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=device, head_on=False)
        us_off = time_steps(st_off, hidden, ids, stream, min(args.steps, 1000), args.warmup)
        us_on = ms_step * 1e3
        head_overhead = {"us_head_off": round(us_off, 2), "us_head_on": round(us_on, 2),
                         "overhead_us": round(us_on - us_off, 2), "overhead_pct": round(100.0 * (us_on / us_off - 1.0), 2),
                         "note": "head off = W_lm projection + softmax/top-k + tree only (R = 0)"}
        del st_off

    # ---- the same step with the input-projection table emb . W_ih^T (built once, outside the
    #      timed region): the GRU reads its input-gate sums as table rows instead of projecting
    #      the embedding rows (no X GEMM at larger B)
    input_table = None
    if st.head_on:
        st_tab = DraftStep(st.w, c.B, c.K, c.H, c.V, c.k, c.N, Ds=c.Ds, R=c.R, device=device, input_table=True)
        us_tab = time_steps(st_tab, hidden, ids, stream, min(args.steps, 1000), args.warmup)
        input_table = {"us_per_step": round(us_tab, 2), "launches_per_step": st_tab.launches_per_step(),
                       "table_bytes": st_tab.x_table.numel() * 4,
                       "note": "us_per_step here: the same step reading the GRU's input-gate sums from the table; "
                               "the line's value and us_per_step are the step without it"}
        del st_tab

    # ---- the step after the draft: verification of this step's trees against synthetic target
    #      logits [B, N+1, V] fp32, greedy and at temperature 1 (timing only; parity is in the tests)
    verify = verify_timing(st, c, device, stream) if c.B <= 4 else None
    # ---- the sequential draft loop (the paper's inference loop) on the same weights
    rollout = rollout_timing(st, wl, c, hidden, device, stream)
    # ---- context: the vocabulary GEMM + log_softmax + topk the unfused way in PyTorch
    unfused = torch_unfused_timing(st, c, hidden, stream)

    # ---- roofline of the dominant kernel, measured in the timed region
    peaks = load_peaks()
    dominant = max(kern, key=lambda n: kern[n][0])
    roof = vocab_roofline(c, kern, num_sms, peaks, wl.weights.get("b2") is not None, k_steps)
    breakdown = {n: {"us_per_step": round(v[0] / k_steps * 1e3, 2), "launches": v[1]} for n, v in kern.items()
                 if v[1] > 0}

    line = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 5), "us_per_step": round(ms_step * 1e3, 2),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded, Qwen3-shaped, random-init weights)", "config": config_dict(c),
        "roofline": roof,
        "step_roofline": step_roofline(c, peaks, ms_step * 1e3),
        "kernel_breakdown": breakdown, "dominant_kernel": dominant,
        "e2e": {"value": round(e2e_value, 3), "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "steps": n_e2e, "api": "domino_draft_step_host (synchronous per step)"},
        "gpu_launches": args.steps * launches, "clocks": clocks,
        "head_overhead": head_overhead, "input_table_step": input_table, "torch_unfused": unfused,
        "tree_verify": verify,
        "rollout_greedy": rollout,
    }
    # ---- last for this workload: the same step replayed from a CUDA graph (one captured step,
    #      replayed back to back); a failed capture is reported in the line
    line["graph_replay"] = graph_replay(st, hidden, ids, device, min(args.steps, 1000), c.B)
    del st, hidden, ids
    torch.cuda.empty_cache()
    # ---- the other Qwen3-shaped workloads: 1.7B at B = 1 (HBM-bound), the 8B and 32B serving
    #      batches (tensor-bound), each timed the same way
    if args.extra_configs:
        line["configs"] = {}
        for name in args.extra_configs.split(","):
            if name and name != c.name:
                steps = max(20, min(args.steps, 2000 // max(1, inputs.CONFIGS[name].B)))
                line["configs"][name] = measure_config(name, device, stream, steps, args.warmup, num_sms, peaks)
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, args.cpu_seconds)
    print(json.dumps(line), flush=True)
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=30)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--extra-configs", default=",".join(EXTRA_CONFIGS),
                    help="other workloads timed in the same run (comma-separated; empty for none)")
    ap.add_argument("--step-only", action="store_true",
                    help="run only the step of --config (warm-up, steps, one verification at B <= 4): "
                         "a short launch sequence for profiler captures; prints no benchmark line")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    rank, world, _ = dist_env()
    refusal = single_gpu_refusal(world, args.gpus)
    if refusal is not None:
        if rank == 0:
            print(json.dumps(refusal), flush=True)
        return 0
    return run_step_only(args) if args.step_only else run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
