"""Benchmark of Jacobi decoding (one "step" = one Jacobi iteration of the whole
hot path: embed, 32 decoder layers, LM head + argmax, accept/commit/refill)
on a 7B LLaMA-style decoder with random-init weights.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload llama7b-n16|llama7b-n64|coder7b-b8]

Prints one JSON line (rank 0).  ``value`` is committed tokens/s of the Jacobi
decode loop with every input resident in device memory (graph replays, one
8-byte status read per iteration), timed with CUDA events on the engine's
stream over exactly K iterations after W warm-up iterations.  ``e2e`` is the
same metric through cllm_jacobi_decode with host buffers (prefill, H2D of the
prompt and D2H of the tokens inside the timed region).  The same-kernel AR
decode (n = 1) is timed the same way.  ``--impl reference`` times the oracle
(the plain fp64 CPU decoder) on the host cores instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "committed tokens/s and Jacobi-step latency vs AR step, 7B n=16-64; % HBM roofline"

WORKLOADS = {
    # name: (config, batch, prompt lengths, n, max_new)
    "llama7b-n16": ("llama2-7b", 1, (128, 128), 16, 256),
    "llama7b-n64": ("llama2-7b", 1, (512, 512), 64, 512),
    "coder7b-b8": ("coder-7b", 8, (256, 1024), 32, 256),
}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as fh:
            d = json.load(fh)
        return float(d["hbm_gbs"]), float(d["bf16_tflops_sustained"]), "measured"
    return 6800.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self._t = threading.Thread(target=self._read, daemon=True)
            self._t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def rank_aggregate(dist, device, elapsed, count):
    """Whole-job numbers of a replicas-only run (every rank decodes its own
    sequences, nothing is exchanged on the data path): the slowest rank's
    elapsed time and the sum of the ranks' counts.  Single process (dist is
    None): unchanged."""
    if dist is None:
        return float(elapsed), float(count)
    import torch
    t = torch.tensor([float(elapsed)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    c = torch.tensor([float(count)], device=device, dtype=torch.float64)
    dist.all_reduce(c)
    return float(t.item()), float(c.item())


# Table 3's fast-forwarded token counts (accepted tokens per iteration,
# including the head) of the CLLMs, per n-token length and dataset.  The step
# time does not depend on acceptance, so tokens/s at the paper's acceptance is
# the measured step time with that mean -- synthetic, labelled as such.
TABLE3_FAST_FORWARD = {16: (2.8, "CLLM-LLaMA-2-7B, GSM8K, n=16"),
                       32: (4.0, "CLLM-Deepseek-coder-7B, Code-Search-Net Python, n=32")}


def emulated_acceptance(workload, B, ms_step):
    n = WORKLOADS[workload][3]
    if n not in TABLE3_FAST_FORWARD or not ms_step:
        return None
    a, src = TABLE3_FAST_FORWARD[n]
    return {"mean_accepted": a, "source": f"Table 3, {src}", "kind": "synthetic (measured step time x paper's acceptance)",
            "tokens_per_s": a * B / (ms_step / 1e3)}


def kernel_sources_digest():
    """First 16 hex digits of the SHA-256 of the persistent kernel's sources:
    its translation unit and every CUDA header (names and contents)."""
    h = hashlib.sha256()
    src = os.path.join(ROOT, "paper_2403_00835_gb300", "csrc")
    for name in sorted(os.listdir(src)):
        if name == "persistent.cu" or name.endswith(".cuh"):
            h.update(name.encode())
            with open(os.path.join(src, name), "rb") as f:
                h.update(f.read())
    return h.hexdigest()[:16]


def measured_traffic(kernel, workload, layers):
    """DRAM bytes (read + write) per launch of `kernel` from the committed ncu
    summary of this workload, or None when there is none or the kernel sources
    changed since it was taken."""
    if layers:
        return None
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload.replace('-', '_')}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    d = re.search(r"kernel_sources_sha256_16:\s*([0-9a-f]{16})", text)
    if not m or not d or d.group(1) != kernel_sources_digest():
        return None
    return float(m.group(1))


def step_bytes(cfg, B, n, L_mean):
    """Algorithmic HBM bytes of one Jacobi iteration: every weight once, the
    KV cache read of each sequence's context, the block's K/V written."""
    d, F, V = cfg.d_model, cfg.ffn, cfg.vocab
    dq, dkv = cfg.n_heads * cfg.head_dim, cfg.n_kv_heads * cfg.head_dim
    wbytes = 2 * (cfg.n_layers * (d * (dq + 2 * dkv) + dq * d + 3 * d * F) + V * d)
    kv = 2 * 2 * cfg.n_layers * dkv * B * (L_mean + n)
    return wbytes + kv


def gateup_bytes(cfg, T):
    """Algorithmic bytes of one gate/up launch: both weight matrices once, the
    normalised input read, the SwiGLU output written."""
    d, F = cfg.d_model, cfg.ffn
    return 2 * (2 * F * d) + 2 * T * d + 2 * T * F


# ----------------------------------------------------------------------------------------
# oracle (CPU) baseline: bounded sample of the same workload
# ----------------------------------------------------------------------------------------

def host_cores():
    """Cores this process may run on (its CPU affinity set)."""
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


def oracle_sample(cfg, n, steps=3, warmup=0, layers=2, seed=0, plen=128, threads=(None,)):
    """Time the oracle's Jacobi iteration (n rows) of a 7B-shaped decoder on the
    host cores.  Sample: the first `layers` decoder layers plus the LM head,
    over a `plen`-token prompt (the workload's; prefilled on every core), every
    iteration from the same committed state (a fresh guess block each time),
    timed with each thread count in `threads` (None: the oracle's default).
    Returns, per thread count, the measured time per sampled iteration and,
    separately, the factor that scales it to the full depth by weight bytes
    (weight streaming dominates the oracle's cost)."""
    from dataclasses import replace

    from oracle import oracle as orc
    from paper_2403_00835_gb300 import synthetic as syn
    Ls = layers
    sub = replace(cfg, n_layers=Ls)
    w = syn.make_weights(sub, seed=seed, device="cpu")
    om = orc.OracleModel(orc.OracleArch(**syn.oracle_arch_kwargs(sub)), w, orc.ORC_BF16)
    prompt = syn.make_prompts(cfg.vocab, [plen], seed=1)[0]
    sess = om.session(plen + n + 8)
    head, _, _ = orc.prefill(sess, prompt)
    L = len(prompt)
    lw = 2 * (cfg.d_model * cfg.vocab)
    per_layer_bytes = (step_bytes(sub, 1, n, L) - lw) / Ls
    scale = (cfg.n_layers * per_layer_bytes + lw) / (Ls * per_layer_bytes + lw)
    prev = orc.num_threads()
    out = []
    try:
        for th in threads:
            if th:
                orc.set_num_threads(th)
            used = orc.num_threads()
            times, acc = [], []
            for it in range(warmup + steps):
                blk = [head] + [orc.guess_token(2, 0, it, k, cfg.vocab) for k in range(1, n)]
                t0 = time.perf_counter()
                st = orc.jacobi_step(sess, blk, L)
                dt = time.perf_counter() - t0
                if it >= warmup:
                    times.append(dt)
                    acc.append(st.accepted)
            sample_s = sum(times) / len(times)
            out.append({
                "sample_s_per_step": sample_s, "scale_to_full_depth": scale, "step_s": sample_s * scale,
                "accepted_total": sum(acc), "steps": len(times), "threads": used,
                "sample": (f"oracle Jacobi iteration, n={n}, layers 1-{Ls} of {cfg.n_layers} + LM head "
                           f"of the {cfg.name} shape, {plen}-token prompt, {len(times)} iteration(s) from "
                           f"one committed state on {used} thread(s); measured time per sampled "
                           f"iteration {sample_s * 1e3:.1f} ms, scaled x{scale:.2f} to {cfg.n_layers} "
                           f"layers by weight bytes")})
    finally:
        orc.set_num_threads(prev)
        sess.close()
    return out


def oracle_tiny_decodes(max_new=64, n=8):
    """Wall time of the oracle's full decodes of the tiny fp32 configuration
    (32-token prompt): greedy AR and Jacobi (refill policy, block n)."""
    from oracle import oracle as orc
    from paper_2403_00835_gb300 import synthetic as syn
    cfg = syn.TINY
    w = syn.make_weights(cfg, seed=0, device="cpu")
    om = orc.OracleModel(orc.OracleArch(**syn.oracle_arch_kwargs(cfg)), w, orc.ORC_F32)
    prompt = syn.make_prompts(cfg.vocab, [32], seed=1)[0]
    t0 = time.perf_counter()
    ar = orc.ar_decode(om, prompt, max_new)
    t1 = time.perf_counter()
    jr = orc.jacobi_decode(om, prompt, n, max_new, seed=2)
    t2 = time.perf_counter()
    return {"config": "tiny fp32 (2 layers, d 256, vocab 2048), prompt 32, max_new 64",
            "ar_s": t1 - t0, "ar_tokens_per_s": len(ar.tokens) / (t1 - t0),
            "jacobi_n8_s": t2 - t1, "jacobi_n8_tokens_per_s": len(jr.tokens) / (t2 - t1),
            "jacobi_n8_iterations": jr.iterations, "threads": orc.num_threads()}


def cpu_baseline_entry(cfg, n, plen):
    """The bench line's cpu_baseline: the oracle on every host core and on one
    core (7B-shaped sample), plus full tiny-config decodes."""
    cores = host_cores()
    cb, one = oracle_sample(cfg, n, steps=2, warmup=0, layers=2, plen=plen, threads=(cores, 1))
    value = cb["accepted_total"] / (cb["step_s"] * cb["steps"])
    return {"value": value, "unit": "tokens/s", "cores": cb["threads"], "kind": "oracle",
            "sample": cb["sample"], "host_cores": cores,
            "sample_ms_per_step": cb["sample_s_per_step"] * 1e3,
            "scale_to_full_depth": cb["scale_to_full_depth"],
            "extrapolated_ms_per_step": cb["step_s"] * 1e3,
            "one_core": {"value": one["accepted_total"] / (one["step_s"] * one["steps"]),
                         "sample_ms_per_step": one["sample_s_per_step"] * 1e3,
                         "extrapolated_ms_per_step": one["step_s"] * 1e3, "cores": 1},
            "tiny_full_decodes": oracle_tiny_decodes()}


# ----------------------------------------------------------------------------------------

def run_reference(args, rank):
    """The reference arm: the oracle (this tier has no reference implementation
    to install), timed as it stands on the host cores over a bounded sample of
    the workload -- every step one Jacobi iteration of the first 2 of the 32
    layers plus the LM head.  ms_per_step is the measured time of that sampled
    step; value extrapolates it to the full depth by weight bytes (the factor
    is reported as scale_to_full_depth)."""
    from paper_2403_00835_gb300 import synthetic as syn
    if rank != 0:
        return 0  # under torchrun only rank 0 runs the CPU reference
    cname, B, lens, n, max_new = WORKLOADS[args.workload]
    cfg = syn.CONFIGS[cname]
    cores = host_cores()
    res = oracle_sample(cfg, n, steps=args.steps, warmup=args.warmup, layers=args.cpu_layers,
                        plen=lens[0] if lens[0] == lens[1] else 128, threads=(cores,))[0]
    value = res["accepted_total"] / (res["step_s"] * res["steps"])
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": res["sample_s_per_step"] * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(args.workload),
        "scale_to_full_depth": res["scale_to_full_depth"],
        "extrapolated_ms_per_step": res["step_s"] * 1e3,
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": res["threads"], "kind": "oracle",
                         "sample": res["sample"], "host_cores": cores},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def decode_loop_ms(eng, nblk, max_new, steps, warmup, seed, stream, dist=None):
    """`steps` iterations of the device-resident decode loop after `warmup`
    untimed ones, timed with CUDA events on the engine's stream; a decode that
    reaches max_new is restarted from the prefill (inside the timed region).
    Returns (ms, committed tokens, restarts)."""
    import torch

    def run(iters):
        committed, restarts = 0, 0
        left = iters
        while left > 0:
            it, c = eng.decode_run(left)
            left -= it
            committed += c
            if left > 0:
                eng.decode_begin(nblk, max_new, seed=seed)
                restarts += 1
        return committed, restarts

    eng.decode_begin(nblk, max_new, seed=seed)
    run(warmup)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.nvtx.range_push(f"decode_n{nblk}")  # (profiler filter: the timed iterations)
    ev0.record(stream)
    committed, restarts = run(steps)
    ev1.record(stream)
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    return ev0.elapsed_time(ev1), committed, restarts


def extra_workload(name, steps, warmup, local, weights=None):
    """Step time of another workload of the metric's range (Jacobi and the
    same-kernel AR step), for the bench line's extra keys.  `weights` reuses
    device weights of the same configuration."""
    import numpy as np
    import torch

    from paper_2403_00835_gb300 import synthetic as syn
    from paper_2403_00835_gb300.cllm import Engine
    cname, B, lens_rng, n, max_new = WORKLOADS[name]
    cfg = syn.CONFIGS[cname]
    lens = [lens_rng[0]] * B if lens_rng[0] == lens_rng[1] else syn.ragged_lens(B, *lens_rng, seed=1)
    prompts = syn.make_prompts(cfg.vocab, lens, seed=1)
    w = weights if weights is not None else syn.make_weights(cfg, seed=0, device=f"cuda:{local}")
    stream = torch.cuda.current_stream()
    eng = Engine(cfg, w, max_batch=B, max_seq=max(lens) + max_new + n + 16, max_block=n, stream=stream)
    try:
        eng.prefill(prompts)
        with ClockSampler(local) as clk:
            ms_j, com_j, _ = decode_loop_ms(eng, n, max_new, steps, warmup, 2, stream)
            ms_a, _, _ = decode_loop_ms(eng, 1, max_new, steps, warmup, 2, stream)
        persistent = bool(eng.uses_persistent(n))
    finally:
        eng.close()
    hbm, _, peak_kind = measured_peaks()
    ms_step, ms_ar = ms_j / steps, ms_a / steps
    sb = step_bytes(cfg, B, n, float(np.mean(lens)) + max_new / 2)
    return {"workload": workload_config(name)["workload"], "steps": steps, "warmup": warmup,
            "ms_per_step": ms_step, "ar_ms_per_step": ms_ar, "jacobi_over_ar_step": ms_step / ms_ar,
            "tokens_per_s": com_j / (ms_j / 1e3),
            "step_hbm_roofline": {"bytes": sb, "achieved_gbs": sb / (ms_step / 1e3) / 1e9, "peak_gbs": hbm,
                                  "frac": sb / (ms_step / 1e3) / 1e9 / hbm, "peak_kind": peak_kind},
            "path": "persistent kernel" if persistent else "per-GEMM kernels", "clocks": clk.summary()}


def workload_config(name):
    cname, B, lens, n, max_new = WORKLOADS[name]
    return {"workload": f"{cname} random-init N(0,0.02), batch {B}, prompt {lens[0]}"
                        + (f"-{lens[1]}" if lens[1] != lens[0] else "") + f", n={n}, max_new {max_new}",
            "batch": B, "prompt": list(lens), "n": n, "max_new": max_new,
            "l2": "inputs larger than L2: 13.2 GB of weights streamed per step"}


def run_ours(args, world, rank, local):
    import numpy as np
    import torch

    from paper_2403_00835_gb300 import synthetic as syn
    from paper_2403_00835_gb300.cllm import Engine

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    cname, B, lens_rng, n, max_new = WORKLOADS[args.workload]
    cfg = syn.CONFIGS[cname]
    if args.layers:
        from dataclasses import replace
        cfg = replace(cfg, n_layers=args.layers)
    lens = [lens_rng[0]] * B if lens_rng[0] == lens_rng[1] else syn.ragged_lens(B, *lens_rng, seed=1)
    prompts = syn.make_prompts(cfg.vocab, lens, seed=1 + rank)
    w = syn.make_weights(cfg, seed=0, device=f"cuda:{local}")
    stream = torch.cuda.current_stream()
    max_seq = max(lens) + max_new + n + 16
    eng = Engine(cfg, w, max_batch=B, max_seq=max_seq, max_block=n, stream=stream)
    eng.prefill(prompts)
    total_new = B * max_new

    def timed_loop(nblk, steps, warmup, seed):
        ms, committed, restarts = decode_loop_ms(eng, nblk, max_new, steps, warmup, seed, stream, dist)
        ms, committed = rank_aggregate(dist, "cuda", ms, committed)
        return ms, committed, restarts

    # Jacobi (n) and the same-kernel AR baseline (n = 1)
    with ClockSampler(local) as clk:
        ms_j, com_j, rs_j = timed_loop(n, args.steps, args.warmup, seed=2)
        ms_a, com_a, _ = timed_loop(1, args.steps, args.warmup, seed=2)
    clocks = clk.summary()
    value = com_j / (ms_j / 1e3)
    ms_step = ms_j / args.steps
    ms_ar = ms_a / args.steps

    # per-kernel device time from a profiled pass (CUDA events between kernels)
    eng.set_profiling(True)
    eng.decode_begin(n, max_new, seed=2)
    eng.decode_run(min(8, max_new))
    prof = eng.profile_read()
    eng.set_profiling(False)
    launches_per_iter = eng.kernels_per_iteration(n)

    # end to end through the C ABI with host buffers (prefill + decode + copies)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    t0 = time.perf_counter()
    out, iters = eng.jacobi_decode(prompts, n, max_new, seed=2)
    e2e_s = time.perf_counter() - t0
    e2e_s, e2e_tokens = rank_aggregate(dist, "cuda", e2e_s, int(np.sum(out >= 0)))
    e2e_val = e2e_tokens / e2e_s
    e2e_iters = max(1, int(np.max(iters)))
    # host<->device bytes of that call, per decode iteration: the prompt
    # tokens and lengths in, the status word (12 bytes) out every iteration,
    # and the committed tokens and iteration counts out at the end
    e2e_h2d = 4 * (sum(lens) + B) / e2e_iters
    e2e_d2h = 12 + 4 * (B * max_new + B) / e2e_iters

    # acceptance profile (untimed): a shrink-policy decode of the same prompts
    # with the trajectory recorded, analysed on the host (Sec. 3.3, Table 3)
    from paper_2403_00835_gb300 import trajectory as tj
    from paper_2403_00835_gb300.cllm import CLLM_BLOCK_SHRINK
    prof_new = min(max_new, 128)
    tout, titers, traj = eng.jacobi_decode(prompts, n, prof_new, seed=2, block_mode=CLLM_BLOCK_SHRINK,
                                           record_cap=prof_new + 1)
    tstat = tj.analyse_batch(traj, tout, titers, n)
    hist = np.bincount(np.asarray(tstat.accepted), minlength=n + 1)[1:].tolist()

    hbm, tflops, peak_kind = measured_peaks()
    T = B * n
    L_mean = float(np.mean(lens)) + max_new / 2
    sbytes = step_bytes(cfg, B, n, L_mean)
    persistent = "step_persistent" in prof
    if persistent:
        # the whole iteration is one kernel: its bytes are the step's bytes
        k_ms, k_cnt = prof["step_persistent"]
        k_name, k_bytes = "step_persistent", sbytes
        phases = {k[len("phase:"):]: v for k, v in prof.items() if k.startswith("phase:")}
    else:
        k_ms, k_cnt = prof.get("gemm_gateup", (0.0, 0))
        k_name, k_bytes = "gemm_gateup", gateup_bytes(cfg, T)
        phases = prof
    k_avg = k_ms / max(k_cnt, 1)
    achieved = k_bytes / (k_avg / 1e3) / 1e9 if k_avg > 0 else None
    tot_prof = sum(v[0] for v in phases.values())
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic (random-init weights, uniform-random prompts)",
        "config": workload_config(args.workload),
        "ar_ms_per_step": ms_ar, "jacobi_over_ar_step": ms_step / ms_ar,
        "ar_tokens_per_s": com_a / (ms_a / 1e3),
        "mean_accepted": com_j / (args.steps * B) if args.steps else None,
        "acceptance_profile": {
            "policy": "shrink (Alg. 3), trajectory recorded on the GPU, analysed on the host",
            "tokens": prof_new, "mean_accepted_per_iteration": tstat.mean_accepted,
            "accepted_histogram_1_to_n": hist,
            "mean_stationary_per_window": tstat.mean_stationary,
            "windows": len(tstat.window_stationary)},
        "emulated_acceptance": emulated_acceptance(args.workload, B, ms_step),
        "step_hbm_roofline": {"bytes": sbytes, "achieved_gbs": sbytes / (ms_step / 1e3) / 1e9,
                              "peak_gbs": hbm, "frac": sbytes / (ms_step / 1e3) / 1e9 / hbm,
                              "peak_kind": peak_kind},
        "roofline": {"bound": "hbm", "kernel": k_name, "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": (achieved / hbm) if achieved else None,
                     "traffic": measured_traffic(k_name, args.workload, args.layers),
                     "peak_kind": f"{peak_kind} (copy bandwidth)",
                     "algorithmic_bytes_per_launch": k_bytes, "avg_launch_ms": k_avg},
        "kernel_share": {k: round(v[0] / tot_prof, 4) for k, v in sorted(phases.items())} if tot_prof else {},
        "kernel_avg_us": {k: round(1e3 * v[0] / max(v[1], 1), 2) for k, v in sorted(phases.items())},
        "persistent_kernel": persistent,
        "e2e": {"value": e2e_val, "unit": "tokens/s",
                "h2d_bytes_per_step": e2e_h2d, "d2h_bytes_per_step": e2e_d2h,
                "what": f"cllm_jacobi_decode of {B}x{max_new} tokens incl. prefill, wall clock, "
                        f"host buffers; {e2e_iters} iterations"},
        "gpu_launches": launches_per_iter * args.steps + rs_j,
        "clocks": clocks,
    }
    eng.close()
    if world == 1 and not args.layers and args.workload == "llama7b-n16" and not args.no_extra:
        # the rest of the metric's range, in the same run and clock record:
        # the wide block (prompt 512, n = 64) and the ragged coder batch
        extra_steps = max(3, min(args.steps, 10))
        line["n64"] = extra_workload("llama7b-n64", extra_steps, args.warmup, local, weights=w)
        del w
        torch.cuda.empty_cache()
        line["coder_b8"] = extra_workload("coder7b-b8", extra_steps, args.warmup, local)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline_entry(cfg, n, lens[0] if len(set(lens)) == 1 else 128)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(line), flush=True)
    return 0


def run_sweep(args):
    """Step microbenchmark (LLaMA-2-7B shape): decode-loop step time over cache
    length L, block width n and batch B, each point after a prefill of B
    random prompts of length L; prints one JSON object per point, then a
    markdown table.  Not the default bench line."""
    import numpy as np
    import torch

    from paper_2403_00835_gb300 import synthetic as syn
    from paper_2403_00835_gb300.cllm import Engine

    cfg = syn.LLAMA7B
    if args.layers:
        from dataclasses import replace
        cfg = replace(cfg, n_layers=args.layers)
    Ls, ns, Bs = (256, 1024, 4096), (1, 16, 32, 64, 128), (1, 4, 16)
    if args.point:  # one point of the sweep: L,B,n
        L0, B0, n0 = (int(v) for v in args.point.split(","))
        Ls, ns, Bs = (L0,), (n0,), (B0,)
    w = syn.make_weights(cfg, seed=0, device="cuda")
    stream = torch.cuda.current_stream()
    max_new = 256
    eng = Engine(cfg, w, max_batch=max(Bs), max_seq=max(Ls) + max_new + max(ns) + 16,
                 max_block=max(ns), stream=stream)
    hbm, _, _ = measured_peaks()
    rows = []
    for L in Ls:
        for B in Bs:
            prompts = syn.make_prompts(cfg.vocab, [L] * B, seed=1)
            for n in ns:
                eng.prefill(prompts)
                eng.decode_begin(n, max_new, seed=2)
                left = args.warmup
                while left > 0:
                    it, _ = eng.decode_run(left)
                    left -= it
                    if left > 0:
                        eng.decode_begin(n, max_new, seed=2)
                torch.cuda.synchronize()
                ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.nvtx.range_push(f"sweep_L{L}_B{B}_n{n}")
                ev0.record(stream)
                left, committed = args.steps, 0
                while left > 0:
                    it, c = eng.decode_run(left)
                    left -= it
                    committed += c
                    if left > 0:
                        eng.decode_begin(n, max_new, seed=2)
                ev1.record(stream)
                torch.cuda.nvtx.range_pop()
                torch.cuda.synchronize()
                ms = ev0.elapsed_time(ev1) / args.steps
                sb = step_bytes(cfg, B, n, L + max_new / 2)
                r = {"L": L, "n": n, "B": B, "ms_per_step": ms, "tokens_per_s": committed / (args.steps * ms / 1e3),
                     "hbm_frac": sb / (ms / 1e3) / 1e9 / hbm, "persistent": bool(eng.uses_persistent(n))}
                rows.append(r)
                print(json.dumps(r), flush=True)
    eng.close()
    print("\n| L | B | n | ms/step | tokens/s | step bytes / time vs copy peak | path |")
    print("|---|---|---|---|---|---|---|")
    for r in rows:
        print("| %d | %d | %d | %.3f | %.1f | %.1f %% | %s |" % (
            r["L"], r["B"], r["n"], r["ms_per_step"], r["tokens_per_s"], 100 * r["hbm_frac"],
            "persistent" if r["persistent"] else "per-GEMM kernels"))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama7b-n16", choices=sorted(WORKLOADS))
    ap.add_argument("--cpu-layers", type=int, default=2)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the extra keys (n64, coder_b8) of the default workload's line")
    ap.add_argument("--layers", type=int, default=0,
                    help="decoder layers (default: the full model); a small count gives a "
                         "same-shape case for profiler captures")
    ap.add_argument("--point", default="",
                    help="with --sweep: only this point, 'L,B,n'")
    ap.add_argument("--sweep", action="store_true",
                    help="step microbenchmark over cache length, block width and batch "
                         "(prints a table instead of the bench line)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.sweep:
        return run_sweep(args)
    world, rank, local = dist_setup()
    if args.impl == "reference":
        return run_reference(args, rank)
    return run_ours(args, world, rank, local)


if __name__ == "__main__":
    sys.exit(main())
