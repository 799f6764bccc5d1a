"""Decode-step benchmark of the GB300 T-LoopFormer library.

python bench.py [--gpus N] [--steps K] [--warmup W] [--config c4] [--impl ours|reference]

One step = one tlf_decode_step over a batch of B sequences (router,
compaction, every loop's shared block on its active tokens, recursion-wise
attention, LM head). Default workload: the long-context GQA model (d 2048,
16 q / 8 kv heads x 128, 2 layers, ffn 5504, M = 6) with batch 16 at 32768
tokens of context, the configuration the attention bandwidth target is set on.
The sequences' caches are built by prefilling the seeded prompts through the
library before timing (prefill is not part of the step; its time is reported);
--prefill snapshot restores synthetic caches instead.

Prints one JSON line. ``value`` is decode tokens/s over all ranks, timed with
CUDA events on the launching stream with logits left on the device; ``e2e``
is the same metric through the public call with host token ids in and host
logits out (copies inside the timed region). Under torchrun each rank runs
its own batch of sequences (weak scaling, no collective on the data path).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_15160_gb300 import synth  # noqa: E402

DESCR = {
    "c1": "tiny fp32 looped LM (V256 d64 4x16 J1 ff176 M4), batch 1, 32-token prompt",
    "c2": "small bf16 looped LM (V32000 d512 8x64 J2 ff1376 M4), batch 8, 512-token prompts",
    "c3": "mid bf16 looped LM (V50304 d1024 16x64 J4 ff2752 M8), batch 64, 2048-token prompts",
    "c4": "long-context GQA looped LM (d2048 16q/8kv x128 J2 ff5504 M6), batch 16, 32768-token context",
    "c5": "C3 model, ragged prompts U[128,8192], batch 32, routed depths",
    "c5f": "C3 model, ragged prompts U[128,8192], batch 32, every token forced to 8 loops",
    "c2c": "C2 workload on a model with time/step AdaLN conditioning (Sec. 3.1, App. A)",
    "c3c": "C3 workload on a model with time/step AdaLN conditioning (Sec. 3.1, App. A)",
}


def _measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d.get("hbm_gbs", 6800.0), "measured"
    return 6800.0, "fallback"


def _attn_traffic(alg_bytes_per_launch: float):
    """DRAM bytes per attention launch, scaled from the committed ncu capture (None if absent)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(p) as f:
            ratio = json.load(f)["k_attn_decode"]["traffic_over_algorithmic"]
    except (OSError, KeyError, ValueError):
        return None
    return ratio * alg_bytes_per_launch


class ClockSampler:
    """nvidia-smi clock / throttle samples (every 20 ms) while a workload runs, in a temporary file."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.proc = None
        fd, self.path = tempfile.mkstemp(prefix="tlf_clocks_", suffix=".csv")
        self.f = os.fdopen(fd, "w")
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={gpu}", f"--query-gpu={self.Q}", "--format=csv",
                                          "-lms", "20"], stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            self.f.close()
            os.unlink(self.path)
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            lines = f.read().splitlines()[1:]
        os.unlink(self.path)
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1].split()[0]))
                mx.append(float(parts[2].split()[0]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm), "window": "warm-up, device-timed and end-to-end passes, 20 ms poll"}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(values, device="cpu"):
    """Element-wise maximum of per-rank floats over the process group (identity without one)."""
    import torch
    import torch.distributed as dist

    t = torch.tensor(values, dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_tokens_per_s(world_size: int, batch_per_rank: int, steps: int, slowest_ms: float) -> float:
    """Whole-job decode throughput: the tokens of every rank over the slowest rank's time."""
    return world_size * batch_per_rank * steps / (slowest_ms * 1e-3)


def _oracle_sample_cmd(cfg_name: str, tokens: int, rank_seed: int) -> str:
    return f"""
import sys, time, json, numpy as np
sys.path.insert(0, {ROOT!r})
from paper_2609_15160_gb300 import synth
from oracle import tlf_oracle as O
wl = synth.get_config({cfg_name!r}); m = wl.model
w = synth.make_weights(m)
om = O.OracleModel.from_config(m, w)
L = int(max(len(p) for p in synth.make_prompts(wl, batch=1)))
snap = synth.make_cache_snapshot(m, L, {rank_seed})
seq = O.load_snapshot(om, snap, cache_dtype=np.float32)
toks = synth.make_decode_tokens(wl, steps={tokens}, batch=1)[:, 0]
t = time.perf_counter()
for x in toks:
    O.decode_token(om, seq, int(x))
print(json.dumps({{"seconds": time.perf_counter() - t, "tokens": {tokens}, "context": L}}))
"""


def cpu_baseline(cfg_name: str, tokens: int = 3) -> dict:
    """The oracle timed on this host's cores on a bounded sample: one sequence of the workload."""
    cores = os.cpu_count() or 1
    env = dict(os.environ, OMP_NUM_THREADS=str(cores), OPENBLAS_NUM_THREADS=str(cores),
               MKL_NUM_THREADS=str(cores), CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-c", _oracle_sample_cmd(cfg_name, tokens, 11)], capture_output=True,
                       text=True, env=env, timeout=900)
    if r.returncode != 0:
        return {"value": None, "unit": "tokens/s", "cores": cores, "kind": "oracle", "error": r.stderr[-300:]}
    d = json.loads(r.stdout.strip().splitlines()[-1])
    return {"value": d["tokens"] / d["seconds"], "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"1 sequence of the workload at context {d['context']}, {d['tokens']} decode tokens "
                      f"(float64 numpy oracle, BLAS threads = cores)"}


def run_reference(args):
    ws, rank, _ = _dist()
    if rank != 0:
        return
    cfg = args.config
    cores = os.cpu_count() or 1
    per_step = []
    # each step: one decode token of one sequence of the workload through the oracle
    env = dict(os.environ, OMP_NUM_THREADS=str(cores), OPENBLAS_NUM_THREADS=str(cores), CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "-c", _oracle_sample_cmd(cfg, args.warmup + args.steps, 11)],
                       capture_output=True, text=True, env=env, timeout=3600)
    if r.returncode != 0:
        print(json.dumps({"impl": "reference", "unavailable": "oracle run failed: " + r.stderr[-200:]}))
        return
    d = json.loads(r.stdout.strip().splitlines()[-1])
    sec_per_tok = d["seconds"] / d["tokens"]
    value = 1.0 / sec_per_tok
    wl = synth.get_config(cfg)
    line = {"impl": "reference", "metric": "decode_tokens_per_s", "value": value, "unit": "tokens/s",
            "n_gpus": ws, "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * sec_per_tok,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            # the same workload keys as the timed arm's line, then the model description
            "config": {**synth.describe(wl), "workload": DESCR[cfg], "name": cfg, "batch_per_gpu": wl.batch,
                       "context": int(wl.prompt_len[1]),
                       "parallelism": f"replicas x{ws} (rank 0 times the oracle; the others exit)"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"1 sequence at context {d['context']}, 1 decode token per step"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


_WEIGHTS = {}


def model_weights(m):
    """Seeded weights of a model, generated once per model in this process (C3 and C5 share them)."""
    if m not in _WEIGHTS:
        _WEIGHTS[m] = synth.make_weights(m)
    return _WEIGHTS[m]


def setup_workload(T, wl, rank: int, gemm_impl="auto", prefill="auto", extra_tokens: int = 0, ablation="none"):
    m = wl.model
    w = model_weights(m)
    B = wl.batch
    prompts = synth.make_prompts(wl)
    lengths = [len(p) for p in prompts]
    steps_cap = max(wl.decode_steps, extra_tokens) + 64
    # default: real (batched) prefill through the library. Full-length caches (dense-cache ablation)
    # prefill position by position, far too slow for long prompts: they restore snapshots instead
    use_snapshot = prefill == "snapshot" or (prefill == "auto" and ablation == "dense_cache")
    ids = [rank * 100000 + b for b in range(B)]
    if use_snapshot:
        # uniform lengths: two distinct host snapshots (values uploaded); ragged lengths: one
        # snapshot per sequence with only positions, values filled on the device
        host_values = wl.prompt_len[0] == wl.prompt_len[1] and ablation != "dense_cache"
        distinct = {}
        snaps = []
        for b, L in enumerate(lengths):
            key = (L, b % 2) if host_values else (L, b)
            if key not in distinct:
                depths = None if wl.forced_loops is None else np.full(L, wl.forced_loops, np.int32)
                make = synth.make_cache_snapshot if host_values else synth.make_cache_positions
                distinct[key] = make(m, L, seed=1000 * rank + len(distinct), depths=depths)
            snaps.append(distinct[key])
        pages = sum(sum((len(p) + 63) // 64 for p in s["positions"]) for s in snaps) + B * m.max_loops * (
            steps_cap // 64 + 2)
        if ablation == "dense_cache":  # every loop cache holds a slot per position
            pages = B * m.max_loops * ((max(lengths) + steps_cap) // 64 + 2)
    else:
        snaps = None
        pages = B * m.max_loops * ((max(lengths) + steps_cap) // 64 + 2)
    ctx = T.Context(m, w, max_seqs=B, max_batch=B, max_seq_len=max(lengths) + steps_cap, kv_pool_pages=pages,
                    gemm_impl=gemm_impl, ablation=ablation)
    if snaps is not None:
        for b in range(B):
            ctx.load_cache(ids[b], snaps[b])
    else:
        forced = None if wl.forced_loops is None else [np.full(len(p), wl.forced_loops, np.int32) for p in prompts]
        t_pf = time.time()
        ctx.prefill(ids, prompts, forced=forced, logits=False)
        ctx.prefill_seconds = time.time() - t_pf
        ctx.prefill_tokens = sum(len(p) for p in prompts)
    if snaps is None:
        how = "prefill through the library"
    elif "k" in snaps[0]:
        how = "restored synthetic snapshot (host values)"
    else:
        how = "restored synthetic snapshot (values filled on the device)"
    return ctx, ids, how


def gemm_operands(m, gemm_impl="auto"):
    """Which operand path the decode GEMMs of this model take."""
    if m.dtype != "bf16" or gemm_impl != "auto":
        return "CUDA-core GEMM, operands in the model dtype"
    if os.environ.get("TLF_NO_OPERAND_LO") == "1":
        return "tcgen05, one bf16 plane per activation operand"
    return "tcgen05, two-term bf16 activation operands (hi + lo planes)"


NEAR_TIE = 1e-3


def measure(T, wl, args, rank: int, ws: int, local: int, steps: int, warmup: int, breakdown: bool = True):
    """Prefill the workload through the library, then time decode steps three ways.

    device-timed: CUDA events on the launching stream, logits left on the device;
    end to end: the public call with host token ids in and host logits out (copies timed);
    profiled: per-kernel events, for the attention roofline and the kernel breakdown.
    Returns the raw figures of this rank.
    """
    import torch

    m = wl.model
    B = wl.batch
    t0 = time.time()
    ctx, ids, how = setup_workload(T, wl, rank, prefill=args.prefill, extra_tokens=3 * (warmup + steps),
                                   ablation=args.ablation)
    setup_s = time.time() - t0
    stream = torch.cuda.current_stream()
    n_steps = warmup + steps
    toks = synth.make_decode_tokens(wl, steps=3 * n_steps + 2, batch=B)
    forced = None if wl.forced_loops is None else np.full(B, wl.forced_loops, np.int32)
    logits_dev = torch.empty((B, m.vocab), dtype=torch.float32, device="cuda")
    logits_host = torch.empty((B, m.vocab), dtype=torch.float32).pin_memory().numpy()

    def barrier():
        if ws > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()

    # L2 between timed steps: a step whose working set (weights + the KV pages in use) is at least
    # twice the L2 streams from HBM anyway; a smaller one gets the L2 flushed (a write larger than
    # it) before every timed step, outside the timed intervals.
    eb_w = 2 if m.dtype == "bf16" else 4
    l2_bytes = int(getattr(torch.cuda.get_device_properties(local), "L2_cache_size", 0) or (128 << 20))
    _, free_pages, total_pages = ctx.stats()
    working_set = (m.n_layers * m.layer_params() + m.vocab * m.d_model) * eb_w + \
        (total_pages - free_pages) * T.tlf_page_bytes(ctx.cfg)
    flush_buf = torch.empty(2 * l2_bytes // 4, dtype=torch.int32, device="cuda") if working_set < 2 * l2_bytes \
        else None
    l2_note = ("L2 flushed before every timed step (a %d MB write outside the timed intervals; working set %d MB)"
               % (2 * l2_bytes >> 20, working_set >> 20)) if flush_buf is not None else \
        ("inputs larger than L2 (working set %d MB: KV cache and weights stream from HBM every step)"
         % (working_set >> 20))

    # --- device-timed pass (logits stay on the device) ---
    clocks = ClockSampler(local)
    for s in range(warmup):
        ctx.decode_step(ids, toks[s], forced=forced, logits=logits_dev, stream=stream)
    barrier()
    loops_seen, margins = [], []
    if flush_buf is None:
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
        ev[0].record(stream)
        for s in range(steps):
            _, lp, mg = ctx.decode_step(ids, toks[warmup + s], forced=forced, logits=logits_dev, stream=stream)
            ev[s + 1].record(stream)
            loops_seen.append(lp)
            margins.append(mg)
        barrier()
        step_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(steps)]
        total_ms = ev[0].elapsed_time(ev[-1])
    else:
        st_ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
        en_ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
        for s in range(steps):
            flush_buf.zero_()
            st_ev[s].record(stream)
            _, lp, mg = ctx.decode_step(ids, toks[warmup + s], forced=forced, logits=logits_dev, stream=stream)
            en_ev[s].record(stream)
            loops_seen.append(lp)
            margins.append(mg)
        barrier()
        step_ms = [st_ev[i].elapsed_time(en_ev[i]) for i in range(steps)]
        total_ms = float(sum(step_ms))

    # --- end-to-end pass: host tokens in, host logits out ---
    barrier()
    if flush_buf is None:
        t = time.perf_counter()
        for s in range(steps):
            ctx.decode_step(ids, toks[n_steps + s], forced=forced, logits=logits_host, stream=stream)
        barrier()
        e2e_ms = (time.perf_counter() - t) * 1e3
    else:
        e2e_ms = 0.0
        for s in range(steps):
            flush_buf.zero_()
            torch.cuda.synchronize()
            t = time.perf_counter()
            ctx.decode_step(ids, toks[n_steps + s], forced=forced, logits=logits_host, stream=stream)
            torch.cuda.synchronize()
            e2e_ms += (time.perf_counter() - t) * 1e3
        barrier()
    clk = clocks.stop()

    # --- kernel-level pass: attention kernel time and algorithmic KV bytes ---
    ctx.set_profiling(True)
    att_ms, att_bytes, launches, att_launches = 0.0, 0.0, 0, 0
    kernel_ms = {}
    for s in range(steps):
        ctx.decode_step(ids, toks[2 * n_steps + s], forced=forced, logits=logits_dev, stream=stream)
        ms, by, nl = ctx.last_step_profile()
        att_ms += ms
        att_bytes += by
        launches += nl
        att_launches += m.n_layers * m.max_loops
        if breakdown:
            for kname, kms in ctx.last_step_kernel_times().items():
                kernel_ms[kname] = kernel_ms.get(kname, 0.0) + kms / steps
    ctx.set_profiling(False)

    # algorithmic HBM bytes of the timed steps: the weights of every loop that had an active
    # token (read once per loop), the LM head, and the K/V every active token reads and writes
    eb = 2 if m.dtype == "bf16" else 4
    w_loop = m.n_layers * m.layer_params() * eb
    kv_entry = m.n_layers * 2 * m.n_kv_heads * m.head_dim * eb
    step_bytes = [int(lp.max()) * w_loop + m.vocab * m.d_model * eb + int(lp.sum()) * kv_entry for lp in loops_seen]
    alg_bytes = float(np.mean(step_bytes)) + att_bytes / steps
    r = dict(total_ms=total_ms, e2e_ms=e2e_ms, step_ms=step_ms, att_ms=att_ms, att_bytes=att_bytes,
             launches=launches, att_launches=att_launches, kernel_ms=kernel_ms, alg_bytes=alg_bytes,
             loops=np.concatenate(loops_seen), margins=np.concatenate(margins), how=how, l2_note=l2_note,
             setup_s=setup_s, clocks=clk,
             prefill=({"tokens": ctx.prefill_tokens, "seconds": ctx.prefill_seconds,
                       "tokens_per_s": ctx.prefill_tokens / ctx.prefill_seconds}
                      if hasattr(ctx, "prefill_seconds") else None))
    ctx.close()
    return r


def summarize(wl, r, steps: int, ws: int, total_ms: float, e2e_ms: float, peak: float, peak_kind: str):
    """Per-workload figures of the JSON line (rank 0, times already maxed over ranks)."""
    m = wl.model
    B = wl.batch
    att_gbs = r["att_bytes"] / (r["att_ms"] * 1e-3) / 1e9 if r["att_ms"] > 0 else None
    near = int(np.sum(np.abs(r["margins"]) <= NEAR_TIE)) if wl.forced_loops is None else 0
    return {
        "tokens_per_s": job_tokens_per_s(ws, B, steps, total_ms),
        "ms_per_step": total_ms / steps,
        "p50_step_ms": float(np.percentile(r["step_ms"], 50)),
        "p90_step_ms": float(np.percentile(r["step_ms"], 90)),
        "e2e_tokens_per_s": job_tokens_per_s(ws, B, steps, e2e_ms),
        "step_roofline_frac": (r["alg_bytes"] / (peak * 1e9) * 1e3) / (total_ms / steps),
        "step_floor_ms": r["alg_bytes"] / (peak * 1e9) * 1e3,
        "attention_gbs": att_gbs,
        "attention_frac": (att_gbs / peak) if att_gbs else None,
        "mean_loops": float(r["loops"].mean()),
        "depth_histogram": np.bincount(r["loops"], minlength=m.max_loops + 1)[1:].tolist(),
        "near_tie_tokens": near,
        "near_tie_rule": ("router margin <= 1e-3 among the timed tokens" if wl.forced_loops is None
                          else "every token forced to %d loops: no router decision" % wl.forced_loops),
        "gpu_launches": int(r["launches"]),
    }


# The five workloads beside the headline one, each timed in the same run (at one GPU).
SUB_CONFIGS = ("c1", "c2", "c3", "c5", "c5f")


def run_ours(args):
    import torch

    from paper_2609_15160_gb300 import tlf as T

    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    T.load_library()
    wl = synth.get_config(args.config)
    if args.decode_batch:
        wl = wl.with_batch(args.decode_batch)
    m = wl.model
    B = wl.batch
    r = measure(T, wl, args, rank, ws, local, args.steps, args.warmup)
    total_ms, e2e_ms = max_over_ranks([r["total_ms"], r["e2e_ms"]], device="cuda")
    peak, peak_kind = _measured_peaks()
    configs = {}
    if ws == 1 and not args.no_configs:
        for name in SUB_CONFIGS:
            if name == args.config:
                continue
            swl = synth.get_config(name)
            sr = measure(T, swl, args, rank, ws, local, args.steps, args.warmup, breakdown=False)
            configs[name] = {"workload": DESCR[name], "batch": swl.batch, "cache": sr["how"], "l2": sr["l2_note"],
                             "gemm_operands": gemm_operands(swl.model),
                             **summarize(swl, sr, args.steps, ws, sr["total_ms"], sr["e2e_ms"], peak, peak_kind),
                             "clocks": sr["clocks"]}
    if rank == 0:
        s = summarize(wl, r, args.steps, ws, total_ms, e2e_ms, peak, peak_kind)
        att_gbs = s["attention_gbs"]
        h2d = B * 12
        d2h = B * m.vocab * 4 + B * 8
        line = {
            "metric": "decode_tokens_per_s", "value": s["tokens_per_s"], "unit": "tokens/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": s["ms_per_step"],
            "p50_step_ms": s["p50_step_ms"], "p90_step_ms": s["p90_step_ms"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": m.dtype,
            "data": "synthetic",
            "config": {"workload": DESCR[args.config], "name": args.config, "batch_per_gpu": B,
                       "context": int(wl.prompt_len[1]), "cache": r["how"],
                       "l2": r["l2_note"],
                       "parallelism": f"replicas x{ws} (independent sequences per GPU)",
                       "ablation": args.ablation, "gemm_operands": gemm_operands(m)},
            "mean_loops": s["mean_loops"],
            "near_tie_tokens": s["near_tie_tokens"],
            "step_roofline": {"bound": "hbm", "algorithmic_bytes_per_step": r["alg_bytes"],
                              "floor_ms": s["step_floor_ms"], "frac": s["step_roofline_frac"],
                              "peak_gbs": peak, "peak_kind": peak_kind},
            "attention_gbs": att_gbs,
            "roofline": {"bound": "hbm", "kernel": "k_attn_decode (recursion-wise split-K attention)",
                         "achieved": att_gbs, "peak": peak, "unit": "GB/s",
                         "frac": (att_gbs / peak) if att_gbs else None, "peak_kind": peak_kind,
                         "traffic": _attn_traffic(r["att_bytes"] / max(1, r["att_launches"])),
                         "traffic_source": "ncu dram bytes / algorithmic bytes of one captured launch "
                                           "(profiles/traffic.json) x this launch's algorithmic bytes",
                         "algorithmic_bytes_per_launch": r["att_bytes"] / max(1, r["att_launches"]),
                         "avg_launch_ms": r["att_ms"] / max(1, r["att_launches"])},
            "e2e": {"value": s["e2e_tokens_per_s"], "unit": "tokens/s",
                    "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": s["gpu_launches"],
            "kernel_ms_per_step_profiled": {k: round(v, 4) for k, v in r["kernel_ms"].items()},
            "setup_s": r["setup_s"],
            "prefill": r["prefill"],
        }
        if r["clocks"]:
            line["clocks"] = r["clocks"]
        if configs:
            line["configs"] = configs
        if not args.no_cpu_baseline and ws == 1:
            line["cpu_baseline"] = cpu_baseline(args.config)
        print(json.dumps(line))
    if ws > 1:
        torch.distributed.destroy_process_group()


def run_attn_op(args):
    """The recursion-wise attention kernels alone (tlf_attn_decode) on C4 shapes: GB/s of K/V streamed."""
    import torch

    from paper_2609_15160_gb300 import tlf as T

    T.load_library()
    n, L = args.batch, args.context
    hq, hkv, hd, J = args.hq, args.hkv, args.hd, args.layers
    rng = np.random.default_rng(5)
    need = (L + 63) // 64
    n_pages = n * need + 1
    # pool of bf16 bit patterns of multiples of 1/64 in [-2, 2), built without a float32 copy
    table = (np.arange(-128, 128, dtype=np.float32) / 64.0).view(np.uint32) >> 16
    pool = torch.empty((n_pages, J, 2, hkv, 64, hd), dtype=torch.int16, device="cuda")
    for p0 in range(0, n_pages, 256):
        p1 = min(n_pages, p0 + 256)
        codes = rng.integers(0, 256, size=(p1 - p0, J, 2, hkv, 64, hd), dtype=np.int16)
        pool[p0:p1] = torch.from_numpy(table[codes].astype(np.uint16).view(np.int16))
    pt = torch.from_numpy(rng.permutation(n_pages)[: n * need].reshape(n, need).astype(np.int32)).cuda()
    lens = torch.full((n,), L, dtype=torch.int32, device="cuda")
    q = torch.randn((n, hq, hd), dtype=torch.float32, device="cuda")
    out = torch.empty((n, hq * hd), dtype=torch.int16, device="cuda")
    err = torch.zeros(4, dtype=torch.int32, device="cuda")
    a = T.attn_args(n, hq, hkv, hd, J, 1, "bf16", need, n_pages, q, pool, pt, lens, out, err)
    nbytes = T.tlf_attn_decode_scratch_bytes(a)
    scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        T.tlf_attn_decode(a, scratch, nbytes, stream)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    ev[0].record(stream)
    for s in range(args.steps):
        T.tlf_attn_decode(a, scratch, nbytes, stream)
        ev[s + 1].record(stream)
    torch.cuda.synchronize()
    assert int(err[0].item()) == 0, "device error word set"
    ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)]
    kv_bytes = n * L * hkv * hd * 2 * 2
    io_bytes = n * hq * hd * (4 + 2)
    peak, kind = _measured_peaks()
    med = float(np.median(ms))
    gbs = (kv_bytes + io_bytes) / (med * 1e-3) / 1e9
    print(json.dumps({"metric": "attention_op_gbs", "value": gbs, "unit": "GB/s", "steps": args.steps,
                      "warmup": args.warmup, "ms_per_call_p50": med, "higher_is_better": True,
                      "config": {"op": "tlf_attn_decode", "rows": n, "keys_per_row": L, "hq": hq, "hkv": hkv,
                                 "head_dim": hd, "dtype": "bf16", "l2": "K/V larger than L2"},
                      "roofline": {"bound": "hbm", "achieved": gbs, "peak": peak, "unit": "GB/s",
                                   "frac": gbs / peak, "peak_kind": kind,
                                   "algorithmic_bytes_per_call": kv_bytes + io_bytes}}))


def run_sweep(args):
    """Decode throughput and mean depth under the SURVIVAL rule of Eq. 4 at several thresholds.

    The paper sweeps the router threshold (Fig. 4c: perplexity and average depth); here the
    workload's model is rebuilt with exit_rule = survival at each threshold (optionally with the
    two-layer MLP router), its prompts are prefilled through the library (so the cached tokens carry
    that threshold's routing too), and decode steps are timed with CUDA events. The ARGMAX rule of
    the workload is the first row.
    """
    import dataclasses

    import torch

    from paper_2609_15160_gb300 import tlf as T

    T.load_library()
    wl0 = synth.get_config(args.config)
    rows = []
    variants = [("argmax", None)] + [("survival", float(t)) for t in args.thresholds.split(",")]
    for rule, th in variants:
        m = dataclasses.replace(wl0.model, exit_rule=rule, threshold=th if th is not None else 0.5,
                                router_hidden=args.router_hidden)
        wl = dataclasses.replace(wl0, model=m)
        t0 = time.time()
        ctx, ids, how = setup_workload(T, wl, 0, prefill=args.prefill, extra_tokens=args.warmup + args.steps + 2)
        setup_s = time.time() - t0
        B = wl.batch
        toks = synth.make_decode_tokens(wl, steps=args.warmup + args.steps, batch=B)
        logits = torch.empty((B, m.vocab), dtype=torch.float32, device="cuda")
        st = torch.cuda.current_stream()
        for k in range(args.warmup):
            ctx.decode_step(ids, toks[k], logits=logits, stream=st)
        torch.cuda.synchronize()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        loops = []
        ev[0].record(st)
        for k in range(args.steps):
            _, lp, _ = ctx.decode_step(ids, toks[args.warmup + k], logits=logits, stream=st)
            loops.append(lp)
        ev[1].record(st)
        torch.cuda.synchronize()
        ms = ev[0].elapsed_time(ev[1]) / args.steps
        lp = np.concatenate(loops)
        rows.append({"exit_rule": rule, "threshold": th, "ms_per_step": ms, "tokens_per_s": B / (ms * 1e-3),
                     "mean_loops": float(lp.mean()),
                     "depth_histogram": np.bincount(lp, minlength=m.max_loops + 1)[1:].tolist(),
                     "cache": how, "setup_s": setup_s})
        ctx.close()
    print(json.dumps({"metric": "decode_tokens_per_s_vs_router_threshold", "unit": "tokens/s",
                      "higher_is_better": True, "steps": args.steps, "warmup": args.warmup, "dtype": wl0.model.dtype,
                      "data": "synthetic",
                      "config": {"workload": DESCR[args.config], "name": args.config,
                                 "router": f"two-layer MLP, hidden {args.router_hidden}" if args.router_hidden
                                 else "linear"},
                      "sweep": rows}))


def run_ttft(args):
    """Time to first token: one prompt of each length through tlf_prefill (logits of its last token).

    The paper reports TTFT for prompts of 128, 512, 1024 and 2048 tokens (Fig. 4d); the prompts here are
    seeded uniform random ids on the chosen workload's model. Also reports the prefill throughput of the
    workload's whole batch of prompts (--full).
    """
    import torch

    from paper_2609_15160_gb300 import tlf as T

    T.load_library()
    wl = synth.get_config(args.config)
    m = wl.model
    w = synth.make_weights(m)
    lengths = [int(x) for x in args.ttft_lengths.split(",")]
    B = wl.batch
    full_prompts = synth.make_prompts(wl) if args.full else []
    max_len = max(lengths + [len(p) for p in full_prompts])
    n_pages = max(len(full_prompts), 1) * m.max_loops * ((max_len + 63) // 64 + 2) + 64
    ctx = T.Context(m, w, max_seqs=max(B, 2), max_batch=min(B, 256), max_seq_len=max_len + 8,
                    kv_pool_pages=n_pages)
    rng = np.random.default_rng(4)
    out = []
    for L in lengths:
        prompt = rng.integers(0, m.vocab, size=L).astype(np.int32)
        times = []
        for it in range(args.warmup + args.steps):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            ctx.prefill([7], [prompt])
            times.append(time.perf_counter() - t0)
            ctx.release(7)
        ms = 1e3 * float(np.median(times[args.warmup:]))
        out.append({"prompt_len": L, "ttft_ms": ms})
    line = {"metric": "ttft_ms", "unit": "ms", "higher_is_better": False, "config": {"workload": DESCR[args.config],
            "model": args.config, "dtype": m.dtype, "data": "synthetic uniform random prompts"}, "ttft": out}
    if args.full:
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        ctx.prefill(list(range(100, 100 + B)), full_prompts, logits=False)
        torch.cuda.synchronize()
        sec = time.perf_counter() - t0
        ntok = sum(len(p) for p in full_prompts)
        line["full_prefill"] = {"sequences": B, "tokens": ntok, "seconds": sec, "tokens_per_s": ntok / sec}
    print(json.dumps(line))
    ctx.close()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--op", default=None, choices=["attn", "ttft", "sweep"],
                    help="time one operation alone: the attention kernels, prefill (time to first token), "
                         "or decode under the survival rule at several thresholds")
    ap.add_argument("--thresholds", default="0.2,0.3,0.4,0.5,0.6,0.7,0.8", help="--op sweep: survival thresholds")
    ap.add_argument("--router-hidden", type=int, default=0,
                    help="--op sweep: hidden width of the two-layer MLP router (0 = the workload's linear router)")
    ap.add_argument("--ttft-lengths", default="128,512,1024,2048")
    ap.add_argument("--full", action="store_true", help="--op ttft: also prefill the workload's whole batch")
    ap.add_argument("--batch", type=int, default=16)
    ap.add_argument("--context", type=int, default=32768)
    ap.add_argument("--hq", type=int, default=16, help="--op attn: query heads")
    ap.add_argument("--hkv", type=int, default=8, help="--op attn: kv heads")
    ap.add_argument("--hd", type=int, default=128, help="--op attn: head dim")
    ap.add_argument("--layers", type=int, default=2, help="--op attn: layers stored per page")
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--config", default="c4", choices=sorted(DESCR))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--prefill", default="auto", choices=["auto", "snapshot", "real"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="time only the chosen workload (by default a 1-GPU run also times C1, C2, C3, C5 "
                         "routed and C5 forced-8 and reports them under configs)")
    ap.add_argument("--decode-batch", type=int, default=0, help="override the workload's batch (C5 sweep)")
    ap.add_argument("--ablation", default="none", choices=["none", "no_gather", "dense_cache"],
                    help="no_gather: all rows every loop, exited rows masked (no gather of Eq. 6); "
                         "dense_cache: full-length loop caches read under the mask of Eq. 10 "
                         "(no recursion-wise cache)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.op == "attn":
        run_attn_op(args)
    elif args.op == "ttft":
        run_ttft(args)
    elif args.op == "sweep":
        run_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
