"""Benchmark of the CAI-dLLM fused decoding head + commit rule on GB300.

One bench "step" is one whole generation of the workload: every block, each
block run step by step (step zero, then denoising steps until every sequence
exits, with the host polling the device's done flag one step behind), every
step being gather -> LM head with online softmax -> merge + commit.  The metric
is masked positions decoded per second, summed over all steps (sum of M_t)
and over all ranks, divided by the device time of the timed region.

Default workload (N = 1): LLaDA-8B-shaped, B = 1, H = 4096, V = 126464,
generation length 256 in 8 blocks of 32, up to 32 steps per block, seeded
synthetic bf16 weight and hidden states (``synth``).  The weight (1.04 GB) is
larger than L2, so every step reads it from HBM.

Arms:
  (default)          the sm_103a path through the C ABI (``paper_2608_22646_gb300``);
  --impl reference   the fp64 CPU oracle as it stands, on the host cores, on a
                     bounded sample of the same workload (there is no published
                     implementation of the method to run).

Multi-GPU: under torchrun each rank decodes its own batch (sequences are
independent, no collective on the data path); value = all ranks' positions /
the slowest rank's time ("weak" scaling).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "masked positions decoded/s (fused head+commit) at 1 GB300; % of HBM/tensor roofline"
UNIT = "positions/s"
FINAL_NORM_EPS = 1e-5
PROFILES = os.path.join(ROOT, "profiles")


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained"), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def _workload_desc(wl, gen):
    return {"workload": f"{wl.name}: B={wl.B} H={wl.H} V={wl.V} gen_len={wl.gen_len} "
                        f"block={wl.P} T={wl.T}",
            "B": wl.B, "H": wl.H, "V": wl.V, "gen_len": wl.gen_len, "block": wl.P,
            "max_steps_per_block": wl.T, "hidden_generator": gen,
            "l2": ("inputs larger than L2 (LM-head weight %.2f GB read every step)"
                   % (wl.V * wl.H * 2 / 1e9)) if wl.V * wl.H * 2 > 129e6 else
                  "weight fits in L2 (small case; not a bench workload)"}


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during a region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = os.path.join("/tmp", f"cai_clocks_{os.getpid()}.csv")

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, ValueError):
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return None
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx = float(parts[2])
                except ValueError:
                    continue
                for n, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(n)
        os.remove(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def source_code_sha(path: str) -> str:
    """sha256 prefix of a kernel source's code and of the local headers it
    includes (recursively, each once): comments and blank lines removed, so
    that a comment edit does not count as a change of the kernel."""
    import re
    seen, parts = set(), []

    def add(fp):
        fp = os.path.normpath(fp)
        if fp in seen or not os.path.exists(fp):
            return
        seen.add(fp)
        with open(fp) as f:
            s = f.read()
        for inc in re.findall(r'^\s*#\s*include\s+"([^"]+)"', s, flags=re.M):
            add(os.path.join(os.path.dirname(fp), inc))
        s = re.sub(r"/\*.*?\*/", "", s, flags=re.S)
        s = re.sub(r"//[^\n]*", "", s)
        parts.append("\n".join(line.rstrip() for line in s.splitlines() if line.strip()))

    add(path)
    return hashlib.sha256("\n".join(parts).encode()).hexdigest()[:16]


def _traffic_record(workload: str):
    """DRAM bytes per launch of the workload's dominant LM-head kernel from the
    committed ncu summaries, if they were taken on the current kernel code."""
    p = os.path.join(PROFILES, "lm_head_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        recs = json.load(f).get("records", [])
    for rec in recs:
        if rec.get("workload") != workload:
            continue
        src = os.path.join(ROOT, "paper_2608_22646_gb300", "csrc", rec["source"])
        if not os.path.exists(src):
            return None
        return rec if rec.get("source_code_sha") == source_code_sha(src) else None
    return None


def run_trajectory(cai, ctx, hidden, wl, lag_poll=True, stream=None):
    """All blocks of one generation.  ``hidden[blk][t]`` is the step's input.
    A kernel's failed bounded wait raises with the device error bits named."""
    try:
        for blk in range(wl.n_blocks):
            if blk:
                cai.cai_block_advance(ctx, stream)
            cai.cai_first_step(ctx, hidden[blk][0], stream)
            for t in range(1, wl.T):
                if lag_poll and t >= 2 and cai.cai_poll(ctx, 1, 60000):
                    break
                cai.cai_denoise_step(ctx, hidden[blk][t], stream)
    except cai.CaiError as e:
        if e.status == cai.CAI_ERR_DEVICE:
            bits = cai.cai_device_error_bits(ctx)
            names = [n for k, n in enumerate(cai.DEVERR_NAMES) if bits >> k & 1]
            e.args = (f"{e.args[0]} [device error bits {bits:#x}: {', '.join(names)}]",)
        raise


def cpu_baseline(wl, W, hs_fn, budget_s: float = 12.0, norm=None):
    """The oracle as it stands on the host cores: full steps of the same
    trajectory (all masked rows of each step), for about budget_s seconds.
    ``norm`` = (weight, eps) when the final RMSNorm is part of the head."""
    import oracle
    cfg = oracle.Config(B=wl.B, P=wl.P, T=wl.T, n_blocks=wl.n_blocks)
    st = oracle.State(cfg)
    Wb = oracle.bf16_bits(W)
    threads = os.cpu_count() or 1
    rows = 0
    steps = 0
    t0 = time.perf_counter()
    for blk in range(wl.n_blocks):
        for t in range(wl.T):
            h = oracle.bf16_bits(hs_fn(blk, t))
            out = oracle.step(st, Wb, h, blk, t, threads, *(norm or ()))
            rows += out["M"]
            steps += 1
            if np.all(st.exit_reason[:, blk] != 0) or time.perf_counter() - t0 > budget_s:
                break
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    return {"value": rows / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"first {steps} denoising steps of the trajectory ({rows} masked rows, "
                      f"fp64, one thread per row), {dt:.1f} s"}


def _trajectory_summary(st: dict) -> dict:
    """One generation of the workload: steps per block (max over the batch),
    the masked rows M_t decoded at each step of each block, exits by reason,
    tokens left unresolved, and the step-zero budgets."""
    ex = st["exit_reason"]
    reasons = {"done": 1, "grinding": 2, "t_exhausted": 3}
    bud = st["budget"].reshape(-1)
    steps = st["exit_step"].max(axis=0) + 1
    return {"steps_per_block": [int(x) for x in steps],
            "m_t": [[int(m) for m in st["m_hist"][b, :int(steps[b])]] for b in range(len(steps))],
            "exits": {k: int((ex == v).sum()) for k, v in reasons.items()},
            "unresolved_tokens": int(st["unresolved"].sum()),
            "budgets": {str(b): int((bud == b).sum()) for b in (8, 32, 64)}}


def _diagnostics_summary(st: dict) -> dict:
    """Stability step t_i^* against the first-step confidence s_i (the shape of
    Section 2.1's token pattern), and the mean drift D^(t) per block."""
    s0, stable = st["s0"].reshape(-1), st["stable"].reshape(-1).astype(np.int64)
    out = {}
    for name, sel in (("s0>0.50", s0 > 0.5), ("0.25<=s0<=0.50", (s0 >= 0.25) & (s0 <= 0.5)),
                      ("s0<0.25", (s0 < 0.25) & (s0 > 0))):
        ts = stable[sel & (stable >= 0)]
        out[name] = {"tokens": int(sel.sum()), "stable": int(ts.size),
                     "mean_t_star": round(float(ts.mean()), 2) if ts.size else None}
    d = st["drift"]
    out["mean_drift_per_block"] = [round(float(np.nanmean(d[:, b, :])), 4)
                                   if np.isfinite(d[:, b, :]).any() else None
                                   for b in range(d.shape[1])]
    return out


def pg_timeout():
    """Process-group timeout: a rank that died leaves the others' next barrier
    or collective failing after this long instead of waiting for ever
    (CAI_PG_TIMEOUT_S, default 300 s)."""
    import datetime
    return datetime.timedelta(seconds=float(os.environ.get("CAI_PG_TIMEOUT_S", "300")))


def aggregate(ms: float, positions: int, dist=None, device=None):
    """Whole-job figures over ranks: the slowest rank's time and the sum of
    every rank's decoded positions (each rank decodes its own batch)."""
    if dist is None:
        return ms, positions
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    n = torch.tensor([positions], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), int(n.item())


def _roofline(wl, st0, stats1, head_ms, head_launches, step_ms, ms, steps, steps_issued,
              profiled):
    """Roofline of the dominant kernel (the LM head), launch by launch: a
    launch that decodes M rows reads 2 V H + 2 M H bytes (W once, the rows
    once) and does 2 M V H flops; its roof is the slower of the two at the
    measured peaks.  Launches of empty steps (M = 0) have no algorithmic work.

    achieved / frac: algorithmic work per launch / the LM head's average
    launch duration, from CUDA events around every LM-head launch on its
    stream (the profiled pass: each launch runs alone, with its launch latency
    and, in single-kernel steps, the commit tail; this is the figure that
    carries over to a decoder whose model forward runs between two steps).
    live: the same work over the timed region of back-to-back generations
    times the LM head's share of step time (consecutive steps overlap there)."""
    hbm, tf_burst, tf_sus, peak_kind = _peaks()
    tf = tf_sus or tf_burst
    m_t = [int(x) for x in st0["m_hist"].reshape(-1) if x > 0]
    bytes_t = [2.0 * wl.V * wl.H + 2.0 * m * wl.H for m in m_t]
    flops_t = [2.0 * m * wl.V * wl.H for m in m_t]
    t_hbm = sum(b / (hbm * 1e9) for b in bytes_t)
    t_tc = sum(f / (tf * 1e12) for f in flops_t)
    t_roof = sum(max(b / (hbm * 1e9), f / (tf * 1e12)) for b, f in zip(bytes_t, flops_t))
    share = min(1.0, head_ms / step_ms) if step_ms > 0 else 1.0
    head_live_s = ms / 1e3 / steps * share
    head_iso_s = (head_ms / 1e3 / steps) if profiled and head_ms > 0 else head_live_s
    per_launch = max(1, (head_launches if head_launches else int(steps_issued) * steps) // steps)
    kps = int(stats1["kernels_per_step"])
    if kps == 1 and stats1.get("head_rows"):
        kernel = ("lm_head_rows_kernel (single-kernel step: LM head with the rows as the MMA's A "
                  "operand, softmax and commit)")
    elif kps == 1:
        kernel = "lm_head_softmax_kernel (single-kernel step: LM head, softmax and commit)"
    elif stats1["pair_swap_max_n"] >= 32:
        kernel = (f"lm_head_pair_kernel (every step; swapped orientation for tiles up to "
                  f"{stats1['pair_swap_max_n']} rows wide)")
    elif stats1["pair_grid"]:
        kernel = "lm_head_pair_kernel (>= 32 rows) / lm_head_softmax_kernel (< 32 rows)"
    else:
        kernel = "lm_head_softmax_kernel"
    tr = _traffic_record(wl.name)
    hb = t_hbm >= t_tc
    work = sum(bytes_t) if hb else sum(flops_t)
    scale = 1e9 if hb else 1e12
    peak = hbm if hb else tf
    achieved = work / head_iso_s / scale
    live = work / head_live_s / scale
    roof = {"bound": "hbm" if hb else "tensor", "achieved": round(achieved, 1), "peak": peak,
            "unit": "GB/s" if hb else "TFLOP/s", "frac": round(achieved / peak, 4),
            "traffic": tr["dram_bytes_per_launch"] if tr else None,
            "traffic_basis": ("ncu dram read+write of one launch with M = %d (%s); algorithmic "
                              "bytes of that launch %d" % (
                                  tr["captured_M"], tr["summary"],
                                  tr["algorithmic_bytes_of_profiled_launch"])) if tr else None,
            ("algorithmic_bytes_per_launch" if hb else "algorithmic_flops_per_launch"):
                round(work / per_launch),
            "peak_source": f"{peak_kind} " + ("hbm_gbs" if hb else "bf16 sustained"),
            "kernel": kernel, "head_launches": head_launches,
            "avg_launch_us": round(head_iso_s / per_launch * 1e6, 2),
            "roofline_time_frac": round(t_roof / head_iso_s, 4),
            "live": {"achieved": round(live, 1), "frac": round(live / peak, 4),
                     "roofline_time_frac": round(t_roof / head_live_s, 4),
                     "head_share_of_step_time": round(share, 4)},
            "timing": "achieved/frac: CUDA events around every LM-head launch on its stream in a "
                      "second pass of the same K generations (each launch alone); live: CUDA "
                      "events around the timed region of K generations back to back times the "
                      "LM head's share of step time (consecutive steps overlap under "
                      "programmatic dependent launch)"}
    return roof


def measure(cai, wl, generator, args, dist, dev, steps, warmup, with_e2e=True, cpu_leg=False):
    """One workload: `warmup` untimed generations, `steps` timed ones (the
    value), a profiled pass (the roofline), the end-to-end pass through host
    buffers, and optionally the oracle's CPU baseline."""
    import torch
    import synth
    rank = int(os.environ.get("RANK", "0"))
    local = dev.index or 0
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w, device=dev)
    hs = synth.HiddenStates(wl, W, generator, seed=wl.seed_h + 1000 * rank)
    norm = None
    if args.final_norm:
        norm = (synth.final_norm_weight(wl.H, device=dev), FINAL_NORM_EPS)
        hs = synth.PreNormHidden(hs)
    hidden = [[hs(blk, t) for t in range(wl.T)] for blk in range(wl.n_blocks)]
    torch.cuda.synchronize()

    cfg = cai.cai_config_default(cai.CAI_PRESET_LLADA, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    if args.diagnostics:
        cfg.flags |= cai.CAI_DIAGNOSTICS
    ctx = cai.cai_init_rmsnorm(cfg, W, *norm) if norm else cai.cai_init(cfg, W)
    stream = torch.cuda.current_stream(dev)

    for _ in range(warmup):
        cai.cai_reset(ctx)
        run_trajectory(cai, ctx, hidden, wl)
    torch.cuda.synchronize()
    st0 = cai.cai_state_download(ctx)
    positions = int(st0["m_hist"].sum())
    nonzero_launch = int((st0["m_hist"] > 0).sum())   # steps that decoded rows
    stats0 = cai.cai_get_stats(ctx)

    # Timed region 1 (the value): K generations back to back, device time by
    # CUDA events on the stream, no per-kernel events in between (an event
    # between two kernels serialises them and would defeat the programmatic
    # dependent launch the library uses).
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with Clocks(local) as clk:
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        for _ in range(steps):
            cai.cai_reset(ctx)
            run_trajectory(cai, ctx, hidden, wl)
        ev1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
    ms = ev0.elapsed_time(ev1)
    stats1 = cai.cai_get_stats(ctx)
    st1 = cai.cai_state_download(ctx)
    assert np.array_equal(st1["m_hist"], st0["m_hist"]), "trajectory changed between runs"
    gpu_launches = stats1["launches"] - stats0["launches"]
    steps_issued = (stats1["steps"] - stats0["steps"]) // steps

    # Timed region 2 (the roofline figure): the same K generations with CUDA
    # events around every step and its LM-head launch(es) on the stream.
    head_ms, head_launches, step_ms = 0.0, 0, 0.0
    if not args.no_profile:
        cai.cai_profile(ctx, True)
        torch.cuda.synchronize()
        for _ in range(steps):
            cai.cai_reset(ctx)
            run_trajectory(cai, ctx, hidden, wl)
        torch.cuda.synchronize()
        cai.cai_profile(ctx, False)
        stats2 = cai.cai_get_stats(ctx)
        head_launches = stats2["head_launches"] - stats1["head_launches"]
        head_ms = stats2["head_ms"] - stats1["head_ms"]
        step_ms = stats2["step_ms"] - stats1["step_ms"]

    ms, total_positions = aggregate(ms, positions * steps, dist, dev)
    rec = {
        "value": round(total_positions / (ms / 1e3), 1), "unit": UNIT,
        "ms_per_generation": round(ms / steps, 4),
        "ms_per_step_call": round(ms / steps / max(1, steps_issued), 5),
        "config": {**_workload_desc(wl, generator),
                   "final_norm_in_head": bool(args.final_norm),
                   "positions_per_generation": positions,
                   "denoising_steps_per_generation": nonzero_launch,
                   "step_calls_per_generation": int(steps_issued)},
        "roofline": _roofline(wl, st0, stats1, head_ms, head_launches, step_ms, ms, steps,
                              steps_issued, not args.no_profile),
        "trajectory": _trajectory_summary(st0),
        "gpu_launches": int(gpu_launches),
        "clocks": clk.summary(),
    }
    if args.diagnostics:
        rec["config"]["diagnostics"] = True
        rec["diagnostics"] = _diagnostics_summary(st0)
    if with_e2e and not args.no_e2e:
        rec["e2e"] = e2e_run(cai, ctx, hs, wl, max(3, steps // 3), dist, dev)
    if cpu_leg:
        rec["cpu_baseline"] = cpu_baseline(wl, W, lambda b, t: hidden[b][t], norm=norm)
    cai.cai_free(ctx)
    del hidden, W, hs
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return rec


# The other configurations measured beside the headline workload (N = 1):
# name in the line -> (workload, hidden-state generator).
EXTRA_WORKLOADS = {
    "dream": ("dream", "calibrated"),
    "llada_batched": ("llada_batched", "calibrated"),
    "dream_long": ("dream_long", "calibrated"),
    "llada_literal": ("llada", "literal"),
}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llada")
    ap.add_argument("--generator", default="calibrated", choices=["calibrated", "literal"])
    ap.add_argument("--extra", default=None,
                    help="comma-separated names of EXTRA_WORKLOADS measured beside the headline "
                         "(default: all of them at N = 1 on the default workload, none otherwise)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-profile", action="store_true",
                    help="time the region without per-kernel events (no roofline figure)")
    ap.add_argument("--diagnostics", action="store_true",
                    help="track stability steps and hidden-state drift (CAI_DIAGNOSTICS) and "
                         "summarise them in the line")
    ap.add_argument("--vocab-shards", type=int, default=0,
                    help="measure the vocabulary-parallel head over this many shards instead "
                         "(one per rank under torchrun; all on this GPU otherwise)")
    ap.add_argument("--final-norm", action="store_true",
                    help="the model's final RMSNorm inside the head (cai_init_rmsnorm): inputs "
                         "are the rows before that norm")
    args = ap.parse_args()

    import torch
    import synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local), timeout=pg_timeout())
    wl = synth.WORKLOADS[args.workload]

    if args.impl == "reference":
        if rank != 0:
            if dist:
                dist.barrier()
                dist.destroy_process_group()
            return
        run_reference(args, wl)
        if dist:
            dist.barrier()
            dist.destroy_process_group()
        return

    import paper_2608_22646_gb300 as cai
    from paper_2608_22646_gb300 import build as cai_build
    cai_build.build()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    if args.vocab_shards > 0:
        run_vocab_shards(cai, args, wl, dist, dev, world, rank)
        if dist:
            dist.destroy_process_group()
        return

    head = measure(cai, wl, args.generator, args, dist, dev, args.steps, args.warmup,
                   cpu_leg=(rank == 0 and world == 1 and not args.no_cpu_baseline))
    if args.extra is None:
        default = (world == 1 and args.workload == "llada" and args.generator == "calibrated"
                   and not args.final_norm and not args.diagnostics)
        extra = list(EXTRA_WORKLOADS) if default else []
    else:
        extra = [x for x in args.extra.split(",") if x]
    workloads = {}
    for name in extra:
        wname, gen = EXTRA_WORKLOADS[name]
        r = measure(cai, synth.WORKLOADS[wname], gen, args, dist, dev, args.steps, args.warmup)
        workloads[name] = r

    cfg = head["config"]
    line = {
        "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": head["ms_per_generation"],
        "step_unit": (f"one bench step = one whole generation of the workload "
                      f"({cfg['step_calls_per_generation']} step calls, "
                      f"{cfg['positions_per_generation']} masked positions decoded)"),
        "ms_per_generation": head["ms_per_generation"],
        "ms_per_step_call": head["ms_per_step_call"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded LLaDA/Dream-shaped weight and hidden states; no model weights)",
        "config": {**cfg, "parallelism": f"replicas x{world}",
                   "positions_per_step": cfg["positions_per_generation"]},
        "roofline": head["roofline"],
        "trajectory": head["trajectory"],
        "gpu_launches": head["gpu_launches"],
        "clocks": head["clocks"],
    }
    for k in ("diagnostics", "e2e", "cpu_baseline"):
        if k in head:
            line[k] = head[k]
    if workloads:
        line["workloads"] = workloads
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def e2e_run(cai, ctx, hs, wl, steps, dist, dev):
    """Same metric through the public C ABI with host buffers: every step's
    hidden states come from pinned host memory (copied inside the step call),
    every step's done flag is read from host-mapped memory, and each
    generation's tokens are copied back to pinned host memory."""
    import torch
    host = [[hs(blk, t).cpu().pin_memory() for t in range(wl.T)] for blk in range(wl.n_blocks)]
    out = torch.empty((wl.B, wl.n_blocks * wl.P), dtype=torch.int32).pin_memory()
    stream = torch.cuda.current_stream(dev)
    cai.cai_reset(ctx)
    run_trajectory(cai, ctx, host, wl)
    cai.cai_read_tokens(ctx, out)
    torch.cuda.synchronize()
    s0 = cai.cai_get_stats(ctx)["steps"]
    if dist:
        dist.barrier()
    t0 = time.perf_counter()
    for _ in range(steps):
        cai.cai_reset(ctx)
        run_trajectory(cai, ctx, host, wl)
        cai.cai_read_tokens(ctx, out)
        stream.synchronize()
    dt = time.perf_counter() - t0
    st = cai.cai_state_download(ctx)
    n_step_calls = (cai.cai_get_stats(ctx)["steps"] - s0) / steps
    dt_ms, positions = aggregate(dt * 1e3, int(st["m_hist"].sum()) * steps, dist, dev)
    # Every step call copies the block's rows ([B, P, H] bf16) to the device.
    h2d = n_step_calls * wl.B * wl.P * wl.H * 2
    return {"value": round(positions / (dt_ms / 1e3), 1), "unit": UNIT,
            "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(wl.B * wl.n_blocks * wl.P * 4 + n_step_calls * 32),
            "timing": "host wall clock around whole generations, pinned host inputs (each step "
                      "call's rows copied on the context's side stream while the previous step "
                      "runs)"}


def run_vocab_shards(cai, args, wl, dist, dev, world, rank):
    """``--vocab-shards G``: the vocabulary-parallel head on the workload.  With
    G ranks under torchrun each rank holds one slice of W (one shard context)
    and a step is the shard's LM head, an NCCL all-gather of the triples and
    the merge + commit on every rank.  On one GPU the G shard contexts run one
    after another in one stream and the exchange is a device-side stack: the
    line then reports each shard's own LM-head time per launch (what a rank
    holding that shard spends) and the merge + commit time, not a multi-GPU
    throughput.  Prints one JSON line."""
    import torch
    import synth
    from paper_2608_22646_gb300.shard import exchange_triples, vocab_slices
    G = args.vocab_shards
    if dist and world != G:
        raise SystemExit(f"--vocab-shards {G} under torchrun needs {G} ranks, not {world}")
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w, device=dev)
    hs = synth.HiddenStates(wl, W, args.generator)
    hidden = [[hs(blk, t) for t in range(wl.T)] for blk in range(wl.n_blocks)]
    cfg = cai.cai_config_default(cai.CAI_PRESET_LLADA, wl.B, wl.P, wl.H, wl.V, wl.T, wl.n_blocks)
    slices = vocab_slices(wl.V, G)
    mine = [rank] if dist else list(range(G))
    ctxs = [cai.cai_init_vocab_shard(cfg, W[v0:v0 + n].contiguous(), v0)
            for v0, n in (slices[k] for k in mine)]
    del W
    rows = cai.cai_shard_rows(ctxs[0])
    bufs = [torch.empty((rows, 4), dtype=torch.float32, device=dev) for _ in ctxs]
    stream = torch.cuda.current_stream(dev)
    prof = {"head": [[] for _ in ctxs], "commit": []}

    def step(h, timed):
        evs = []
        for k, (c, b) in enumerate(zip(ctxs, bufs)):
            if timed:
                e = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                e[0].record(stream)
            cai.cai_shard_head(c, h, b)
            if timed:
                e[1].record(stream)
                evs.append(("head", k, e))
        gathered = exchange_triples(bufs[0]) if dist else torch.stack(bufs)
        if timed:
            e = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
            e[0].record(stream)
        for c in ctxs:
            cai.cai_shard_commit(c, gathered)
        if timed:
            e[1].record(stream)
            evs.append(("commit", 0, e))
        return evs

    def generation(timed=False):
        evs = []
        for c in ctxs:
            cai.cai_reset(c)
        for blk in range(wl.n_blocks):
            if blk:
                for c in ctxs:
                    cai.cai_block_advance(c)
            evs += step(hidden[blk][0], timed)
            for t in range(1, wl.T):
                if t >= 2 and cai.cai_poll(ctxs[0], 1, 60000):
                    break
                evs += step(hidden[blk][t], timed)
        return evs

    for _ in range(args.warmup):
        generation()
    torch.cuda.synchronize()
    st0 = cai.cai_state_download(ctxs[0])
    for c in ctxs[1:]:
        assert np.array_equal(cai.cai_state_download(c)["tok"], st0["tok"]), "shards disagree"
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    local = dev.index or 0
    with Clocks(local) as clk:
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        ev0.record(stream)
        for _ in range(args.steps):
            generation()
        ev1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
    ms = ev0.elapsed_time(ev1)
    positions = int(cai.cai_state_download(ctxs[0])["m_hist"].sum()) * args.steps
    if dist:
        ms, _ = aggregate(ms, 0, dist, dev)   # every rank decodes the same positions
    evs = generation(timed=True)
    torch.cuda.synchronize()
    for kind, k, (a, b) in evs:
        (prof["head"][k] if kind == "head" else prof["commit"]).append(a.elapsed_time(b))
    n_calls = len(prof["commit"])
    head_us = [round(1e3 * sum(x) / max(1, len(x)), 2) for x in prof["head"]]
    line = {
        "metric": "masked positions decoded/s, vocabulary-parallel head (fused head + commit)",
        "value": round(positions / (ms / 1e3), 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True,
        "vocab_shards": G,
        "mode": ("one shard per GPU, NCCL all-gather of the triples" if dist else
                 "one GPU: the shards run one after another in one stream, the exchange is a "
                 "device-side stack (value = all shards' work on this GPU)"),
        "ms_per_generation": round(ms / args.steps, 4),
        "step_calls_per_generation": n_calls,
        "shard_rows": [n for _, n in slices],
        "per_shard_head_us": head_us if not dist else head_us[:1],
        "merge_commit_us_per_step": round(1e3 * sum(prof["commit"]) / max(1, n_calls), 2),
        "exchange_bytes_per_step": rows * 16 * G,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{wl.name}: B={wl.B} H={wl.H} V={wl.V} gen_len={wl.gen_len} "
                               f"block={wl.P} T={wl.T}", "hidden_generator": args.generator},
        "clocks": clk.summary(),
    }
    for c in ctxs:
        cai.cai_free(c)
    if rank == 0:
        print(json.dumps(line), flush=True)


def run_reference(args, wl):
    """The oracle on the host cores: each bench step is one denoising step of
    the trajectory (every masked row of that step), in trajectory order."""
    import torch
    import oracle
    import synth
    oracle.build()
    W = synth.lm_head_weight(wl.V, wl.H, seed=wl.seed_w, device="cpu")
    hs = synth.HiddenStates(wl, W, args.generator)
    norm = ()
    if args.final_norm:
        norm = (synth.final_norm_weight(wl.H), FINAL_NORM_EPS)
        hs = synth.PreNormHidden(hs)
    cfg = oracle.Config(B=wl.B, P=wl.P, T=wl.T, n_blocks=wl.n_blocks)
    st = oracle.State(cfg)
    Wb = oracle.bf16_bits(W)
    threads = os.cpu_count() or 1
    order = [(b, t) for b in range(wl.n_blocks) for t in range(wl.T)]
    pos = 0
    rows = 0
    dt = 0.0
    k = 0

    def one():
        nonlocal pos
        while True:
            b, t = order[pos % len(order)]
            pos += 1
            if t == 0 and b == 0:
                st.__init__(cfg)
            if np.all(st.exit_reason[:, b] != 0):
                continue
            h = oracle.bf16_bits(hs(b, t))
            t0 = time.perf_counter()
            out = oracle.step(st, Wb, h, b, t, threads, *norm)
            return out["M"], time.perf_counter() - t0

    for _ in range(args.warmup):
        one()
    for _ in range(args.steps):
        m, s = one()
        rows += m
        dt += s
        k += 1
    v = rows / dt
    line = {"impl": "reference", "metric": METRIC, "value": round(v, 3), "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(dt / k * 1e3, 3),
            "step_unit": "one bench step = one denoising step call of the trajectory (every "
                         "masked row of that step), in trajectory order",
            "ms_per_step_call": round(dt / k * 1e3, 3),
            "same_config": {"workload": True, "metric": True, "unit": True,
                            "differs": "the GPU arm's bench step is a whole generation; this "
                                       "arm times K step calls of the same trajectory (a "
                                       "bounded sample): both report masked positions "
                                       "decoded per second"},
            "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {**_workload_desc(wl, args.generator),
                       "final_norm_in_head": bool(args.final_norm)},
            "cpu_baseline": {"value": round(v, 3), "unit": UNIT, "cores": threads,
                             "kind": "oracle",
                             "sample": f"{k} denoising steps of the trajectory, {rows} masked rows"},
            "e2e": {"value": round(v, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
