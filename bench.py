#!/usr/bin/env python
"""Throughput of the energy-guided cached DiT step on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
audio segment energy, then per layer the energy-guided selection (drift score
+ top-K) and the block on the selected latents (gather, self-attention with
K/V over all latents, cross-attention to the audio tokens, FFN, int8 cache
write, merge).  Default workload: one Wan2.2-S2V-shaped block, 21x30x52 =
32760 latent tokens, D 5120, 40 heads x 128, FFN 13824, 672 audio tokens,
refresh ratio 1/5 (6552 active tokens), synthetic speech-like audio,
random-init weights.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle on
the host cores instead: complete, unsampled cached steps of the same workload
while a time budget lasts, plus whole-run timings of the small workloads.
Multi-GPU: independent replicas (the step does not shard; no collective on
the data path); value = tokens of all ranks / max rank time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "cached DiT step latent tokens/s"
UNIT = "tokens/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="wan_block_32760")
    ap.add_argument("--ratio", default=None, help="num/den refresh ratio override")
    ap.add_argument("--profile", default="audio", help="audio profile")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--ref-budget-s", type=float, default=150.0,
                    help="--impl reference: complete oracle steps are timed while this many "
                         "seconds last (at least one step)")
    ap.add_argument("--no-full-runs", action="store_true",
                    help="--impl reference: skip the full-run timing of the small workloads")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--adaptive", default=None, metavar="R_MIN,R_MAX,ALPHA",
                    help="adaptive update rate (Sec. 3.3) instead of a fixed ratio, e.g. "
                         "0.1,0.5,0.2; the change of Eq. 1 between consecutive step outputs "
                         "and the host rule are part of every timed step")
    ap.add_argument("--cache", default="int8", choices=["int8", "bf16", "ref"],
                    help="cache form: plain int8 (default), full-precision bf16 (ablation) or "
                         "reference plus int8 residual (Sec. 3.4)")
    ap.add_argument("--tau", type=float, default=0.9, help="--cache ref: similarity threshold")
    ap.add_argument("--seg-len", type=int, default=0,
                    help="--cache ref: tokens per scan segment (default: the frame width W')")
    ap.add_argument("--select", default="energy", choices=["energy", "uniform", "random"],
                    help="token selection: energy-guided (default) or the Uniform / Random "
                         "ablations")
    ap.add_argument("--latents", default="iid", choices=["iid", "smooth"],
                    help="synthetic latents: i.i.d. (default) or spatially smooth rows "
                         "(AR(1) along each frame row, rho 0.95)")
    ap.add_argument("--reuse-kv", action="store_true",
                    help="keep every layer's K/V of all tokens on the device across steps and "
                         "recompute, at layers >= 1, only the rows whose input changed (the "
                         "outputs are bit for bit those without)")
    ap.add_argument("--graph", action="store_true",
                    help="replay each step (audio energy included) as a captured CUDA graph; "
                         "one host launch per step")
    ap.add_argument("--sweep", action="store_true",
                    help="refresh-ratio x audio-profile sweep against the uncached block "
                         "(one JSON line per point and a break-even summary)")
    return ap.parse_args()


# ---------------------------------------------------------------------------
class ClockSampler:
    """nvidia-smi clock / throttle-reason samples during the timed region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index, self.lines, self.proc = index, [], None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ln in self.lines:
            p = [x.strip() for x in ln.split(",")]
            if len(p) < 8:
                continue
            try:
                sm.append(float(p[0]))
                mx = float(p[1])
            except ValueError:
                continue
            for nm, v in zip(names, p[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
def algorithmic_work(name, m, n, k, K, xbytes=2):
    """(flops, bytes) one launch must do, from its recorded shape."""
    if name == "gemm_tcgen05":
        return 2.0 * m * n * k, None
    if name == "attention":
        return 4.0 * m * n * k, None
    if name == "drift_score":
        return None, m * n * (xbytes + 1) + 8.0 * m
    if name == "dequant_merge":
        # inactive rows: codes and scale in, bf16 out; the active rows are
        # already in y (stored by the FFN-down epilogue); the row map once
        NT, D = m, n
        return None, (NT - K) * (3.0 * D + 4) + 4.0 * NT
    if name == "merge_quant":
        # every row once: an inactive row's codes and scale in, bf16 out; an
        # active row's bf16 value and row max in, codes and scale out; the row
        # map once
        NT, D = m, n
        return None, NT * (3.0 * D + 8) + 4.0 * K
    if name == "quant_scatter":
        return None, m * n * 3 + 8.0 * m
    if name == "layernorm_gather":
        # k = input element bytes; the LN over every latent (m > K rows) also
        # writes the K active rows' copy
        return None, m * n * ((k or 2) + 2.0) + (2.0 * K * n if m > K else 0.0)
    if name == "step_delta" and m > 0:
        return None, 2.0 * m * n
    return None, None


SUSTAINED_MIN_S = 2.0   # timed regions at least this long are held to the sustained peak


def tensor_peak(peaks, timed_s):
    """(peak TFLOP/s, source): the burst peak for a timed region shorter than
    SUSTAINED_MIN_S (the GPU has not settled at its power cap), else the
    sustained one."""
    if timed_s is not None and timed_s >= SUSTAINED_MIN_S:
        return peaks["bf16_tflops_sustained"], (
            f"{peaks.get('source', 'measured')} bf16_tflops_sustained: timed region "
            f"{timed_s:.2f} s >= {SUSTAINED_MIN_S:.0f} s")
    region = "unknown" if timed_s is None else f"{timed_s:.2f} s"
    return peaks["bf16_tflops"], (
        f"{peaks.get('source', 'measured')} bf16_tflops (burst): timed region {region} "
        f"< {SUSTAINED_MIN_S:.0f} s")


def roofline(records, K, peaks, timed_s=None):
    agg = {}
    for name, m, n, k, ms in records:
        a = agg.setdefault((name, m, n, k), [0, 0.0])
        a[0] += 1
        a[1] += ms
    by_kernel = {}
    for (name, m, n, k), (cnt, ms) in agg.items():
        b = by_kernel.setdefault(name, [0, 0.0])
        b[0] += cnt
        b[1] += ms
    total = sum(v[1] for v in by_kernel.values())
    # the dominant kernel: the (kernel, launch shape) with the largest share of the
    # step among those with an algorithmic flop or byte count (the latency-bound
    # energy, top-K and row-map kernels have none)
    measurable = [kk for kk in agg if algorithmic_work(*kk, K) != (None, None)]
    key = max(measurable or agg, key=lambda kk: agg[kk][1])
    cnt, tot_ms = agg[key]
    avg_ms, (name, m, n, k) = tot_ms / cnt, key
    flops, byts = algorithmic_work(name, m, n, k, K)
    traffic = measured_traffic(name, [m, n, k])
    if flops is None and byts is None:
        out = {"bound": "latency", "kernel": name, "shape": [m, n, k], "achieved": None,
               "peak": None, "unit": None, "frac": None, "traffic": traffic,
               "launch_ms": round(avg_ms, 4)}
    elif flops is not None:
        achieved = flops / (avg_ms * 1e-3) / 1e12
        peak, source = tensor_peak(peaks, timed_s)
        out = {"bound": "tensor", "kernel": name, "shape": [m, n, k], "achieved": round(achieved, 2),
               "peak": peak, "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
               "traffic": traffic, "algorithmic_flops": flops, "launch_ms": round(avg_ms, 4),
               "peak_source": source}
        if "bf16_tflops_sustained" in peaks:   # beside it, always: the power-capped figure
            out["frac_of_sustained"] = round(achieved / peaks["bf16_tflops_sustained"], 4)
    else:
        achieved = byts / (avg_ms * 1e-3) / 1e9
        peak = peaks["hbm_gbs"]
        out = {"bound": "hbm", "kernel": name, "shape": [m, n, k], "achieved": round(achieved, 1),
               "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 4), "traffic": traffic,
               "algorithmic_bytes": byts, "launch_ms": round(avg_ms, 4),
               "peak_source": f"{peaks.get('source', 'measured')} hbm_gbs"}
    table = {}
    for (nm, m, n, k), (c, ms) in sorted(agg.items(), key=lambda kv: -kv[1][1]):
        f, b = algorithmic_work(nm, m, n, k, K)
        row = {"launches": c, "ms_per_launch": round(ms / c, 4), "share": round(ms / total, 4)}
        if f is not None:
            row["tflops"] = round(f / (ms / c * 1e-3) / 1e12, 1)
        if b is not None:
            row["gbs"] = round(b / (ms / c * 1e-3) / 1e9, 1)
        table[f"{nm}[{m}x{n}x{k}]"] = row
    return out, table


def measured_traffic(kernel, shape):
    """DRAM bytes per launch from profiles/traffic.json, only while the kernel's
    source file is unchanged since the capture (else None)."""
    import hashlib
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    e = json.load(open(p)).get(kernel)
    if not e or list(e["shape"]) != list(shape):
        return None
    src = os.path.join(ROOT, e["source"])
    if not os.path.exists(src):
        return None
    if hashlib.sha256(open(src, "rb").read()).hexdigest()[:16] != e["sha256_16"]:
        return None
    return e["bytes"]


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d["bf16_tflops_sustained"], "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


# ---------------------------------------------------------------------------
def oracle_sample(w, audio, W, cond, x1, q, s, rnum, rden, budget_s=25.0, adaptive=False,
                  form="int8", selection="energy", tau=0.9, seg_len=None):
    """Time the CPU oracle on a bounded sample of one cached step and extrapolate.

    Measured in full: audio energy, drift + top-K over all tokens (or the
    Uniform / Random selection), the merge (reconstruction of the inactive
    rows) and the cache write of the active rows in the cache form asked for.
    Sampled: K/V projection of `s_kv` rows (scaled by NT / s_kv) and the
    active-row block (Q', attention over all NT keys, cross-attention, FFN) of
    `s_a` rows (scaled by K / s_a).  The cache starts as the cache form of the
    previous step's rows q, s reconstruct to."""
    import numpy as np
    import oracle
    t = {}
    prev = oracle.cache.dequantize_rows(q, s)
    if form == "int8":
        c = oracle.refcache.Int8Cache(w.NT, w.D)
        c.q, c.s = q.copy(), s.copy()
    elif form == "bf16":
        c = oracle.refcache.FullCache(w.NT, w.D)
        c.v = prev
    else:
        c = oracle.refcache.RefCache(w.NT, w.D, w.NT, seg_len or w.Wp, tau)
        c.write(np.arange(w.NT), prev)
    t0 = time.perf_counter()
    _, e = oracle.energy.audio_energy(audio, w.T)
    t["energy"] = time.perf_counter() - t0
    e32 = e.astype(np.float32)
    t0 = time.perf_counter()
    K = oracle.select.refresh_budget(w.NT, rnum, rden)
    if selection == "uniform":
        idx = oracle.select.uniform(w.NT, K)
    elif selection == "random":
        idx = oracle.select.random_subset(np.random.default_rng(0).random(w.NT, dtype=np.float32), K)
    else:
        sc = oracle.select.scores_from(x1, c.reconstruct_f32(), e32, w.T, w.N)
        idx = oracle.select.top_k(sc, K)
    t["select"] = time.perf_counter() - t0
    s_kv = min(w.NT, 4096)
    t0 = time.perf_counter()
    oracle.block.self_kv(x1[:s_kv], W)
    t["kv_sample"] = time.perf_counter() - t0
    Kc, Vc = oracle.block.cross_kv(cond, W)
    kv_stand_in = x1.astype(np.float64)      # any [NT, D] array: only the timing is used
    s_a = min(K, 128)
    t0 = time.perf_counter()
    oracle.block.active_rows(x1, idx[:s_a], W, w.H, kv_stand_in, kv_stand_in, Kc, Vc)
    t["active_sample"] = time.perf_counter() - t0
    t0 = time.perf_counter()
    c.reconstruct_bf16()
    c.write(idx, x1[idx])
    t["merge_write"] = time.perf_counter() - t0
    per_layer = (t["select"] + t["kv_sample"] * w.NT / s_kv + t["active_sample"] * K / s_a
                 + t["merge_write"])
    step_s = t["energy"] + w.layers * per_layer
    if adaptive:
        t0 = time.perf_counter()
        oracle.schedule.step_delta(kv_stand_in, x1)   # two [NT, D] arrays: timing only
        t["step_delta"] = time.perf_counter() - t0
        step_s += t["step_delta"]
    sel = "drift+top-K over all" if selection == "energy" else f"{selection} selection of"
    sample = (f"oracle on one {w.name} cached step: energy, {sel} {w.NT} tokens, "
              f"merge and {form} cache write in full; K/V projection timed on {s_kv} of {w.NT} "
              f"rows and the active-row block on {s_a} of {K} rows, each scaled to the full "
              f"count; one layer timed, times {w.layers} layers"
              + ("; the step-level Eq. 1 change over all NT x D values in full" if adaptive else "")
              + f"; {sum(t.values()):.1f} s of CPU time")
    return step_s, sample, t


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def cpu_model():
    """The host CPU's model line from /proc/cpuinfo (or the machine type)."""
    import platform
    parts = {"0xd4f": "Neoverse-V2", "0xd40": "Neoverse-V1", "0xd0c": "Neoverse-N1"}
    try:
        for line in open("/proc/cpuinfo"):
            k = line.split(":")[0].strip().lower()
            if k in ("model name", "cpu model", "hardware"):
                return line.split(":", 1)[1].strip()
            if k == "cpu part":
                v = line.split(":", 1)[1].strip().lower()
                return f"{platform.machine()} {parts.get(v, 'part ' + v)}"
    except OSError:
        pass
    return platform.machine()


# ---------------------------------------------------------------------------
def build_inputs(w, profile, latents="iid"):
    import numpy as np
    from synth import generate as G
    audio = G.audio(w, profile)
    W = G.block_weights(w, 0)
    cond = G.cond_tokens(w, audio)
    x0 = G.latents(w) if latents == "iid" else G.latents_smooth(w)
    xs = [G.step_input(w, x0, t) for t in (1, 2)]
    return audio, W, cond, x0, xs


def workload_config(args, w, rnum, rden, K, world):
    """The `config` object of the JSON line; both arms print the same one."""
    return {"workload": w.name, "tokens": w.NT, "active_tokens": K,
            "ratio": f"{rnum}/{rden}" if not args.adaptive else "adaptive",
            "D": w.D, "heads": f"{w.H}x{w.d}",
            "ffn": w.F, "audio_tokens": w.Lc, "layers": w.layers,
            "audio": args.profile, "parallelism": f"replicas{world}",
            "cache": args.cache, "selection": args.select,
            "latents": args.latents, "graph": bool(args.graph),
            "reuse_kv": bool(getattr(args, "reuse_kv", False)),
            "l2": "inputs larger than L2 (x 335 MB, weights 702 MB per block)"}


def oracle_cache(w, form, q, s, tau=0.9, seg_len=None):
    """The oracle's cache of the given form, holding what q, s reconstruct to."""
    import numpy as np
    import oracle
    if form == "int8":
        c = oracle.refcache.Int8Cache(w.NT, w.D)
        c.q, c.s = q.copy(), s.copy()
    elif form == "bf16":
        c = oracle.refcache.FullCache(w.NT, w.D)
        c.v = oracle.cache.dequantize_rows(q, s)
    else:
        c = oracle.refcache.RefCache(w.NT, w.D, w.NT, seg_len or w.Wp, tau)
        c.write(np.arange(w.NT), oracle.cache.dequantize_rows(q, s))
    return c


def oracle_step(w, audio, Ws, cond, x, caches, budget, selection="energy", keys=None):
    """One complete cached step of the oracle, nothing sampled: the audio
    energy, then per layer the selection (energy-guided, or the Uniform /
    Random ablation), the block on the selected latents with K/V over every
    latent, the merge and the cache write.  `budget` is (ratio_num, ratio_den).
    Returns the last layer's output (bf16 values) and the new caches."""
    import numpy as np
    import oracle
    _, e = oracle.energy.audio_energy(audio, w.T)
    e32 = e.astype(np.float32)
    K = oracle.select.refresh_budget(w.NT, *budget)
    out = []
    for l, (W, c) in enumerate(zip(Ws, caches)):
        idx = None
        if selection == "uniform":
            idx = oracle.select.uniform(w.NT, K)
        elif selection == "random":
            idx = oracle.select.random_subset(keys, K)
        r = oracle.step.cached_layer_step_cache(x, c, e32, W, cond, w.T, w.N, w.H, *budget,
                                                idx=idx)
        out.append(r.cache)
        x = r.y_bf16
    return x, out


def time_full_runs(names=("tiny_256", "stack4_7800")):
    """The oracle's whole generation run (every step, every layer, step 0 full)
    of the small workloads, timed in full: {name: figures}."""
    import numpy as np
    import oracle
    from synth import ALL, generate as G
    res = {}
    for nm in names:
        w = ALL[nm]
        audio = G.audio(w)
        Ws = [G.block_weights(w, l) for l in range(w.layers)]
        cond = G.cond_tokens(w, audio)
        xs = list(G.step_inputs(w, G.latents(w), w.steps))
        t0 = time.perf_counter()
        e32 = oracle.energy.audio_energy(audio, w.T)[1].astype(np.float32)
        oracle.step.generation(xs, Ws, [cond] * w.layers, e32, w.T, w.N, w.H, w.ratio_num,
                               w.ratio_den)
        dt = time.perf_counter() - t0
        res[nm] = {"steps": w.steps, "layers": w.layers, "s_total": round(dt, 3),
                   "ms_per_step": round(1e3 * dt / w.steps, 2),
                   "tokens_per_s": round(w.NT * w.steps / dt, 2),
                   "note": "step 0 full, the others cached at the workload's ratio; "
                           "timed in full, nothing sampled"}
    return res


def run_reference(args, w, rnum, rden, rank, world):
    """The reference arm: the CPU oracle as it stands, on the host cores.

    Complete cached steps of the same workload are timed, unsampled, one after
    another while the time budget lasts (at least one); `steps` is the number
    timed.  The small workloads' whole generation runs are timed in full beside
    them, and the sampled estimate that the GPU arm's cpu_baseline uses is
    reported as a separate, extrapolated figure."""
    if rank != 0:
        return
    import numpy as np
    import oracle
    from synth import generate as G
    audio, W, cond, x0, xs = build_inputs(w, args.profile, args.latents)
    Ws = [W] + [G.block_weights(w, l) for l in range(1, w.layers)]
    q, s, _ = oracle.cache.quantize_rows(x0)
    caches = [oracle_cache(w, args.cache, q, s, args.tau, args.seg_len or None)
              for _ in range(w.layers)]
    budget = (rnum, rden)
    if args.adaptive:    # the first cached step of the adaptive rule (no change known yet)
        r_min, r_max, alpha = (float(v) for v in args.adaptive.split(","))
        budget = (oracle.schedule.adaptive_budget(1.0, 1.0, w.NT, r_min, r_max, alpha), w.NT)
    K = oracle.select.refresh_budget(w.NT, *budget)
    keys = np.random.default_rng(0).random(w.NT, dtype=np.float32)
    times = []
    t_start = time.perf_counter()
    while len(times) < args.steps:
        t0 = time.perf_counter()
        _, caches = oracle_step(w, audio, Ws, cond, xs[len(times) % 2], caches, budget,
                                args.select, keys)
        times.append(time.perf_counter() - t0)
        if time.perf_counter() - t_start + times[-1] > args.ref_budget_s:
            break
    ms = 1e3 * statistics.mean(times)
    val = w.NT / (ms * 1e-3)
    full_runs = time_full_runs() if not args.no_full_runs else None
    est_s, est_sample, _ = oracle_sample(w, audio, W, cond, xs[0], q, s, *budget,
                                         adaptive=bool(args.adaptive), form=args.cache,
                                         selection=args.select, tau=args.tau,
                                         seg_len=args.seg_len or None)
    sample = (f"{len(times)} complete cached step(s) of {w.name} ({w.layers} layer(s), "
              f"{K} of {w.NT} tokens refreshed), nothing sampled: energy, drift + top-K over "
              f"every token, K/V over every token, the block on the selected tokens, merge "
              f"and {args.cache} cache write")
    line = {"impl": "reference", "metric": METRIC, "value": round(val, 2), "unit": UNIT,
            "n_gpus": args.gpus, "steps": len(times), "warmup": 0,
            "requested": {"steps": args.steps, "warmup": args.warmup,
                          "note": "complete oracle steps are timed while the "
                                  f"{args.ref_budget_s:.0f} s budget lasts; the oracle has no "
                                  "warm-up state, so none is run"},
            "ms_per_step": round(ms, 2), "step_ms": [round(1e3 * t, 1) for t in times],
            "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(args, w, rnum, rden, K, world),
            "cpu_baseline": {"value": round(val, 2), "unit": UNIT, "cores": cpu_cores(),
                             "cpu_model": cpu_model(), "kind": "oracle", "sample": sample,
                             "extrapolated": False},
            "sampled_estimate": {"value": round(w.NT / est_s, 2), "unit": UNIT,
                                 "ms_per_step": round(est_s * 1e3, 1), "sample": est_sample,
                                 "extrapolated": True},
            "full_runs": full_runs,
            "e2e": {"value": round(val, 2), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def slowest_rank_ms(ms: float, world: int, device=None) -> float:
    """The step time of the job: the maximum over ranks (replicas run in
    lock-step between barriers, so the slowest one sets the pace)."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_replica: int, world: int, ms: float) -> float:
    """Whole-job throughput: every replica processes its own tokens."""
    return world * tokens_per_replica / (ms * 1e-3)


def copy_overlap(stack, xh, xs_d, rnum, rden, audio_d, n=3):
    """How much of a pinned host-to-device copy hides behind the step's kernels
    on this machine: 1 = fully (the copy engine runs beside the SMs), 0 = not at
    all.  Three steps alone, three copies alone, then both on two streams."""
    import torch
    dev = xs_d[0].device
    main, side = torch.cuda.current_stream(dev), torch.cuda.Stream(dev)
    xd = torch.empty_like(xs_d[0])

    def steps():
        for i in range(n):
            stack.set_audio(audio_d)
            stack.step(xs_d[i % 2], rnum, rden)

    def copies():
        with torch.cuda.stream(side):
            for _ in range(n):
                xd.copy_(xh, non_blocking=True)

    def wall(f):
        torch.cuda.synchronize(dev)
        t = time.perf_counter()
        f()
        torch.cuda.synchronize(dev)
        return time.perf_counter() - t
    t_s, t_c = wall(steps), wall(copies)
    t_b = wall(lambda: (copies(), steps()))
    return {"steps_s": round(t_s, 4), "copies_s": round(t_c, 4), "both_s": round(t_b, 4),
            "fraction": round(max(0.0, min(1.0, (t_s + t_c - t_b) / t_c)), 3) if t_c > 0 else None}


def make_stack(args, w, blocks, dev):
    """The CachedStack of the requested cache form and selection."""
    from paper_2608_02474_gb300 import echocache as ec
    from paper_2608_02474_gb300.pipeline import CachedStack
    kinds = {"int8": ec.CACHE_INT8, "bf16": ec.CACHE_BF16, "ref": ec.CACHE_REF}
    return CachedStack(w.T, w.N, w.D, w.H, w.d, w.F, w.Lc, blocks, device=dev,
                       cache_kind=kinds[args.cache], seg_len=args.seg_len or w.Wp, tau=args.tau,
                       selection=args.select, reuse_kv=bool(getattr(args, "reuse_kv", False)))


def run_sweep(args, w, blocks, x0, xs, dev, rank, world):
    """Cached step time for every (audio profile, ratio) and the uncached block."""
    import torch
    from paper_2608_02474_gb300 import echocache as ec
    from paper_2608_02474_gb300.pipeline import CachedStack
    from synth import generate as G

    profiles = w.sweep_profiles or (args.profile,)
    ratios = w.sweep_ratios or ((w.ratio_num, w.ratio_den),)
    stack = make_stack(args, w, blocks, dev)
    x0_d = torch.from_numpy(x0).to(dev, torch.bfloat16)
    xs_d = [torch.from_numpy(x).to(dev, torch.bfloat16) for x in xs]
    stream = torch.cuda.current_stream()

    def timed(fn, steps):
        for i in range(args.warmup):
            fn(i)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(steps):
            fn(i)
        e1.record(stream)
        torch.cuda.synchronize()
        assert ec.echo_get_device_error() == 0
        return e0.elapsed_time(e1) / steps

    summary = {}
    for prof in profiles:
        audio_d = torch.from_numpy(G.audio(w, prof)).to(dev)
        stack.set_audio(audio_d)
        # uncached comparator: every token refreshed (K = NT), same kernels
        full_ms = timed(lambda i: stack.step(xs_d[i % 2], 1, 1, full=True), args.steps)
        stack.step(x0_d, 1, 1, full=True)
        points = []
        for num, den in ratios:
            def one(i, num=num, den=den):
                stack.set_audio(audio_d)
                return stack.step(xs_d[i % 2], num, den)
            ms = timed(one, args.steps)
            K = (num * w.NT + den - 1) // den
            points.append((num / den, ms))
            if rank == 0:
                print(json.dumps({"sweep": w.name, "profile": prof, "ratio": f"{num}/{den}",
                                  "active_tokens": K, "ms_per_step": round(ms, 4),
                                  "tokens_per_s": round(world * w.NT / (ms * 1e-3), 1),
                                  "uncached_ms": round(full_ms, 4),
                                  "speedup_vs_uncached": round(full_ms / ms, 3)}), flush=True)
        # smallest ratio where the cached step is no faster than the uncached one
        be = None
        for (r0, m0), (r1, m1) in zip(points, points[1:]):
            if m0 < full_ms <= m1:
                be = r0 + (r1 - r0) * (full_ms - m0) / (m1 - m0)
                break
        if be is None and points and points[0][1] >= full_ms:
            be = points[0][0]
        summary[prof] = {"uncached_ms": round(full_ms, 4),
                         "break_even_ratio": None if be is None else round(be, 4)}
    if rank == 0:
        print(json.dumps({"sweep_summary": w.name, "tokens": w.NT, "profiles": summary,
                          "note": "break_even_ratio = smallest refresh ratio at which the cached "
                                  "step is no faster than the uncached block (linear "
                                  "interpolation); null = cached faster at every ratio tried"}),
              flush=True)


def main():
    args = parse()
    from synth import ALL
    w = ALL[args.workload]
    rnum, rden = (w.ratio_num, w.ratio_den)
    if args.ratio:
        rnum, rden = (int(v) for v in args.ratio.split("/"))
    args.profile = "speech" if args.profile == "audio" else args.profile

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, w, rnum, rden, rank, world)
        return

    import numpy as np
    import torch
    import torch.distributed as dist
    from paper_2608_02474_gb300 import echocache as ec
    from paper_2608_02474_gb300.pipeline import AdaptiveRate, CachedStack

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    def barrier():
        if world > 1:
            dist.barrier()

    audio, W, cond, x0, xs = build_inputs(w, args.profile, args.latents)
    from synth import generate as G
    blocks = [ec.DeviceBlock.from_host(W if l == 0 else G.block_weights(w, l), cond, device=dev)
              for l in range(w.layers)]
    if args.sweep:
        run_sweep(args, w, blocks, x0, xs, dev, rank, world)
        return
    stack = make_stack(args, w, blocks, dev)
    seg_len = args.seg_len or w.Wp
    audio_d = torch.from_numpy(audio).to(dev)
    x0_d = torch.from_numpy(x0).to(dev, torch.bfloat16)
    xs_d = [torch.from_numpy(x).to(dev, torch.bfloat16) for x in xs]
    stack.set_audio(audio_d)
    rate = None
    if args.adaptive:
        r_min, r_max, alpha = (float(v) for v in args.adaptive.split(","))
        rate = AdaptiveRate(w.NT, r_min, r_max, alpha, device=dev)
        stack.step_adaptive(x0_d, rate, full=True)   # fills every layer's cache (untimed setup)
    else:
        stack.step(x0_d, 1, 1, full=True)          # fills every layer's cache (untimed setup)
    K = w.K if (rnum, rden) == (w.ratio_num, w.ratio_den) else (rnum * w.NT + rden - 1) // rden

    def one_step(x):
        stack.set_audio(audio_d)
        if rate is not None:
            return stack.step_adaptive(x, rate)
        return stack.step(x, rnum, rden)

    eager_step = one_step
    graph_launches = None
    if args.graph:
        if rate is not None or args.select == "random" or args.reuse_kv:
            raise SystemExit("--graph takes a fixed ratio, no random selection and no --reuse-kv")
        stack.set_audio(audio_d)
        stack.step(xs_d[0], rnum, rden)             # one-time kernel set-up outside capture
        ybufs = [torch.empty_like(xs_d[0]) for _ in range(2)]
        c0 = ec.echo_launch_count()
        graphs = {xs_d[b].data_ptr(): stack.capture_step(xs_d[b], rnum, rden, out=ybufs[b],
                                                         audio=audio_d)[0] for b in range(2)}
        graph_launches = (ec.echo_launch_count() - c0) // 2   # kernels recorded per step

        def one_step(x):  # noqa: F811
            graphs[x.data_ptr()].replay()

    for i in range(args.warmup):
        one_step(xs_d[i % 2])
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0

    # ---- device-timed region: inputs resident in HBM ----
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    l0 = ec.echo_launch_count()
    ev0.record(stream)
    host_s = 0.0
    for i in range(args.steps):
        h0 = time.perf_counter()
        one_step(xs_d[i % 2])
        host_s += time.perf_counter() - h0
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = ec.echo_launch_count() - l0
    if graph_launches is not None:   # replays do not pass through the launch counter
        launches = graph_launches * args.steps
    clk = clocks.stop()
    if rate is not None:
        timed_budgets = rate.budgets[-args.steps:]
        K = round(sum(timed_budgets) / len(timed_budgets))
    ms = slowest_rank_ms(ev0.elapsed_time(ev1) / args.steps, world, dev)
    assert ec.echo_get_device_error() == 0
    value = job_tokens_per_s(w.NT, world, ms)

    # ---- per-kernel times: the same steps again with every launch bracketed by events ----
    ec.echo_profile_enable(True)
    for i in range(args.steps):   # graph replays bypass the event pairs: time eager steps
        eager_step(xs_d[i % 2])
    torch.cuda.synchronize()
    ec.echo_profile_enable(False)
    records = ec.echo_profile_read()
    peaks = load_peaks()
    roof, table = roofline(records, K, peaks, timed_s=ms * 1e-3 * args.steps)

    # ---- end to end through the public API with host buffers ----
    # every step uploads its input from pinned host memory and downloads its
    # output into pinned host memory (CachedStack.run_host overlaps those
    # copies with the neighbouring steps' compute)
    e2e = None
    if not args.no_e2e:
        xh = [torch.from_numpy(x).to(torch.bfloat16).pin_memory() for x in xs]
        yh = [torch.empty(w.NT, w.D, dtype=torch.bfloat16).pin_memory() for _ in range(2)]
        nw = max(args.warmup, 2)
        stack.run_host([xh[i % 2] for i in range(nw)], [yh[i % 2] for i in range(nw)], rnum, rden,
                       audio=audio_d, rate=rate)
        torch.cuda.synchronize()
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        h0 = time.perf_counter()
        stack.run_host([xh[i % 2] for i in range(args.steps)],
                       [yh[i % 2] for i in range(args.steps)], rnum, rden, audio=audio_d,
                       rate=rate)
        host_enqueue_ms = (time.perf_counter() - h0) * 1e3 / args.steps
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        ems = slowest_rank_ms(e0.elapsed_time(e1) / args.steps, world, dev)
        e2e = {"value": round(job_tokens_per_s(w.NT, world, ems), 2), "unit": UNIT,
               "h2d_bytes_per_step": xh[0].numel() * 2, "d2h_bytes_per_step": yh[0].numel() * 2,
               "ms_per_step": round(ems, 3),
               # host time to enqueue a step with its copies: near the step time
               # only where pinned copies block the host
               "host_ms_per_step": round(host_enqueue_ms, 3)}
        if rate is not None:   # the budgets this leg ran (the rate state carries on)
            e2e["budgets"] = rate.budgets[-args.steps:]
        else:
            e2e["copy_overlap"] = copy_overlap(stack, xh[0], xs_d, rnum, rden, audio_d)

    cache_bytes = stack.cache_bytes()
    cache_bytes_rs = stack.cache_bytes(right_sized=True)
    peak_bytes = torch.cuda.max_memory_allocated(dev)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        q, s, _ = oracle.cache.quantize_rows(x0)
        cr = (K, w.NT) if rate is not None else (rnum, rden)
        step_s, sample, _ = oracle_sample(w, audio, W, cond, xs[0], q, s, *cr,
                                          adaptive=rate is not None, form=args.cache,
                                          selection=args.select, tau=args.tau,
                                          seg_len=args.seg_len or None)
        cpu = {"value": round(w.NT / step_s, 2), "unit": UNIT, "cores": cpu_cores(),
               "cpu_model": cpu_model(),
               "kind": "oracle", "sample": sample, "ms_per_step": round(step_s * 1e3, 1),
               "extrapolated": True,
               "complete_step": "bench.py --impl reference times complete, unsampled steps"}

    if rank == 0:
        line = {"metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "bf16", "data": "synthetic",
                "config": workload_config(args, w, rnum, rden, K, world),
                "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
                "gpu_launches": launches, "kernels": table,
                "host_ms_per_step": round(1e3 * host_s / args.steps, 3)}
        if args.cache == "ref":
            live, hw = stack.caches[-1].stats()
            line["config"]["ref_cache"] = {
                "tau": args.tau, "seg_len": seg_len, "live_references": live,
                "pool_high_water": hw}
        line["peak_memory_bytes"] = peak_bytes
        line["cache_bytes"] = {"allocated": cache_bytes,
                               "right_sized": cache_bytes_rs,
                               "note": "device bytes of every layer's cache after the timed "
                                       "steps; right_sized counts a reference pool at its "
                                       "high-water mark"}
        if rate is not None:
            line["config"]["adaptive"] = {
                "r_min": rate.r_min, "r_max": rate.r_max, "alpha": rate.alpha,
                "timed_budgets": timed_budgets,
                "note": "active_tokens = mean budget of the timed steps; each step reads back "
                        "the change of the step before (one host synchronisation per step)"}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
