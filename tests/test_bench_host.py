"""Host logic of bench.py that decides what the reported line says: the
algorithmic work of each kernel, the choice of the dominant kernel and its
roofline fraction, the DRAM traffic taken from the committed captures, and the
parsing of the clock samples.  No GPU."""
import hashlib
import json
import os

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PEAKS = {"hbm_gbs": 6000.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def test_algorithmic_work_of_the_contractions_and_bandwidth_kernels():
    M, N, Kd = 6552, 5120, 5120
    assert bench.algorithmic_work("gemm_tcgen05", M, N, Kd, 0) == (2.0 * M * N * Kd, None)
    # attention records (M queries, L keys, H*d)
    assert bench.algorithmic_work("attention", 6552, 32760, 5120, 0) == (4.0 * 6552 * 32760 * 5120, None)
    NT, D, K = 32760, 5120, 6552
    # drift: bf16 x + int8 codes per element, scale and score per row
    assert bench.algorithmic_work("drift_score", NT, D, 0, K) == (None, NT * D * 3 + 8.0 * NT)
    # merge: the inactive rows (codes in, bf16 out, scale) and the row map
    assert bench.algorithmic_work("dequant_merge", NT, D, 0, K) == (
        None, (NT - K) * (3.0 * D + 4) + 4.0 * NT)
    # merge + int8 write: 3 bytes per element of every row, the scale or row
    # max and the row map per row, the active rows' scales out
    assert bench.algorithmic_work("merge_quant", NT, D, K, K) == (None, NT * (3.0 * D + 8) + 4.0 * K)
    # the all-latent layernorm also writes the K active rows' copy; a gathered
    # (K-row) layernorm of fp32 input does not
    assert bench.algorithmic_work("layernorm_gather", NT, D, 2, K) == (
        None, NT * D * 4.0 + 2.0 * K * D)
    assert bench.algorithmic_work("layernorm_gather", K, D, 4, K) == (None, K * D * 6.0)
    # latency-bound kernels have no algorithmic count
    assert bench.algorithmic_work("topk_select", NT, K, 0, K) == (None, None)
    assert bench.algorithmic_work("segment_energy_fft", 21, 21, 512, K) == (None, None)


def test_roofline_takes_the_largest_measurable_kernel():
    K = 6552
    recs = [("attention", 6552, 32760, 5120, 2.5), ("attention", 6552, 32760, 5120, 2.5),
            ("gemm_tcgen05", 32760, 10240, 5120, 1.7), ("gemm_tcgen05", 32760, 10240, 5120, 1.7),
            ("segment_energy_fft", 21, 21, 512, 9.0),      # longest, but latency-bound
            ("drift_score", 32760, 5120, 0, 0.08)]
    out, table = bench.roofline(recs, K, PEAKS, timed_s=0.13)
    assert out["kernel"] == "attention" and out["bound"] == "tensor"
    flops = 4.0 * 6552 * 32760 * 5120
    assert out["achieved"] == pytest.approx(flops / 2.5e-3 / 1e12, rel=1e-4)
    # a 0.13 s timed region is held to the burst peak
    assert out["peak"] == PEAKS["bf16_tflops"] and "burst" in out["peak_source"]
    assert out["frac"] == pytest.approx(out["achieved"] / PEAKS["bf16_tflops"], rel=1e-3)
    assert out["launch_ms"] == pytest.approx(2.5)
    assert sum(r["share"] for r in table.values()) == pytest.approx(1.0, abs=1e-3)
    assert table["attention[6552x32760x5120]"]["launches"] == 2
    assert "tflops" in table["gemm_tcgen05[32760x10240x5120]"]
    assert "gbs" in table["drift_score[32760x5120x0]"]


def test_roofline_of_a_bandwidth_bound_step_and_the_latency_fallback():
    out, _ = bench.roofline([("drift_score", 32760, 5120, 0, 0.08)], 6552, PEAKS)
    assert out["bound"] == "hbm" and out["unit"] == "GB/s"
    assert out["achieved"] == pytest.approx((32760 * 5120 * 3 + 8.0 * 32760) / 0.08e-3 / 1e9, rel=1e-4)
    out, _ = bench.roofline([("topk_select", 256, 64, 0, 0.01)], 64, PEAKS)
    assert out["bound"] == "latency" and out["frac"] is None


def test_committed_traffic_matches_the_current_sources():
    """Every DRAM-traffic entry bench.py can report belongs to the kernel source
    as it is now; a kernel changed after its capture must be captured again."""
    d = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))
    for name, e in d.items():
        if not isinstance(e, dict):
            continue
        src = os.path.join(ROOT, e["source"])
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        assert sha == e["sha256_16"], f"{name}: {e['source']} changed since its capture"
        assert os.path.exists(os.path.join(ROOT, "profiles", e["capture"]))
        assert bench.measured_traffic(name, e["shape"]) == e["bytes"]
        # another launch shape of the same kernel has no measured traffic
        assert bench.measured_traffic(name, [s + 1 for s in e["shape"]]) is None


class _DoneProc:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0


def test_clock_samples_are_parsed_into_median_and_reasons(monkeypatch):
    monkeypatch.setattr(bench.time, "sleep", lambda s: None)
    c = bench.ClockSampler(0)
    c.proc = _DoneProc()
    c.lines = [
        "1965, 2070, 900.1, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "2070, 2070, 1200.0, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active",
        "2010, 2070, 1300.5, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
        "garbage line",
        "[N/A], 2070, 1.0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    r = c.stop()
    assert r == {"sm_mhz": 2010.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    c2 = bench.ClockSampler(0)
    c2.proc = _DoneProc()
    c2.lines = ["1800, 2070, 1000, 0x8, Active, Not Active, Active, Not Active"]
    assert c2.stop()["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]
    assert bench.ClockSampler(0).stop() is None        # never started


def test_peaks_come_from_the_measured_file():
    p = bench.load_peaks()
    d = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    assert p["source"] == "measured"
    assert p["hbm_gbs"] == d["hbm_gbs"] and p["bf16_tflops_sustained"] == d["bf16_tflops_sustained"]


def test_tensor_peak_follows_the_length_of_the_timed_region():
    assert bench.tensor_peak(PEAKS, 0.13)[0] == PEAKS["bf16_tflops"]
    assert bench.tensor_peak(PEAKS, None)[0] == PEAKS["bf16_tflops"]
    assert bench.tensor_peak(PEAKS, bench.SUSTAINED_MIN_S)[0] == PEAKS["bf16_tflops_sustained"]
    out, _ = bench.roofline([("attention", 6552, 32760, 5120, 2.5)], 6552, PEAKS, timed_s=3.0)
    assert out["peak"] == PEAKS["bf16_tflops_sustained"] and "sustained" in out["peak_source"]
    # the fraction of the power-capped peak is reported beside the rule's one
    short, _ = bench.roofline([("attention", 6552, 32760, 5120, 2.5)], 6552, PEAKS, timed_s=0.13)
    assert short["peak"] == PEAKS["bf16_tflops"]
    assert short["frac_of_sustained"] == round(short["achieved"] / PEAKS["bf16_tflops_sustained"], 4)


def test_both_arms_print_the_same_config():
    import argparse
    from synth import ALL
    args = argparse.Namespace(adaptive=None, profile="speech", cache="int8", select="energy",
                              latents="iid", graph=False)
    w = ALL["wan_block_32760"]
    c = bench.workload_config(args, w, 1, 5, w.K, 1)
    assert c == bench.workload_config(args, w, 1, 5, w.K, 1)
    assert c["workload"] == "wan_block_32760" and c["active_tokens"] == 6552
    assert c["ratio"] == "1/5" and c["parallelism"] == "replicas1"


def test_reference_arm_times_complete_steps_within_its_budget(capsys):
    """The reference arm on the 256-token workload: every requested step is a
    complete oracle step, the line reports the steps it timed, the sampled
    estimate is marked extrapolated and the config equals the GPU arm's."""
    import argparse
    from synth import ALL
    args = argparse.Namespace(adaptive=None, profile="speech", cache="int8", select="energy",
                              latents="iid", graph=False, steps=2, warmup=1, gpus=1, tau=0.9,
                              seg_len=0, ref_budget_s=600.0, no_full_runs=True)
    w = ALL["tiny_256"]
    bench.run_reference(args, w, w.ratio_num, w.ratio_den, 0, 1)
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["steps"] == 2 and len(line["step_ms"]) == 2
    assert line["ms_per_step"] * line["steps"] <= 1e3 * 600
    assert line["cpu_baseline"]["extrapolated"] is False
    assert line["sampled_estimate"]["extrapolated"] is True
    assert line["config"] == bench.workload_config(args, w, 1, 4, w.K, 1)
    # a budget shorter than one step still times exactly one complete step
    args.ref_budget_s, args.steps = 0.0, 5
    bench.run_reference(args, w, w.ratio_num, w.ratio_den, 0, 1)
    assert json.loads(capsys.readouterr().out.strip().splitlines()[-1])["steps"] == 1
