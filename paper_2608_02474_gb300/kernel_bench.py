"""Run one kernel of the library at one shape, for timing and ncu captures.

    python -m paper_2608_02474_gb300.kernel_bench --kernel gemm --M 32760 --N 10240 --K 5120
    python -m paper_2608_02474_gb300.kernel_bench --kernel attention --M 6552 --L 32760 --H 40 --d 128
    python -m paper_2608_02474_gb300.kernel_bench --kernel drift --T 21 --N 1560 --D 5120
    python -m paper_2608_02474_gb300.kernel_bench --kernel merge --T 21 --N 1560 --D 5120 --K 6552
    python -m paper_2608_02474_gb300.kernel_bench --kernel step_delta --T 21 --N 1560 --D 5120
    python -m paper_2608_02474_gb300.kernel_bench --kernel block --T 21 --N 1560 --D 5120 --K 6552

Inputs are seeded random device tensors of the right shapes (values do not
change the work of these kernels).  Prints the mean time per launch over
--iters launches after --warmup launches, measured with CUDA events on the
launching stream, plus the achieved TFLOP/s or GB/s.
"""
from __future__ import annotations

import argparse
import json

import torch

from . import echocache as ec


def make_parser() -> argparse.ArgumentParser:
    ap = argparse.ArgumentParser()
    ap.add_argument("--kernel", required=True,
                    choices=["gemm", "attention", "drift", "select", "merge", "quant", "layernorm",
                             "energy", "step_delta", "ref_write", "block"])
    ap.add_argument("--M", type=int, default=6552)
    ap.add_argument("--N", type=int, default=5120)
    ap.add_argument("--K", type=int, default=5120)
    ap.add_argument("--L", type=int, default=32760)
    ap.add_argument("--H", type=int, default=40)
    ap.add_argument("--d", type=int, default=128)
    ap.add_argument("--T", type=int, default=21)
    ap.add_argument("--D", type=int, default=5120)
    ap.add_argument("--act", type=int, default=0)
    ap.add_argument("--rows", type=int, default=0, help="layernorm: gather this many rows")
    ap.add_argument("--f32", action="store_true", help="layernorm: fp32 input")
    ap.add_argument("--samples", type=int, default=80960, help="energy: audio samples")
    ap.add_argument("--F", type=int, default=13824, help="block: FFN width")
    ap.add_argument("--Lc", type=int, default=672, help="block: audio condition tokens")
    ap.add_argument("--iters", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=1)
    return ap


def main():
    a = make_parser().parse_args()

    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(0)
    rn = lambda *s: torch.randn(*s, generator=g, device=dev, dtype=torch.float32)

    if a.kernel == "gemm":
        A = rn(a.M, a.K).to(torch.bfloat16)
        W = (rn(a.N, a.K) * 0.02).to(torch.bfloat16)
        b = (rn(a.N) * 0.02).to(torch.bfloat16)
        out = torch.empty(a.M, a.N, dtype=torch.bfloat16, device=dev)
        run = lambda: ec.echo_linear(A, W, b, act=a.act, out=out)
        work, unit = 2.0 * a.M * a.N * a.K, "TFLOP/s"
    elif a.kernel == "attention":
        D = a.H * a.d
        Q = rn(a.M, D).to(torch.bfloat16)
        KV = rn(a.L, 2 * D).to(torch.bfloat16)
        out = torch.empty(a.M, D, dtype=torch.bfloat16, device=dev)
        run = lambda: ec.echo_attention(Q, KV[:, :D], KV[:, D:], a.H, a.d, out=out)
        work, unit = 4.0 * a.M * a.L * D, "TFLOP/s"
    elif a.kernel in ("drift", "select"):
        NT = a.T * a.N
        x = rn(NT, a.D).to(torch.bfloat16)
        q = torch.randint(-127, 128, (NT, a.D), generator=g, device=dev, dtype=torch.int8)
        s = torch.rand(NT, generator=g, device=dev) * 0.05
        e = torch.rand(a.T, generator=g, device=dev)
        idx = torch.empty(NT, dtype=torch.int32, device=dev)
        sc = torch.empty(NT, dtype=torch.float32, device=dev)
        run = lambda: ec.echo_select(x, q, s, e, a.T, a.N, 1, 5, idx=idx, scores=sc)
        work, unit = NT * (3.0 * a.D + 8), "GB/s"
    elif a.kernel in ("merge", "quant"):
        NT = a.T * a.N
        D = a.D
        q = torch.randint(-127, 128, (NT, D), generator=g, device=dev, dtype=torch.int8)
        s = torch.rand(NT, generator=g, device=dev) * 0.05
        perm = torch.randperm(NT, generator=g, device=dev)[:a.K]
        idx = torch.sort(perm).values.to(torch.int32)
        yact = rn(a.K, D).to(torch.bfloat16)
        if a.kernel == "quant":
            run = lambda: ec.echo_cache_quant(yact, idx, q, s)
            work = a.K * (3.0 * D + 8)
        else:
            # K = 0 block step is exactly the merge kernel plus the row map
            dims = ec.BlockDims(a.T, a.N, D, a.H, a.d, 4096, 16)
            y = torch.empty(NT, D, dtype=torch.bfloat16, device=dev)
            fake = torch.zeros(64, dtype=torch.bfloat16, device=dev)

            class _W:
                cstruct = ec.BlockWeightsC(*([fake.data_ptr()] * 15))
            ws = torch.empty(ec.echo_workspace_size(dims, 0), dtype=torch.uint8, device=dev)
            x = torch.empty(NT, D, dtype=torch.bfloat16, device=dev)
            run = lambda: ec.echo_block_step(_W, dims, x, None, 0, q, s, y=y, workspace=ws)
            work = NT * (D + 4.0) + NT * 2.0 * D + 4.0 * NT
        unit = "GB/s"
    elif a.kernel == "step_delta":
        n = a.T * a.N * a.D
        hp = rn(n).to(torch.bfloat16)
        hc = (hp.float() + 0.05 * rn(n)).to(torch.bfloat16)
        out = torch.empty(3, dtype=torch.float64, device=dev)
        ws = torch.empty(ec.echo_step_delta_workspace_size(n), dtype=torch.uint8, device=dev)
        run = lambda: ec.echo_step_delta(hp, hc, out=out, workspace=ws)
        work, unit = 4.0 * n, "GB/s"
    elif a.kernel == "ref_write":
        # reference-plus-residual cache write of K rows (scan segments of 52
        # tokens, tau 0.9) into a cache filled with rows alike along the token
        # order; the rows written are alike too (AR(1), rho 0.95)
        NT, D = a.T * a.N, a.D
        # AR(1) along the token order within each run of 52 tokens
        x = rn(NT, D)
        x = x.view(-1, 52, D) if NT % 52 == 0 else x.view(1, NT, D)
        for k in range(1, x.shape[1]):
            x[:, k] = 0.95 * x[:, k - 1] + (1 - 0.95 ** 2) ** 0.5 * x[:, k]
        full = x.reshape(NT, D).to(torch.bfloat16)
        cache = ec.DeviceCache(ec.CACHE_REF, NT, D, seg_len=52, tau=0.9, device=dev)
        cache.write(full, torch.arange(NT, dtype=torch.int32, device=dev))
        rows = torch.sort(torch.randperm(NT, generator=g, device=dev)[:a.K]).values.to(torch.int32)
        src = full[rows.long()].contiguous()
        ws = torch.empty(cache.write_workspace_size(a.K), dtype=torch.uint8, device=dev)
        run = lambda: cache.write(src, rows, workspace=ws)
        work, unit = a.K * (3.0 * D + 8), "GB/s"
    elif a.kernel == "block":
        # one cached layer step (echo_block_step) on K of T*N tokens with
        # random weights: every kernel of the block, for captures of any of them
        NT, D, K = a.T * a.N, a.D, a.K
        W = {}
        for nm in ("q", "k", "v", "o", "qc", "kc", "vc", "oc"):
            W["W" + nm] = (rn(D, D) * 0.02).to(torch.bfloat16)
            W["b" + nm] = (rn(D) * 0.02).to(torch.bfloat16)
        W["W1"], W["b1"] = (rn(a.F, D) * 0.02).to(torch.bfloat16), (rn(a.F) * 0.02).to(torch.bfloat16)
        W["W2"], W["b2"] = (rn(D, a.F) * 0.02).to(torch.bfloat16), (rn(D) * 0.02).to(torch.bfloat16)
        blk = ec.DeviceBlock.from_host(W, rn(a.Lc, D).to(torch.bfloat16), device=dev)
        del W
        dims = ec.BlockDims(a.T, a.N, D, a.H, a.d, a.F, a.Lc)
        x = rn(NT, D).to(torch.bfloat16)
        q = torch.randint(-127, 128, (NT, D), generator=g, device=dev, dtype=torch.int8)
        s = torch.rand(NT, generator=g, device=dev) * 0.05
        idx = torch.sort(torch.randperm(NT, generator=g, device=dev)[:K]).values.to(torch.int32)
        y = torch.empty(NT, D, dtype=torch.bfloat16, device=dev)
        ws = torch.empty(ec.echo_workspace_size(dims, K), dtype=torch.uint8, device=dev)
        run = lambda: ec.echo_block_step(blk, dims, x, idx, K, q, s, y=y, workspace=ws)
        work = (2.0 * NT * D * 2 * D + 4 * 2.0 * K * D * D + 4.0 * K * NT * D
                + 4.0 * K * a.Lc * D + 2 * 2.0 * K * D * a.F)
        unit = "TFLOP/s"
    elif a.kernel == "energy":
        audio = rn(a.samples)
        band = torch.empty(a.T, 8, dtype=torch.float32, device=dev)
        seg = torch.empty(a.T, dtype=torch.float32, device=dev)
        run = lambda: ec.echo_audio_energy(audio, a.T, band=band, seg=seg)
        work, unit = 4.0 * a.samples, "GB/s"
    else:  # layernorm
        NT = a.T * a.N
        x = rn(NT, a.D) if a.f32 else rn(NT, a.D).to(torch.bfloat16)
        n = a.rows if a.rows else NT
        rows = torch.sort(torch.randperm(NT, generator=g, device=dev)[:n]).values.to(torch.int32) \
            if a.rows else None
        out = torch.empty(n, a.D, dtype=torch.bfloat16, device=dev)
        run = lambda: ec.echo_layernorm(x, rows=rows, out=out)
        work, unit = n * (x.element_size() + 2.0) * a.D, "GB/s"

    for _ in range(a.warmup):
        run()
    torch.cuda.synchronize()
    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(a.iters):
        run()
    e1.record(st)
    torch.cuda.synchronize()
    assert ec.echo_get_device_error() == 0
    ms = e0.elapsed_time(e1) / a.iters
    rate = work / (ms * 1e-3) / (1e12 if unit == "TFLOP/s" else 1e9)
    print(json.dumps({"kernel": a.kernel, "ms": round(ms, 4), unit: round(rate, 1),
                      "args": vars(a)}))


if __name__ == "__main__":
    main()
