"""Benchmark of the MixFP4 W4A4 linear layer on GB300.

One step = one pass of the hot path over one batch of the Llama-3-8B
attention-projection workload (X 2048x4096 bf16 Student-t activations with
outlier channels, W 4096x4096 bf16 weights): amax + MixFP4 quantization of X
(Algorithm 1), then the MixFP4 x MixFP4 GEMM against W quantized once
beforehand.  The metric is the layer's throughput in TFLOP/s (2*M*N*K per
step); the quantizer's GB/s on a 2^28-element activation (larger than L2) is
reported beside it.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (launched by torch.distributed.run) every rank runs an independent
replica on its own GPU -- the layer has no cross-GPU exchange -- and rank 0
prints ONE JSON line with the whole-job throughput (max time over ranks).
``--impl reference`` times the plain CPU oracle on bounded samples of the same
workload on the host cores.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "MixFP4 GEMM TFLOP/s + quantizer GB/s, each as % of GB300 roofline"
WORKLOAD = "attn"
QUANT_BYTES_PER_ELEM = 2.0 + 0.5 + 1.0 / 16.0   # bf16 in, nibble codes + scale bytes out


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def kernel_hash(name: str) -> str:
    src = os.path.join(ROOT, "paper_2605_31035_gb300", "csrc", name)
    return hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]


def ncu_traffic(key: str, src: str):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel source; otherwise None."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p)).get(key)
    if not d or d.get("source_sha") != kernel_hash(src):
        return None
    return d.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float | None = None):
        rows = []
        if self.path and os.path.exists(self.path):
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
                except ValueError:
                    continue
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, flags in rows for i, f in enumerate(flags) if f.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


class L2Flush:
    """Empties the 129 MB L2 between timed launches by writing a 256 MiB
    buffer (the timed kernel then starts cold; its first reads also write the
    flush's dirty lines back to HBM)."""
    NOTE = "flushed before every timed step, outside its events: 256 MiB write"

    def __init__(self, dev):
        import torch
        self.w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def __call__(self):
        self.w.zero_()


def dist_setup(n_gpus: int):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    if ws > 1:
        import torch.distributed as dist
        backend = "nccl" if os.environ.get("MIXFP4_BENCH_BACKEND", "nccl") == "nccl" else "gloo"
        dist.init_process_group(backend)
        return dist.get_rank(), ws, int(os.environ.get("LOCAL_RANK", "0"))
    return 0, 1, 0


def reduce_max(value: float, device) -> float:
    """Max of a per-rank scalar over the job (identity without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(work_per_rank: float, world: int, max_ms: float) -> float:
    """Whole-job rate of N independent replicas: the work every rank did,
    divided by the slowest rank's time (ms), per second."""
    return world * work_per_rank / (max_ms * 1e-3)


def barrier():
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        dist.barrier()


# ----------------------------------------------------------------------------- ours
def run_ours(args):
    import torch
    from paper_2605_31035_gb300 import build, ops, synth

    rank, world, local = dist_setup(args.gpus)
    build.build()
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    lin = synth.workloads()[WORKLOAD].linears[0]
    M, N, K = lin.M, lin.N, lin.K
    flops = 2.0 * M * N * K
    pk = peaks()

    x_cpu = lin.make_x()
    x = x_cpu.to(dev)
    w_q = ops.mixfp4_quantize(lin.make_w().to(dev))          # weights quantized once
    q_x = ops.empty_qtensor(M, K, dev)
    ws = torch.empty(1, dtype=torch.int32, device=dev)
    C = torch.empty(M, N, dtype=torch.float32, device=dev)
    flush = L2Flush(dev)

    def step():
        ops.mixfp4_quantize(x, out=q_x, workspace=ws)
        ops.mixfp4_gemm(q_x, w_q, out=C)

    for _ in range(args.warmup):
        flush()
        step()
    torch.cuda.synchronize(dev)

    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(local) as clk:
        for i in range(args.steps):
            flush()
            ev[i][0].record(stream)
            ops.mixfp4_quantize(x, out=q_x, workspace=ws)
            ev[i][1].record(stream)
            ops.mixfp4_gemm(q_x, w_q, out=C)
            ev[i][2].record(stream)
        torch.cuda.synchronize(dev)
    barrier()
    step_ms = [e[0].elapsed_time(e[2]) for e in ev]
    quant_ms = [e[0].elapsed_time(e[1]) for e in ev]
    gemm_ms = [e[1].elapsed_time(e[2]) for e in ev]
    total_ms = reduce_max(sum(step_ms), dev)
    ms_per_step = total_ms / args.steps
    value = job_rate(args.steps * flops, world, total_ms) / 1e12
    gemm_avg = statistics.mean(gemm_ms)
    gemm_tflops = flops / (gemm_avg * 1e-3) / 1e12
    quant_avg = statistics.mean(quant_ms)
    clocks = clk.summary()

    # Quantizer on a 2^28-element activation (512 MiB bf16 > L2): the quantize
    # kernel alone with the tensor scale given, and with the amax pass.
    xs = synth.sweep_activation(28).to(dev)
    qs = ops.empty_qtensor(xs.shape[0], xs.shape[1], dev)
    ops.mixfp4_quantize(xs, out=qs, workspace=ws)
    given = qs.tensor_scale.clone()
    qc0 = ops.mixfp4_quantize_colwise_rht(xs, workspace=ws)
    given_rht_col = qc0.tensor_scale.clone()
    del qc0

    def time_quant(fn, reps=10):
        for _ in range(3):
            fn()
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
        for e in evs:
            e[0].record(stream)
            fn()
            e[1].record(stream)
        torch.cuda.synchronize(dev)
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    given_ms = time_quant(lambda: ops.mixfp4_quantize(xs, out=qs, tensor_scale=given))
    four_six_ms = time_quant(lambda: ops.mixfp4_quantize(xs, ops.MODE_FOUR_SIX, out=qs, tensor_scale=given))
    sweep_ms = time_quant(lambda: ops.mixfp4_quantize(xs, out=qs, workspace=ws))
    ops.mixfp4_quantize_rht(xs, out=qs, workspace=ws)
    given_rht = qs.tensor_scale.clone()
    rht_given_ms = time_quant(lambda: ops.mixfp4_quantize_rht(xs, out=qs, tensor_scale=given_rht))
    rht_ms = time_quant(lambda: ops.mixfp4_quantize_rht(xs, out=qs, workspace=ws))
    # Native block-scaled FP4 variant on the same workload: the weights are
    # split once (like their quantization), the activations every call.
    nw = ops.mixfp4_split_native(w_q)
    # Share of blocks that chose E1M2 (type bit set) in the quantized X and W.
    try:
        e1m2_share = {"x": round(float((q_x.scales >> 7).float().mean().item()), 4),
                      "w": round(float((w_q.scales >> 7).float().mean().item()), 4)}
    except Exception:  # a reporting extra; never costs the bench line
        e1m2_share = None
    nx = ops.mixfp4_split_native(q_x)
    Cn = torch.empty_like(C)

    def time_flushed(fn, reps=50):
        for _ in range(3):
            fn()
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
        for e in evs:
            flush()
            e[0].record(stream)
            fn()
            e[1].record(stream)
        torch.cuda.synchronize(dev)
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    native_gemm_ms = time_flushed(lambda: ops.mixfp4_gemm_native(nx, nw, out=Cn))
    native_split_ms = time_flushed(lambda: ops.mixfp4_split_native(q_x, out=nx))
    native_layer_ms = time_flushed(lambda: (ops.mixfp4_quantize(x, out=q_x, workspace=ws),
                                            ops.mixfp4_split_native(q_x, out=nx),
                                            ops.mixfp4_gemm_native(nx, nw, out=Cn)))
    del nw, nx, Cn

    # Training-flow orientations on the same 2^28-element tensor: 16-row
    # blocks down the columns (WGRAD operand) and 16 x 16 blocks (weights),
    # each with the tensor scale given (the same bytes as the row-wise kernel).
    qc = ops.empty_qtensor(xs.shape[1], xs.shape[0], dev)
    colwise_ms = time_quant(lambda: ops.mixfp4_quantize_colwise(xs, out=qc, tensor_scale=given))
    del qc
    q2d_ms = time_quant(lambda: ops.mixfp4_quantize_2d(xs, out=qs, tensor_scale=given))
    qt = ops.QTensor(torch.empty(xs.shape[1], xs.shape[0] // 2, dtype=torch.uint8, device=dev),
                     torch.empty(xs.shape[1], xs.shape[0] // 16, dtype=torch.uint8, device=dev), qs.tensor_scale)
    transpose_ms = time_quant(lambda: ops.mixfp4_transpose_2d(qs, out=qt))
    del qt
    sr_ms = time_quant(lambda: ops.mixfp4_quantize_sr(xs, 1234, 0, out=qs, tensor_scale=given))
    qc = ops.empty_qtensor(xs.shape[1], xs.shape[0], dev)
    crht_ms = time_quant(lambda: ops.mixfp4_quantize_colwise_rht(xs, out=qc, tensor_scale=given_rht_col))
    del qc
    # Candidate-set / block-size ablation (quantize-dequantize, bf16 out, the
    # per-block choice written), tensor scale given.
    fq_out = torch.empty(xs.shape, dtype=torch.bfloat16, device=dev)
    fq_ch = torch.empty(xs.shape[0], xs.shape[1] // 8, dtype=torch.uint8, device=dev)
    ablation = {}
    for name, mask, g in FQ_SETS:
        chv = fq_ch.view(-1)[: xs.shape[0] * (xs.shape[1] // g)].view(xs.shape[0], xs.shape[1] // g)
        ms_ = time_quant(lambda: ops.mixfp4_fake_quantize(xs, mask, g, torch.bfloat16, tensor_scale=given,
                                                          out=fq_out, choice=chv))
        gbs = xs.numel() * (4.0 + 1.0 / g) / (ms_ * 1e-3) / 1e9
        ablation[f"{name}_g{g}"] = {"ms": round(ms_, 4), "alg_gbs": round(gbs, 1),
                                    "frac_of_hbm": round(gbs / pk["hbm_gbs"], 4)}
    del fq_out, fq_ch

    given_gbs = xs.numel() * QUANT_BYTES_PER_ELEM / (given_ms * 1e-3) / 1e9
    sweep_alg_gbs = xs.numel() * QUANT_BYTES_PER_ELEM / (sweep_ms * 1e-3) / 1e9
    sweep_read_gbs = xs.numel() * (QUANT_BYTES_PER_ELEM + 2.0) / (sweep_ms * 1e-3) / 1e9
    xs_numel = xs.numel()
    del xs, qs

    # End to end through the public API with host buffers: every step copies
    # its X in from pinned host memory and its C out to pinned host memory.
    # Two buffer sets and three streams (copy in, compute, copy out) let step
    # i+1's copy-in and step i-1's copy-out overlap step i's kernels; events
    # keep each buffer's uses in order.
    x_host = x_cpu.pin_memory()
    c_host = [torch.empty(M, N, dtype=torch.float32).pin_memory() for _ in range(2)]
    xd = [torch.empty_like(x) for _ in range(2)]
    qd = [ops.empty_qtensor(M, K, dev) for _ in range(2)]
    wsd = [torch.empty(1, dtype=torch.int32, device=dev) for _ in range(2)]
    Cd = [torch.empty(M, N, dtype=torch.float32, device=dev) for _ in range(2)]
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_comp = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]

    def e2e_step(i):
        j = i & 1
        with torch.cuda.stream(s_in):
            if i >= 2:
                s_in.wait_event(ev_comp[j])       # step i-2 has finished reading xd[j]
            xd[j].copy_(x_host, non_blocking=True)
            ev_in[j].record(s_in)
        stream.wait_event(ev_in[j])
        if i >= 2:
            stream.wait_event(ev_out[j])          # step i-2's C has been copied out
        ops.mixfp4_quantize(xd[j], out=qd[j], workspace=wsd[j], stream=stream)
        ops.mixfp4_gemm(qd[j], w_q, out=Cd[j], stream=stream)
        ev_comp[j].record(stream)
        with torch.cuda.stream(s_out):
            s_out.wait_event(ev_comp[j])
            c_host[j].copy_(Cd[j], non_blocking=True)
            ev_out[j].record(s_out)

    for i in range(4):
        e2e_step(i)
    torch.cuda.synchronize(dev)
    e2e_steps = max(10, min(args.steps, 200))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    e0.record(s_in)
    stream.wait_event(e0)
    for i in range(e2e_steps):
        e2e_step(i)
    s_in.wait_stream(s_out)
    s_in.wait_stream(stream)
    e1.record(s_in)
    torch.cuda.synchronize(dev)
    e2e_ms = reduce_max(e0.elapsed_time(e1), dev)
    e2e_value = job_rate(e2e_steps * flops, world, e2e_ms) / 1e12

    configs = None if args.no_configs else config_gemms(dev, flush, stream, pk["bf16_tflops"])
    sweep = None if args.no_sweep else quantizer_sweep(dev, flush, stream, pk["hbm_gbs"])

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(lin, x_cpu, budget_s=args.cpu_budget)

    peak_t = pk["bf16_tflops"]
    traffic = ncu_traffic(f"gemm_{WORKLOAD}", "gemm.cu")
    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": f"Llama-3-8B attention projection: X {M}x{K} . W {N}x{K} (MixFP4 W4A4)",
                   "M": M, "N": N, "K": K, "mode": "MixFP4", "weights": "pre-quantized once",
                   "l2": L2Flush.NOTE,
                   "parallelism": f"replicas x{world}"},
        "roofline": {"bound": "tensor", "kernel": "mixfp4_gemm_kernel",
                     "achieved": round(gemm_tflops, 2), "peak": peak_t, "unit": "TFLOP/s",
                     "frac": round(gemm_tflops / peak_t, 4),
                     "peak_kind": f"bf16 dense burst, {pk['source']} (MEASURED_PEAKS.json)",
                     "traffic": traffic},
        "kernels": {
            "gemm_ms": round(gemm_avg, 5), "gemm_tflops": round(gemm_tflops, 2),
            "e1m2_block_share": e1m2_share,
            "quantize_with_amax_ms": round(quant_avg, 5),
            "quantize_with_amax_gbs_alg": round(M * K * QUANT_BYTES_PER_ELEM / (quant_avg * 1e-3) / 1e9, 1),
            "quantizer_2^28": {
                "quantize_kernel_given_scale": {"ms": round(given_ms, 4), "alg_gbs": round(given_gbs, 1),
                                                "frac_of_hbm": round(given_gbs / pk["hbm_gbs"], 4),
                                                "frac_of_hbm_spec_7900": round(given_gbs / 7900.0, 4)},
                "with_amax_pass": {"ms": round(sweep_ms, 4), "alg_gbs": round(sweep_alg_gbs, 1),
                                   "alg_frac_of_hbm": round(sweep_alg_gbs / pk["hbm_gbs"], 4),
                                   "bytes_incl_amax_read_gbs": round(sweep_read_gbs, 1)},
                "four_over_six_mode_given_scale": {
                    "ms": round(four_six_ms, 4),
                    "alg_gbs": round(xs_numel * QUANT_BYTES_PER_ELEM / (four_six_ms * 1e-3) / 1e9, 1)},
                "alg_bytes_per_element": QUANT_BYTES_PER_ELEM, "hbm_peak_gbs": pk["hbm_gbs"]},
            "native_fp4_variant": {
                "gemm_native_ms": round(native_gemm_ms, 5),
                "gemm_native_tflops": round(flops / (native_gemm_ms * 1e-3) / 1e12, 2),
                "split_x_ms": round(native_split_ms, 5),
                "layer_ms_quantize_split_gemm": round(native_layer_ms, 5),
                "layer_tflops": round(flops / (native_layer_ms * 1e-3) / 1e12, 2),
                "note": "E1M2 blocks split into E2M1 main + residual, kind::mxf4nvf4 products; weights split once"},
            "training_orientations_2^28": {
                "colwise_given_scale": {"ms": round(colwise_ms, 4),
                                        "alg_gbs": round(xs_numel * QUANT_BYTES_PER_ELEM / (colwise_ms * 1e-3) / 1e9, 1)},
                "2d_blocks_given_scale": {"ms": round(q2d_ms, 4),
                                          "alg_gbs": round(xs_numel * QUANT_BYTES_PER_ELEM / (q2d_ms * 1e-3) / 1e9, 1)},
                "colwise_rotated_given_scale": {
                    "ms": round(crht_ms, 4), "alg_gbs": round(xs_numel * QUANT_BYTES_PER_ELEM / (crht_ms * 1e-3) / 1e9, 1)},
                "stochastic_rounding_given_scale": {
                    "ms": round(sr_ms, 4), "alg_gbs": round(xs_numel * QUANT_BYTES_PER_ELEM / (sr_ms * 1e-3) / 1e9, 1)},
                "transpose_2d": {"ms": round(transpose_ms, 4),
                                 "alg_gbs": round(xs_numel * TRANSPOSE_BYTES_PER_ELEM / (transpose_ms * 1e-3) / 1e9, 1),
                                 "alg_bytes_per_element": TRANSPOSE_BYTES_PER_ELEM}},
            "candidate_ablation_2^28": {
                **ablation,
                "alg_bytes_per_element": "2 (bf16 in) + 2 (bf16 out) + 1/g (choice)",
                "note": "quantize-dequantize under a candidate set (E2M1(6), E1M2, E2M1(4), E3M0) and block size g"},
            "rht_quantizer_2^28": {
                "fused_rotation_quantize_given_scale": {
                    "ms": round(rht_given_ms, 4),
                    "alg_gbs": round(xs_numel * QUANT_BYTES_PER_ELEM / (rht_given_ms * 1e-3) / 1e9, 1)},
                "with_amax_pass": {
                    "ms": round(rht_ms, 4),
                    "alg_gbs": round(xs_numel * QUANT_BYTES_PER_ELEM / (rht_ms * 1e-3) / 1e9, 1)}}},
        "configs_gemm": configs,
        "quantizer_sweep": sweep,
        "clocks": clocks,
        "e2e": {"value": round(e2e_value, 2), "unit": "TFLOP/s",
                "h2d_bytes_per_step": x_host.numel() * 2, "d2h_bytes_per_step": c_host[0].numel() * 4,
                "steps": e2e_steps, "pipelining": "copy-in, compute, copy-out streams, two buffer sets"},
        "gpu_launches": 3 * args.steps,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(out), flush=True)


# --------------------------------------------------------------- quantizer sweep
def gpu_t3(dev, rows: int, K: int, seed: int, outliers: bool = True):
    """Student-t(3) x 0.5 activations with floor(0.01 K) x50 outlier channels,
    drawn on the GPU from a seeded generator (the synth.py distribution)."""
    import math
    import torch
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    out = torch.empty(rows, K, dtype=torch.bfloat16, device=dev)
    step = max(1, (1 << 25) // K)
    gc = torch.Generator(device="cpu")
    gc.manual_seed(seed + 1)
    ch = torch.randperm(K, generator=gc)[:int(math.floor(0.01 * K))].to(dev)
    for r0 in range(0, rows, step):
        r1 = min(rows, r0 + step)
        z = torch.randn(4, r1 - r0, K, device=dev, generator=g)
        v = z[0] / torch.sqrt((z[1] * z[1] + z[2] * z[2] + z[3] * z[3]) / 3.0) * 0.5
        if outliers:
            v[:, ch] *= 50.0
        out[r0:r1] = v.to(torch.bfloat16)
    return out


def quant_rates(x, flush, stream, hbm_gbs, reps=10):
    """Quantizer rates on x: MixFP4 and E2M1-only (NVFP4) modes, the quantize
    kernel alone (tensor scale given) and with the amax pass; L2 flushed
    before every launch.  GB/s counts the algorithmic 2.5625 B/element."""
    import torch
    from paper_2605_31035_gb300 import ops
    dev = x.device
    q = ops.empty_qtensor(x.shape[0], x.shape[1], dev)
    ws = torch.empty(1, dtype=torch.int32, device=dev)
    ops.mixfp4_quantize(x, out=q, workspace=ws)
    given = q.tensor_scale.clone()

    def timed(fn):
        for _ in range(3):
            fn()
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
        for e in evs:
            flush()
            e[0].record(stream)
            fn()
            e[1].record(stream)
        torch.cuda.synchronize(dev)
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    n = x.numel()
    rec = {"elements": n}
    for mname, mode in (("mixfp4", ops.MODE_MIX), ("e2m1_only", ops.MODE_E2M1_ONLY)):
        for sname, fn in (("given_scale", lambda: ops.mixfp4_quantize(x, mode, out=q, tensor_scale=given)),
                          ("with_amax", lambda: ops.mixfp4_quantize(x, mode, out=q, workspace=ws))):
            ms = timed(fn)
            gbs = n * QUANT_BYTES_PER_ELEM / (ms * 1e-3) / 1e9
            rec[f"{mname}_{sname}"] = {"us": round(ms * 1e3, 2), "alg_gbs": round(gbs, 1),
                                       "frac_of_hbm": round(gbs / hbm_gbs, 4)}
    return rec


def quantizer_sweep(dev, flush, stream, hbm_gbs, k_min=20, k_max=30):
    """The quantizer-only sweep: the attention activation distribution as
    [2^k / 4096, 4096] for k = k_min..k_max."""
    import torch
    out = {}
    for k in range(k_min, k_max + 1):
        x = gpu_t3(dev, (1 << k) // 4096, 4096, 5000 + k)
        out[f"2^{k}"] = quant_rates(x, flush, stream, hbm_gbs, reps=10 if k >= 26 else 20)
        del x
        torch.cuda.empty_cache()
    return out


# ------------------------------------------------------ the other configs' GEMMs
def config_gemms(dev, flush, stream, peak_t):
    """GEMM time of the other LLM-shaped configs (the MLP, decode-shaped and
    Hadamard-rotated linears) on both GEMM paths.  Inputs are drawn on the GPU
    from a seeded generator with the same distributions as synth.py (Student-t
    activations with 1 % outlier channels x 50, normal weights with lognormal
    row scales; the Hadamard case rotates 128-chunks of both by the normalised
    Sylvester matrix); weights and activations are quantized once, since these
    lines time the GEMM kernels alone (L2 flushed before each launch)."""
    import math
    import torch
    from paper_2605_31035_gb300 import ops

    g = torch.Generator(device=dev)

    def t3(rows, K, seed, outliers=True):
        g.manual_seed(seed)
        out = torch.empty(rows, K, dtype=torch.bfloat16, device=dev)
        step = max(1, (1 << 25) // K)
        for r0 in range(0, rows, step):
            r1 = min(rows, r0 + step)
            z = torch.randn(4, r1 - r0, K, device=dev, generator=g)
            v = z[0] / torch.sqrt((z[1] * z[1] + z[2] * z[2] + z[3] * z[3]) / 3.0) * 0.5
            if outliers:
                gc = torch.Generator(device="cpu")
                gc.manual_seed(seed + 1)
                ch = torch.randperm(K, generator=gc)[:int(math.floor(0.01 * K))].to(dev)
                v[:, ch] *= 50.0
            out[r0:r1] = v.to(torch.bfloat16)
        return out

    def normal(N, K, seed, std, row_sigma, outliers=False):
        g.manual_seed(seed)
        w = torch.randn(N, K, device=dev, generator=g) * std
        if row_sigma:
            w *= torch.exp(torch.randn(N, 1, device=dev, generator=g) * row_sigma)
        if outliers:
            gc = torch.Generator(device="cpu")
            gc.manual_seed(seed + 1)
            w[:, torch.randperm(K, generator=gc)[:int(math.floor(0.01 * K))].to(dev)] *= 50.0
        return w.to(torch.bfloat16)

    def hadamard(x):
        h = torch.ones(1, 1, dtype=torch.float32, device=dev)
        while h.shape[0] < 128:
            h = torch.cat([torch.cat([h, h], 1), torch.cat([h, -h], 1)], 0)
        h = h / math.sqrt(128.0)
        rows, K = x.shape
        return (x.float().reshape(rows, K // 128, 128) @ h.T).reshape(rows, K).to(torch.bfloat16)

    def timed(fn, reps=20):
        for _ in range(3):
            fn()
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
        for e in evs:
            flush()
            e[0].record(stream)
            fn()
            e[1].record(stream)
        torch.cuda.synchronize(dev)
        return statistics.median(a.elapsed_time(b) for a, b in evs)

    cases = [("mlp_gate_up", 4096, 14336, 4096, lambda: t3(4096, 4096, 11), lambda: normal(14336, 4096, 12, 0.02, 0.5)),
             ("mlp_down", 4096, 4096, 14336, lambda: t3(4096, 14336, 13), lambda: normal(4096, 14336, 14, 0.02, 0.5)),
             ("decode", 16, 28672, 8192, lambda: t3(16, 8192, 15), lambda: normal(28672, 8192, 16, 0.015, None)),
             ("hadamard_8192", 8192, 8192, 8192, lambda: hadamard(t3(8192, 8192, 17)),
              lambda: hadamard(normal(8192, 8192, 18, 0.02, None, outliers=True)))]
    out = {}
    hbm = peaks()["hbm_gbs"]
    for name, M, N, K, mx, mw in cases:
        xin, win = mx(), mw()
        quant = None
        if name == "mlp_down":        # the MLP's X' (4096 x 14336), quantized online every call
            quant = {"x": quant_rates(xin, flush, stream, hbm)}
        elif name == "hadamard_8192":  # the rotated 8192 x 8192 X and W
            quant = {"x": quant_rates(xin, flush, stream, hbm), "w": quant_rates(win, flush, stream, hbm)}
        qx, qw = ops.mixfp4_quantize(xin), ops.mixfp4_quantize(win)
        del xin, win
        C = torch.empty(M, N, dtype=torch.float32, device=dev)
        fl = 2.0 * M * N * K
        ms = timed(lambda: ops.mixfp4_gemm(qx, qw, out=C))
        rec = {"M": M, "N": N, "K": K, "gemm_ms": round(ms, 4), "tflops": round(fl / (ms * 1e-3) / 1e12, 1),
               "frac_of_bf16_peak": round(fl / (ms * 1e-3) / 1e12 / peak_t, 4)}
        if M <= 64:
            byts = N * K * (0.5 + 1.0 / 16) + M * K * (0.5 + 1.0 / 16) + M * N * 4
            rec["gbs"] = round(byts / (ms * 1e-3) / 1e9, 1)
            rec["hbm_bytes_per_launch"] = int(byts)
            ms_n = timed(lambda: ops.mixfp4_gemm_native_fewrows(qx, qw, out=C))
            rec["native_fewrows_ms"] = round(ms_n, 4)
            rec["native_fewrows_gbs"] = round(byts / (ms_n * 1e-3) / 1e9, 1)
            rec["native_fewrows_frac_of_hbm"] = round(byts / (ms_n * 1e-3) / 1e9 / peaks()["hbm_gbs"], 4)
        else:
            nx, nw = ops.mixfp4_split_native(qx), ops.mixfp4_split_native(qw)
            ms_n = timed(lambda: ops.mixfp4_gemm_native(nx, nw, out=C))
            rec["native_ms"] = round(ms_n, 4)
            rec["native_tflops"] = round(fl / (ms_n * 1e-3) / 1e12, 1)
            del nx, nw
        if quant is not None:
            rec["quantizer"] = quant
        out[name] = rec
        del qx, qw, C
        torch.cuda.empty_cache()
    return out


# ------------------------------------------------------------------ CPU oracle legs
class OracleLayer:
    """The hot path on the CPU oracle: Algorithm 1 on sampled rows of X (with
    the full tensor's s32) and the float64 GEMM against sampled rows of W,
    which are quantized once up front like the GPU path's weights."""

    def __init__(self, lin, x_cpu, w_cpu, max_w_rows: int):
        import numpy as np
        import oracle
        from paper_2605_31035_gb300 import synth
        self.lin = lin
        self.x_bits = synth.bf16_bits(x_cpu)
        self.s32 = float(np.float32(np.float32(float(x_cpu.abs().max().float())) / np.float32(2688.0)))
        ws32 = float(np.float32(np.float32(float(w_cpu.abs().max().float())) / np.float32(2688.0)))
        self.wq = oracle.quantize(synth.bf16_bits(w_cpu[:max_w_rows]), s32=ws32)

    def run(self, n_rows_x: int, n_rows_w: int, row0: int = 0):
        """Returns (seconds, flops) of one sampled pass."""
        import oracle
        wq = (self.wq[0][:n_rows_w], self.wq[1][:n_rows_w], self.wq[2])
        xs = self.x_bits[row0:row0 + n_rows_x]
        t0 = time.perf_counter()
        xq = oracle.quantize(xs, s32=self.s32)
        oracle.gemm_f64(xq, wq)
        return time.perf_counter() - t0, 2.0 * n_rows_x * n_rows_w * self.lin.K


def _calibrated_rows(layer: OracleLayer, n_rows_x: int, budget_s: float, cap: int) -> int:
    secs, _ = layer.run(1, 16)
    return max(8, min(cap, int(16 * budget_s / (max(secs, 1e-4) * n_rows_x))))


def host_cpu(cpuinfo: str = "/proc/cpuinfo") -> dict:
    """The host the oracle runs on: logical CPUs and the CPU model (the model
    name where the kernel reports one, else the Arm implementer / part codes)."""
    model = platform.processor() or platform.machine()
    fields = {}
    try:
        for line in open(cpuinfo):
            if ":" in line:
                key, val = line.split(":", 1)
                fields.setdefault(key.strip().lower(), val.strip())
    except OSError:
        pass
    if fields.get("model name"):
        model = fields["model name"]
    elif fields.get("cpu part"):
        model = f"implementer {fields.get('cpu implementer', '?')} part {fields['cpu part']}"
    return {"nproc": os.cpu_count(), "cpu": model, "arch": platform.machine()}


def _oracle_job(job):
    """One oracle task in a worker process (spawned: it shares nothing with
    the CUDA context of the bench process).  Returns its seconds."""
    kind, x_bits, s32, wq = job
    import oracle
    t0 = time.perf_counter()
    xq = oracle.quantize(x_bits, s32=s32)
    if kind == "layer":
        oracle.gemm_f64(xq, wq)
    return time.perf_counter() - t0


def oracle_all_cores(kind: str, x_bits, s32: float, wq, nproc: int, repeat: int = 1):
    """Rows of x_bits split over nproc spawned processes (the oracle itself
    is serial C), each part processed `repeat` times; returns (wall seconds,
    processes)."""
    import multiprocessing as mp
    import numpy as np
    parts = [p for p in np.array_split(x_bits, nproc) if len(p)]
    with mp.get_context("spawn").Pool(len(parts)) as pool:
        pool.map(_oracle_job, [("quantize", parts[0][:1], s32, None)] * len(parts))  # workers up and warm
        t0 = time.perf_counter()
        pool.map(_oracle_job, [(kind, p, s32, wq) for p in parts for _ in range(repeat)])
        return time.perf_counter() - t0, len(parts)


def cpu_baseline(lin, x_cpu, budget_s: float = 15.0):
    """The oracle on the host cores: the layer (Algorithm 1 on rows of X + the
    float64 GEMM against pre-quantized rows of W) single-threaded and on all
    cores (rows split over processes), and Algorithm 1 alone (elements/s)."""
    cap = 2048
    layer = OracleLayer(lin, x_cpu, lin.make_w()[:cap], cap)
    secs, _ = layer.run(1, 64)
    per_row = secs / 64.0                      # one X row against one W row
    n_w = cap
    n_x = max(4, min(512, int(budget_s / max(per_row * n_w, 1e-9))))
    secs, flops = layer.run(n_x, n_w)
    nproc = os.cpu_count() or 1
    out = {"value": flops / secs / 1e12, "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
           "sample": f"Algorithm 1 on {n_x} rows of X + float64 GEMM vs {n_w} pre-quantized rows of W "
                     f"(K={lin.K}), {secs:.1f} s single-threaded",
           "host": host_cpu()}
    wq = (layer.wq[0][:n_w], layer.wq[1][:n_w], layer.wq[2])
    try:
        n_all = max(nproc, min(lin.M, n_x * nproc))
        wall, used = oracle_all_cores("layer", layer.x_bits[:n_all], layer.s32, wq, nproc)
        out["all_cores"] = {"value": 2.0 * n_all * n_w * lin.K / wall / 1e12, "unit": "TFLOP/s", "cores": used,
                            "sample": f"{n_all} rows of X vs {n_w} rows of W split over {used} processes, "
                                      f"{wall:.1f} s"}
        rows_q = min(lin.M, 256)
        t0 = time.perf_counter()
        import oracle
        oracle.quantize(layer.x_bits[:rows_q], s32=layer.s32)
        tq = time.perf_counter() - t0
        n_q = rows_q * lin.K
        rep = max(1, int(3.0 * (n_q / tq) * nproc / (lin.M * lin.K)))   # about 3 s on all cores
        wall_q, used_q = oracle_all_cores("quantize", layer.x_bits, layer.s32, None, nproc, rep)
        out["quantizer"] = {
            "unit": "elements/s", "one_core": n_q / tq,
            "all_cores": rep * lin.M * lin.K / wall_q, "cores": used_q,
            "sample": f"Algorithm 1 on {rows_q} rows (one core, {tq:.1f} s) and on all {lin.M} rows of X "
                      f"{rep} times, split over {used_q} processes ({wall_q:.1f} s)"}
    except Exception as e:  # a reporting extra; never costs the bench line
        out["all_cores_error"] = repr(e)
    return out


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2605_31035_gb300 import synth
    lin = synth.workloads()[WORKLOAD].linears[0]
    x_cpu = lin.make_x()
    cap = 1024
    layer = OracleLayer(lin, x_cpu, lin.make_w()[:cap], cap)
    per_step_budget = max(0.01, min(1.0, 150.0 / max(1, args.steps + args.warmup)))
    n_w = _calibrated_rows(layer, 1, per_step_budget, cap)
    for i in range(args.warmup):
        layer.run(1, n_w, row0=i % lin.M)
    tot, fl = 0.0, 0.0
    for i in range(args.steps):
        s, f = layer.run(1, n_w, row0=i % lin.M)
        tot += s
        fl += f
    value = fl / tot / 1e12
    out = {"metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": int(os.environ.get("WORLD_SIZE", "1")),
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": tot / args.steps * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": {"workload": f"Llama-3-8B attention projection: X {lin.M}x{lin.K} . W {lin.N}x{lin.K} (MixFP4 W4A4)",
                      "M": lin.M, "N": lin.N, "K": lin.K, "mode": "MixFP4"},
           "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": 1, "kind": "oracle",
                            "sample": f"per step: Algorithm 1 on 1 row of X + float64 GEMM vs {n_w} "
                                      f"pre-quantized rows of W (K={lin.K}), single-threaded",
                            "host": host_cpu()},
           "gpu_launches": 0,
           "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# 2D transpose: codes in and out (0.5 + 0.5), one scale byte read per 16 x 16
# tile (the tile's rows repeat it) and one written per 16 elements of each
# output row.
TRANSPOSE_BYTES_PER_ELEM = 0.5 + 0.5 + 1.0 / 256 + 1.0 / 16
# (name, candidate mask, block size) of the ablation lines.
FQ_SETS = [("mixfp4", 1 | 2, 16), ("four_over_six", 1 | 4, 16), ("e2_e1_e3", 1 | 2 | 8, 16),
           ("all_four", 15, 16), ("e2_e1_e3", 1 | 2 | 8, 64), ("all_four", 15, 8)]


def run_kernel_only(args):
    """One kernel on one workload, for profilers: `--warmup` untimed launches,
    then `--steps` launches, then exit.  Prints the CUDA-event time per launch."""
    import torch
    from paper_2605_31035_gb300 import build, ops, synth
    build.build()
    dev = torch.device("cuda:0")
    if args.workload.startswith("sweep"):
        x = synth.sweep_activation(int(args.workload[5:])).to(dev)
        w = None
    else:
        lin = synth.workloads()[args.workload].linears[0]
        x = lin.make_x().to(dev)
        w = lin.make_w().to(dev)
    ws = torch.empty(1, dtype=torch.int32, device=dev)
    qx = ops.mixfp4_quantize(x, workspace=ws)
    if args.kernel == "gemm":
        qw = ops.mixfp4_quantize(w, workspace=ws)
        C = torch.empty(x.shape[0], w.shape[0], dtype=torch.float32, device=dev)
        fn = lambda: ops.mixfp4_gemm(qx, qw, out=C)
        work = 2.0 * x.shape[0] * w.shape[0] * x.shape[1]
    elif args.kernel == "gemm_native":
        nx = ops.mixfp4_split_native(qx)
        nw = ops.mixfp4_split_native(ops.mixfp4_quantize(w, workspace=ws))
        C = torch.empty(x.shape[0], w.shape[0], dtype=torch.float32, device=dev)
        fn = lambda: ops.mixfp4_gemm_native(nx, nw, out=C)
        work = 2.0 * x.shape[0] * w.shape[0] * x.shape[1]
    elif args.kernel == "gemm_native_fewrows":
        qw = ops.mixfp4_quantize(w, workspace=ws)
        C = torch.empty(x.shape[0], w.shape[0], dtype=torch.float32, device=dev)
        fn = lambda: ops.mixfp4_gemm_native_fewrows(qx, qw, out=C)
        work = 2.0 * x.shape[0] * w.shape[0] * x.shape[1]
    elif args.kernel == "split_native":
        fn = lambda: ops.mixfp4_split_native(qx)
        work = x.numel() * (0.5 + 1.0 / 16 + 1.0 + 1.0 / 16)
    elif args.kernel == "quantize":
        fn = lambda: ops.mixfp4_quantize(x, out=qx, workspace=ws)
        work = x.numel() * QUANT_BYTES_PER_ELEM
    elif args.kernel == "quantize_colwise":
        qc = ops.empty_qtensor(x.shape[1], x.shape[0], dev)
        fn = lambda: ops.mixfp4_quantize_colwise(x, out=qc, workspace=ws)
        work = x.numel() * QUANT_BYTES_PER_ELEM
    elif args.kernel == "quantize_2d":
        fn = lambda: ops.mixfp4_quantize_2d(x, out=qx, workspace=ws)
        work = x.numel() * QUANT_BYTES_PER_ELEM
    elif args.kernel == "transpose_2d":
        q2 = ops.mixfp4_quantize_2d(x, workspace=ws)
        fn = lambda: ops.mixfp4_transpose_2d(q2)
        work = x.numel() * TRANSPOSE_BYTES_PER_ELEM
    elif args.kernel == "quantize_colwise_rht":
        qc = ops.mixfp4_quantize_colwise_rht(x, workspace=ws)   # its s32, then the quantize pass alone
        ts = qc.tensor_scale.clone()
        fn = lambda: ops.mixfp4_quantize_colwise_rht(x, out=qc, tensor_scale=ts)
        work = x.numel() * QUANT_BYTES_PER_ELEM
    elif args.kernel == "quantize_sr":
        fn = lambda: ops.mixfp4_quantize_sr(x, 1234, 0, out=qx, workspace=ws)
        work = x.numel() * QUANT_BYTES_PER_ELEM
    elif args.kernel == "fake_quantize":
        fo = torch.empty(x.shape, dtype=torch.bfloat16, device=dev)
        fn = lambda: ops.mixfp4_fake_quantize(x, 15, 16, torch.bfloat16, out=fo, workspace=ws)
        work = x.numel() * (4.0 + 1.0 / 16)
    elif args.kernel == "quantize_rht":
        fn = lambda: ops.mixfp4_quantize_rht(x, out=qx, workspace=ws)
        work = x.numel() * QUANT_BYTES_PER_ELEM
    else:
        out = torch.empty(x.shape, dtype=torch.float32, device=dev)
        fn = lambda: ops.mixfp4_dequantize(qx, out=out)
        work = x.numel() * (0.5 + 1.0 / 16 + 4.0)
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    is_gemm = args.kernel.startswith("gemm")
    unit = "TFLOP/s" if is_gemm else "GB/s"
    rate = work / (ms * 1e-3) / (1e12 if is_gemm else 1e9)
    print(json.dumps({"kernel": args.kernel, "workload": args.workload, "ms": round(ms, 5),
                      "rate": round(rate, 1), "unit": unit}))


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the other configs' GEMM lines")
    ap.add_argument("--no-sweep", action="store_true", help="skip the quantizer sweep over 2^20..2^30 elements")
    ap.add_argument("--kernel", choices=["gemm", "gemm_native", "gemm_native_fewrows", "split_native", "quantize", "quantize_rht", "quantize_colwise",
                             "quantize_2d", "transpose_2d", "fake_quantize", "quantize_colwise_rht", "quantize_sr",
                             "dequantize"], default=None,
                    help="profiling mode: launch only this kernel")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="tiny|attn|mlp|decode|hadamard|sweepNN (kernel-only mode)")
    args = ap.parse_args(argv)
    if args.kernel:
        return run_kernel_only(args)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
