#!/usr/bin/env python
"""Benchmark of the PalQuant layer hot path on GB300.

One step = one pass of the whole hot path over one batch of the ResNet-18 stage-1
shaped PalQuant 3x3 layer (batch 64, 56x56, G = 4 groups of 64 channels, 2-bit
activations and weights, cyclic shuffle):
  (1) group-wise activation quantisation of the fp32 NHWC input (205.5 MB) into one
      byte per code in the channel-blocked layout the tensor cores read, and (2) the
      fused layer: B-bit group convolution on the tensor cores, rescale, ReLU,
      cyclic-shuffle output permutation and requantisation into the next layer's
      codes (51.4 MB, same layout).
Inputs are resident in HBM when the timed region starts; two input buffers are used
in turn so each step reads an input larger than L2 that the previous step did not.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "PalQuant layer int TOPS and % of GB300 dense INT8 peak; ResNet-18-shaped images/s"
UNIT = "TOPS"
WORKLOAD = "ResNet-18 stage-1 3x3 PalQuant layer: batch 64, 56x56, G=4 groups of 64->64, b=2, stride 1, pad 1, cyclic shuffle"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "dram_traffic.json")
CSRC = os.path.join(ROOT, "paper_2208_01944_gb300", "csrc")


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--min-warmup-s", type=float, default=0.5,
                    help="keep warming up (and the GPU busy) for at least this long after the clock sampler starts; "
                         "0 for profilers")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target CPU time of the oracle baseline sample")
    ap.add_argument("--profile-layer", default=None, metavar="CONFIG",
                    help="only run the fused layer of CONFIG (config0, config1, config3_0..4, config4) --reps times "
                         "on random codes (codes out), for profilers; prints nothing else")
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--profile-stem", type=int, default=0, metavar="N",
                    help="only run the network's fp32 7x7 stem convolution on N 224x224 images --reps times, "
                         "for profilers; prints nothing else")
    ap.add_argument("--profile-format", default="c16", choices=["c16", "f4", "f32"],
                    help="input of --profile-layer: codes one per byte, packed FP4 nibbles, or fp32 activations "
                         "quantised on load (the benchmark step)")
    ap.add_argument("--no-resnet", action="store_true", help="skip the ResNet-18-shaped network measurement")
    ap.add_argument("--resnet-batch", type=int, default=128)
    ap.add_argument("--resnet-reps", type=int, default=20)
    ap.add_argument("--no-layers", action="store_true", help="skip the per-config layer measurements")
    ap.add_argument("--layer-reps", type=int, default=50)
    return ap.parse_args()


def run_profile_layer(name: str, reps: int, fmt_name: str = "c16"):
    """The fused layer alone, for profiling: random codes and weights of the named workload."""
    import numpy as np
    import torch

    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300 import synth, workloads

    c = workloads.BENCH_CONFIGS[name]
    dev = torch.device("cuda:0")
    gen = synth.generator(0)
    f4 = fmt_name == "f4"
    if fmt_name == "f32":  # fp32 activations, quantised on load: the benchmark step
        x = torch.from_numpy(synth.half_normal((c.N, c.H, c.W, c.G * c.Cin_g), gen)).to(dev)
        wq = synth.random_codes((c.G, c.Cout_g, c.k, c.k, c.Cin_g), c.bits_w, gen, signed=True)
        d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w,
                         c.bits_out, code_format=B.PQ_CODES_C16)
        wp = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d)).to(dev)
        qo = torch.empty(c.out_elems, dtype=torch.uint8, device=dev)
        m = np.full(c.G, 0.01, np.float32)
        inv = np.full(c.G, 1.3, np.float32)
        for _ in range(reps):
            B.palquant_quantize_layer_fused(x, inv, wp, d, m, m, B.shuffle(c.shuffle_kind, c.shuffle_shift), None,
                                            None, None, qo)
        st = B.palquant_sync_check()
        assert st == B.PQ_OK, B.strerror(st)
        return
    if f4:  # two random codes per byte, one per nibble
        lo = synth.random_codes((c.in_elems // 2,), c.bits_a, gen)
        q = torch.from_numpy(lo | (synth.random_codes((c.in_elems // 2,), c.bits_a, gen) << 4)).to(dev)
    else:
        q = torch.from_numpy(synth.random_codes((c.N, c.H, c.W, c.G * c.Cin_g), c.bits_a, gen)).to(dev)
    wq = synth.random_codes((c.G, c.Cout_g, c.k, c.k, c.Cin_g), c.bits_w, gen, signed=True)
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w, c.bits_out,
                     code_format=B.PQ_CODES_C32F4 if f4 else B.PQ_CODES_C16)
    wp = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d)).to(dev)
    qo = torch.empty(c.out_elems // (2 if f4 else 1), dtype=torch.uint8, device=dev)
    m = np.full(c.G, 0.01, np.float32)
    for _ in range(reps):
        B.palquant_layer_fused(q, wp, d, m, m, B.shuffle(c.shuffle_kind, c.shuffle_shift), None, None, None, qo)
    st = B.palquant_sync_check()
    assert st == B.PQ_OK, B.strerror(st)


def run_profile_stem(N: int, reps: int):
    """The network's stem with its max pooling (7x7 stride-2 pad-3 fp32 convolution
    3 -> 128 channels + ReLU, then 3x3 stride-2 pad-1 max pooling, one kernel) on N
    synthetic 224x224 images, for profiling."""
    import torch

    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300 import synth

    dev = torch.device("cuda:0")
    x, params = synth.resnet18_inputs(N, seed=0)
    xd = torch.from_numpy(x).to(dev)
    wd = torch.from_numpy(params["stem"]).to(dev)
    pool = torch.empty((N, 56, 56, wd.shape[0]), dtype=torch.float32, device=dev)
    for _ in range(reps):
        B.palquant_stem_pool_f32(xd, wd, None, pool, N, 224, 224, wd.shape[0])
    st = B.palquant_sync_check()
    assert st == B.PQ_OK, B.strerror(st)


def peaks():
    try:
        with open(PEAKS_FILE) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "source": "fallback"}


def source_sha(files):
    h = hashlib.sha256()
    for fn in files:
        with open(os.path.join(CSRC, fn), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


KERNEL_SOURCES = {
    "pq_conv_tc_kernel<quantise-on-load>": ["conv_tc.cu", "pq_device.cuh", "pq_internal.h"],
    "pq_quantize_c16": ["quantize.cu", "pq_device.cuh", "pq_internal.h"],
    "pq_conv_tc_kernel": ["conv_tc.cu", "pq_device.cuh", "pq_internal.h"],
    "pq_conv_tc_kernel<FP4, quantise-on-load>": ["conv_tc.cu", "pq_device.cuh", "pq_internal.h"],
}


def dram_traffic(kernel):
    """DRAM bytes per launch from the committed ncu summary, if the kernel source is unchanged."""
    try:
        with open(TRAFFIC_FILE) as f:
            d = json.load(f)[kernel]
        if d.get("source_sha") != source_sha(KERNEL_SOURCES[kernel]):
            return None
        return d["bytes_per_launch"]
    except Exception:
        return None


def max_over_ranks(x: float, world: int, device="cpu") -> float:
    """The largest of the ranks' values of x (a time), all_reduce(MAX) over the
    process group (NCCL on the GPU, gloo on the CPU); x itself with one rank."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, world: int, ms: float) -> float:
    """Units per second of the whole job: every rank processed `units_per_rank` in
    `ms` (the slowest rank's time), weak scaling."""
    return units_per_rank * world / (ms / 1e3)


def queue_ahead(stream, ms: float = 3.0):
    """Enqueue a bounded spin kernel (torch's cycle-count sleep, about `ms` at the SM
    clock) on `stream` just before a timed region.  While it runs, the host queues the
    region's start event and its first launches, so the region holds device work
    only: no host launch latency before the first kernel, and no idle GPU entering
    the region."""
    import torch

    with torch.cuda.stream(stream):
        torch.cuda._sleep(int(ms * 1e-3 * 2.0e9))


def timed_region(dev, stream, launch, n):
    """Device time (ms) of `n` back-to-back launches between two CUDA events on
    `stream`, queued behind queue_ahead(); `launch(i)` enqueues launch i on `stream`."""
    import torch

    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    queue_ahead(stream)
    with torch.cuda.stream(stream):
        start.record(stream)
        for i in range(n):
            launch(i)
        stop.record(stream)
    torch.cuda.synchronize(dev)
    return start.elapsed_time(stop)


def launch_spread(dev, stream, launch, n):
    """Diagnostic pass (outside any timed region): `n` launches with an event pair
    around each, queued behind queue_ahead(); min / median / max device time per
    launch in microseconds.  The events between launches keep each launch from
    overlapping its neighbour's tail, so these times sit a little above the
    region average."""
    import torch

    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    queue_ahead(stream)
    with torch.cuda.stream(stream):
        for i in range(n):
            ev[i][0].record(stream)
            launch(i)
            ev[i][1].record(stream)
    torch.cuda.synchronize(dev)
    t = sorted(a.elapsed_time(b) * 1e3 for a, b in ev)
    return {"min_us": t[0], "median_us": t[len(t) // 2], "max_us": t[-1], "launches": n,
            "how": "separate pass, an event pair around each launch"}


class ClockSampler:
    """nvidia-smi clock / throttle sampling while the timed region runs."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.QUERY,
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.25)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        rows = [r.split(",") for r in out.strip().splitlines() if r.strip()]
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [v.strip() for v in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax = float(r[2])
            except ValueError:
                continue
            for name, v in zip(names, r[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        sm.sort()
        med = sm[len(sm) // 2] if sm else None
        return {"sm_mhz": med, "sm_max_mhz": smax, "reasons": sorted(reasons), "samples": len(sm)}


def make_layer_inputs():
    from paper_2208_01944_gb300 import synth, workloads

    c = workloads.CONFIG1
    x, w = synth.layer_inputs(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, seed=0)
    return c, x, w


# ---------------------------------------------------------------------------
# Reference arm: the CPU oracle, as it stands, on the host cores.
# ---------------------------------------------------------------------------
def oracle_sample_step(c, x, w, n_img, inv_s, inv_sw, m_out, m_req):
    import oracle

    xs = x[:n_img]
    q = oracle.quantize_act(xs, c.G, c.bits_a, inv_s)
    wq = oracle.quantize_weights(w, c.bits_w, inv_sw)
    oracle.layer(q, wq, c.stride, c.pad, m_out, m_req, c.shuffle_kind, c.shuffle_shift, relu=c.relu, bits_out=c.bits_out)


def oracle_setup(c, x, w):
    import oracle

    s_a = oracle.act_step(x[:4], c.G, c.bits_a)
    s_w = oracle.weight_step(w, c.bits_w)
    m_out, m_req = oracle.epilogue_scales(s_w, s_a, s_a, 1.0, c.shuffle_kind, c.shuffle_shift)
    return oracle.inv_step(s_a), oracle.inv_step(s_w), m_out, m_req


def oracle_images_for(seconds, c, x, w, setup):
    t0 = time.perf_counter()
    oracle_sample_step(c, x, w, 1, *setup)
    per_img = time.perf_counter() - t0
    return max(1, min(c.N, int(seconds / max(per_img, 1e-6)))), per_img


def cpu_baseline(c, x, w, seconds):
    import oracle

    setup = oracle_setup(c, x, w)
    n_img, _ = oracle_images_for(seconds, c, x, w, setup)
    t0 = time.perf_counter()
    oracle_sample_step(c, x, w, n_img, *setup)
    dt = time.perf_counter() - t0
    ops = c.int_ops * n_img / c.N
    return {"value": ops / dt / 1e12, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{n_img} of the {c.N} images of the workload (quantize + group conv + epilogue), {dt:.2f} s"}


def run_reference(args, rank, world):
    if rank != 0:
        return
    import oracle

    c, x, w = make_layer_inputs()
    setup = oracle_setup(c, x, w)
    # each step: a bounded sample (whole images) sized so K + W steps take a few minutes
    budget = 150.0 / max(1, args.steps + args.warmup)
    n_img, _ = oracle_images_for(min(budget, 20.0), c, x, w, setup)
    for _ in range(args.warmup):
        oracle_sample_step(c, x, w, n_img, *setup)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_sample_step(c, x, w, n_img, *setup)
    dt = (time.perf_counter() - t0) / max(1, args.steps)
    ops = c.int_ops * n_img / c.N
    value = ops / dt / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "sample_images_per_step": n_img, "global_batch": c.N},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
                         "sample": f"{n_img} of {c.N} images per step (quantize + group conv + epilogue)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# The single-layer configs (0, 1, the b/G sweep 3, the 1x1 layer 4) and the
# quantiser alone: per-launch device time of the fused layer, codes in and out.
# ---------------------------------------------------------------------------
L2_BYTES = 126 * 1024 * 1024

# Tensor-core rates (TFLOP/s, 2 x MACs) that an MMA issue-loop probe measured on
# this GB300 by the MMA's N (M = 128, cta_group::1, one CTA per SM issuing nine
# taps of shifted A addresses with nothing else running): the ceiling of the MMA
# shape a layer's plan uses.  N = 64 is bound by shared-memory operand reads (6 KB
# per MMA, 24.6 ns for FP8 K = 32 and block-scaled FP4 K = 64 alike); N >= 128 by
# the tensor core (FP8 4.86, FP4 9.73 PFLOP/s).
MMA_PROBE_TFLOPS = {"fp8": {64: 3238.0, 128: 4843.0, 256: 4858.0},
                    "fp4": {64: 6486.0, 128: 9708.0, 256: 9732.0}}


def measure_layer_configs(dev, args):
    """Each config's fused layer in timed mode (channel-blocked codes in, codes out)
    and the quantiser on the config-1 and config-4 inputs.  Input/output buffer sets
    rotate so that the bytes one pass touches total at least 2x L2; CUDA events on the
    launching stream bracket `reps` launches after 3 warm-up launches."""
    import numpy as np
    import torch

    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300 import synth, workloads

    pk = peaks()
    fp8_peak = 2.0 * pk["bf16_tflops"]
    fp4_peak = 6.0 * pk["bf16_tflops"]
    stream = torch.cuda.Stream(device=dev)
    fmt = B.PQ_CODES_C16
    out = {}
    reps = args.layer_reps

    def timed(launch, n_sets):
        with torch.cuda.stream(stream):
            for i in range(3):
                launch(i % n_sets)
        torch.cuda.synchronize(dev)
        ms = timed_region(dev, stream, lambda i: launch(i % n_sets), reps)
        st = B.palquant_sync_check(stream)
        assert st == B.PQ_OK, B.strerror(st)
        return ms / reps

    for name, c in workloads.BENCH_CONFIGS.items():
        gen = synth.generator(0)
        per_set = c.in_elems + c.out_elems
        n_sets = max(1, min(16, -(-2 * L2_BYTES // per_set)))
        q = torch.from_numpy(synth.random_codes((c.N, c.H, c.W, c.G * c.Cin_g), c.bits_a, gen)).to(dev)
        qs = [q] + [q.clone() for _ in range(n_sets - 1)]
        wq = synth.random_codes((c.G, c.Cout_g, c.k, c.k, c.Cin_g), c.bits_w, gen, signed=True)
        # independent buffer sets: each launch may start loading while the previous one finishes
        d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w, c.bits_out,
                         int(c.relu), code_format=fmt, flags=B.PQ_LAYER_INPUTS_READY)
        wp = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d)).to(dev)
        qo = [torch.empty((c.N, c.Ho, c.Wo, c.G * c.Cout_g), dtype=torch.uint8, device=dev) for _ in range(n_sets)]
        torch.cuda.synchronize(dev)
        m = np.full(c.G, 0.01, np.float32)
        shuf = B.shuffle(c.shuffle_kind, c.shuffle_shift)
        ms = timed(lambda i: B.palquant_layer_fused(qs[i], wp, d, m, m, shuf, None, None, None, qo[i], stream=stream),
                   n_sets)
        byt = c.in_elems + c.out_elems + c.weight_elems
        tops = c.int_ops / (ms / 1e3) / 1e12
        plan = B.palquant_conv_plan(d).as_dict()
        probe = None if plan["pointwise"] else MMA_PROBE_TFLOPS["fp8"].get(plan["n_block"])
        out[name] = {"shape": c.name, "us": ms * 1e3, "tops": tops, "frac_fp8_peak": tops / fp8_peak,
                     "frac_mma_probe": tops / probe if probe else None,
                     "algorithmic_gbs": byt / (ms / 1e3) / 1e9, "frac_hbm": byt / (ms / 1e3) / 1e9 / pk["hbm_gbs"],
                     "buffer_sets": n_sets,
                     "kernel": "pq_pointwise_tc_kernel" if plan["pointwise"] else "pq_conv_tc_kernel",
                     "plan": ({} if plan["pointwise"] else
                              {k: plan[k] for k in ("m_tiles", "n_block", "k_chunk", "weights_resident", "work_items")})}
        del qs, qo, q, wp
        # the same layer with packed FP4 codes (block-scaled FP4 tensor path), where it applies
        d4 = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w,
                          c.bits_out, int(c.relu), code_format=B.PQ_CODES_C32F4, flags=B.PQ_LAYER_INPUTS_READY)
        if B.palquant_conv_plan(d4).supported:
            nin, nout = c.in_elems // 2, c.out_elems // 2
            n4 = max(1, min(16, -(-2 * L2_BYTES // (nin + nout))))
            lo = synth.random_codes((nin,), c.bits_a, gen)
            q4 = torch.from_numpy(lo | (synth.random_codes((nin,), c.bits_a, gen) << 4)).to(dev)
            q4s = [q4] + [q4.clone() for _ in range(n4 - 1)]
            wp4 = torch.from_numpy(B.palquant_pack_weight_codes_host(wq, d4)).to(dev)
            qo4 = [torch.empty(nout, dtype=torch.uint8, device=dev) for _ in range(n4)]
            torch.cuda.synchronize(dev)
            ms4 = timed(lambda i: B.palquant_layer_fused(q4s[i], wp4, d4, m, m, shuf, None, None, None, qo4[i],
                                                         stream=stream), n4)
            tops4 = c.int_ops / (ms4 / 1e3) / 1e12
            byt4 = nin + nout + c.weight_elems // 2
            plan4 = B.palquant_conv_plan(d4).as_dict()
            probe4 = MMA_PROBE_TFLOPS["fp4"].get(plan4["n_block"])
            out[name + "_fp4"] = {"shape": c.name + ", packed FP4 codes", "us": ms4 * 1e3, "tops": tops4,
                                  "frac_fp4_peak": tops4 / fp4_peak, "frac_fp8_peak": tops4 / fp8_peak,
                                  "frac_mma_probe": tops4 / probe4 if probe4 else None,
                                  "algorithmic_gbs": byt4 / (ms4 / 1e3) / 1e9,
                                  "frac_hbm": byt4 / (ms4 / 1e3) / 1e9 / pk["hbm_gbs"], "buffer_sets": n4,
                                  "plan": {k: plan4[k] for k in ("m_tiles", "n_block", "k_chunk", "weights_resident",
                                                                  "work_items")}}
            del q4s, qo4, q4, wp4
    out["table2_4bit_on_2bit"] = measure_bitsplit_vs_palquant(dev, stream, timed, pk, fp8_peak)
    for name in ("config1", "config4"):
        c = workloads.BENCH_CONFIGS[name]
        shape = (c.N, c.H, c.W, c.G * c.Cin_g)
        per_set = c.in_elems * 5
        n_sets = max(1, min(8, -(-2 * L2_BYTES // per_set)))
        x = torch.randn(shape, device=dev).abs_()
        xs = [x] + [x.clone() for _ in range(n_sets - 1)]
        qq = [torch.empty(shape, dtype=torch.uint8, device=dev) for _ in range(n_sets)]
        inv = np.full(c.G, 1.3, np.float32)
        ms = timed(lambda i: B.palquant_quantize_act(xs[i], qq[i], c.N, c.H, c.W, c.G, c.Cin_g, c.bits_a, inv,
                                                     code_format=fmt, stream=stream), n_sets)
        gbs = per_set / (ms / 1e3) / 1e9
        out["quantize_" + name] = {"shape": f"{c.N}x{c.H}x{c.W}x{c.G * c.Cin_g} fp32 -> channel-blocked codes",
                                   "us": ms * 1e3, "gbs": gbs, "frac_hbm": gbs / pk["hbm_gbs"], "buffer_sets": n_sets}
        qq4 = [torch.empty(c.in_elems // 2, dtype=torch.uint8, device=dev) for _ in range(n_sets)]
        ms4 = timed(lambda i: B.palquant_quantize_act(xs[i], qq4[i], c.N, c.H, c.W, c.G, c.Cin_g, c.bits_a, inv,
                                                      code_format=B.PQ_CODES_C32F4, stream=stream), n_sets)
        b4 = c.in_elems * 4 + c.in_elems // 2
        out["quantize_" + name + "_fp4"] = {"shape": f"{c.N}x{c.H}x{c.W}x{c.G * c.Cin_g} fp32 -> packed FP4 codes",
                                            "us": ms4 * 1e3, "gbs": b4 / (ms4 / 1e3) / 1e9,
                                            "frac_hbm": b4 / (ms4 / 1e3) / 1e9 / pk["hbm_gbs"], "buffer_sets": n_sets}
        del xs, qq, x, qq4
    torch.cuda.empty_cache()
    out.update(measure_qat(dev, stream, timed, pk))
    return out


def measure_qat(dev, stream, timed, pk):
    """Quantisation-aware training of the quantiser on the config-1 activation
    tensor (64x56x56x256 fp32, G = 4, learned bounds l, u per group): the forward
    (8 bytes per element) and the straight-through backward with the gradients of l
    and u (12 bytes per element); each tensor is larger than L2, two sets rotate."""
    import numpy as np
    import torch

    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300 import workloads

    c = workloads.CONFIG1
    P, G, Cg = c.N * c.H * c.W, c.G, c.Cin_g
    n = P * G * Cg
    l = np.full(G, 0.05, np.float32)
    u = np.full(G, 2.0, np.float32)
    xs = [torch.randn((P, G * Cg), device=dev).abs_() for _ in range(2)]
    dys = [torch.randn((P, G * Cg), device=dev) for _ in range(2)]
    outs = [torch.empty((P, G * Cg), device=dev) for _ in range(2)]
    dl = torch.empty(G, dtype=torch.float64, device=dev)
    du = torch.empty(G, dtype=torch.float64, device=dev)
    sb = B.palquant_fake_quant_scratch_bytes(P, G, Cg)
    scratch = torch.empty(sb, dtype=torch.uint8, device=dev)
    ms_f = timed(lambda i: B.palquant_fake_quant_forward(xs[i], outs[i], P, G, Cg, c.bits_a, 0, l, u, stream=stream), 2)
    ms_b = timed(lambda i: B.palquant_fake_quant_backward(xs[i], dys[i], outs[i], dl, du, P, G, Cg, c.bits_a, 0, l, u,
                                                          scratch, sb, stream=stream), 2)
    res = {}
    for key, ms, byt in (("qat_forward_config1", ms_f, 8 * n), ("qat_backward_config1", ms_b, 12 * n)):
        gbs = byt / (ms / 1e3) / 1e9
        res[key] = {"shape": f"{c.N}x{c.H}x{c.W}x{G * Cg} fp32, G={G}, b={c.bits_a}", "us": ms * 1e3, "gbs": gbs,
                    "frac_hbm": gbs / pk["hbm_gbs"], "algorithmic_bytes": byt, "buffer_sets": 2}
    del xs, dys, outs
    torch.cuda.empty_cache()
    return res


def measure_bitsplit_vs_palquant(dev, stream, timed, pk, fp8_peak):
    """The GPU analogue of the paper's Table 2 comparison on one 3x3 layer shape
    (batch 128, 28x28, per-group width C = 256): a 4-bit layer C -> C run on 2-bit
    operands by bit-level decomposition (Eq. 4: slice kernel + one pass over the 4
    shifted 2-bit products), the same 4-bit layer run directly (GB300's FP8 tensor
    cores take 4-bit codes natively), and the PalQuant layer that replaces it (G = 2
    groups of C -> C at 2 bits, Sec. 4.1).  All produce next-layer codes."""
    import numpy as np
    import torch

    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300 import synth

    N, H, C, k = 128, 28, 256, 3
    fmt = B.PQ_CODES_C16
    gen = synth.generator(5)
    res = {"shape": f"{N}x{H}x{H}, 3x3, C={C} per group, codes in and out"}
    m1 = np.full(1, 0.01, np.float32)
    # direct 4-bit and decomposed (one group, C -> C)
    d4 = B.layer_desc(N, H, H, 1, C, C, k, 1, 1, 4, 4, 4, 1, code_format=fmt)
    R = 5  # rotating input / output sets: each pass touches more than L2
    q4 = [torch.from_numpy(synth.random_codes((N, H, H, C), 4, gen)).to(dev) for _ in range(R)]
    w4 = synth.random_codes((1, C, k, k, C), 4, gen, signed=True)
    wp4 = torch.from_numpy(B.palquant_pack_weight_codes_host(w4, d4)).to(dev)
    qo = [torch.empty((N, H, H, C), dtype=torch.uint8, device=dev) for _ in range(R)]
    none = B.shuffle(0, 0)
    ms_direct = timed(lambda i: B.palquant_layer_fused(q4[i], wp4, d4, m1, m1, none, None, None, None, qo[i],
                                                       stream=stream), R)
    t = B.palquant_bitsplit_desc(d4, 2)
    wps = torch.from_numpy(B.palquant_bitsplit_pack_weight_codes_host(w4, d4, 2)).to(dev)
    xs_bytes = B.palquant_bitsplit_scratch_bytes(d4, 2)
    xs = torch.empty(xs_bytes, dtype=torch.uint8, device=dev)

    def split_run(i):
        B.palquant_bitsplit_act(q4[i], xs, xs_bytes, d4, 2, stream=stream)
        B.palquant_layer_fused(xs, wps, t, m1, m1, none, None, None, None, qo[i], stream=stream)

    ms_split = timed(split_run, R)
    # PalQuant: 2 groups of C -> C at 2 bits (2C channels), cyclic shuffle
    dp = B.layer_desc(N, H, H, 2, C, C, k, 1, 1, 2, 2, 2, 1, code_format=fmt)
    qp = [torch.from_numpy(synth.random_codes((N, H, H, 2 * C), 2, gen)).to(dev) for _ in range(R)]
    wpq = synth.random_codes((2, C, k, k, C), 2, gen, signed=True)
    wpp = torch.from_numpy(B.palquant_pack_weight_codes_host(wpq, dp)).to(dev)
    qop = [torch.empty((N, H, H, 2 * C), dtype=torch.uint8, device=dev) for _ in range(R)]
    m2 = np.full(2, 0.01, np.float32)
    ms_pal = timed(lambda i: B.palquant_layer_fused(qp[i], wpp, dp, m2, m2, B.shuffle(1, 1), None, None, None, qop[i],
                                                    stream=stream), R)
    ops4 = 2 * N * H * H * C * k * k * C
    res.update({
        "direct_4bit_us": ms_direct * 1e3,
        "bit_decomposed_4bit_on_2bit_us": ms_split * 1e3,
        "palquant_2bit_G2_us": ms_pal * 1e3,
        "speedup_palquant_vs_bit_decomposed": ms_split / ms_pal,
        "int_ops": {"direct_4bit": ops4, "bit_decomposed_2bit_products": 4 * ops4, "palquant_G2": 2 * ops4},
        "note": "the 4 products of Eq. 4 form one tensor-core pass after a slice kernel that writes each "
                "activation slice once (K = 2C slice channels, each meeting its 2 weight slices as taps)",
    })
    return res


# ---------------------------------------------------------------------------
# The ResNet-18-shaped network (config 2): images/s of the whole forward.
# ---------------------------------------------------------------------------
def measure_resnet18_paper(dev, world, args):
    """The same network with the paper's placement of the shuffles (Sec. 4.3): a cyclic
    shuffle module at each stage's start, the channel shuffle at each stage's end (and
    the quantiser that re-codes each stage's output), timed the same way."""
    import torch

    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300 import synth
    from paper_2208_01944_gb300.resnet18 import PalQuantResNet18

    N = args.resnet_batch
    x_np, params = synth.resnet18_inputs(N, seed=0, cyclic_modules=True)
    net = PalQuantResNet18(params, N, device=dev, placement="paper")
    xs = [torch.from_numpy(x_np).to(dev)]
    xs.append(torch.flip(xs[0], dims=[0]).contiguous())
    net.calibrate(xs[0])
    graphs = [net.capture(x) for x in xs]
    for i in range(3):
        net.replay(graphs[i & 1])
    torch.cuda.synchronize(dev)
    R = args.resnet_reps
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    queue_ahead(net.stream)
    e0.record(net.stream)
    for i in range(R):
        net.replay(graphs[i & 1])
    e1.record(net.stream)
    torch.cuda.synchronize(dev)
    st = B.palquant_sync_check(net.stream)
    assert st == B.PQ_OK, B.strerror(st)
    ms = max_over_ranks(e0.elapsed_time(e1) / R, world, dev)
    res = {"images_per_s": whole_job_rate(N, world, ms), "ms_per_batch": ms,
           "palquant_body_tops": whole_job_rate(net.body_int_ops(), world, ms) / 1e12,
           "gpu_launches_per_forward": net.launches_per_forward(),
           "timed": "CUDA-graph replay; 4 cyclic shuffle modules, 20 PalQuant layers, 4 quantisers"}
    marks = []
    net.forward(xs[0], marks)
    torch.cuda.synchronize(dev)
    res["stages_ms"] = {name: marks[i - 1][1].elapsed_time(ev) for i, (name, ev) in enumerate(marks) if i > 0}
    del graphs, net
    torch.cuda.empty_cache()
    return res


def measure_resnet18(dev, world, args):
    """Forward of the ResNet-18-shaped PalQuant network (224x224, G = 2, b = 2, per-group
    widths 64/128/256/512, fp32 stem and FC) on a batch of synthetic images, replayed
    from CUDA graphs; two input batches (154 MB together, more than L2) alternate."""
    import numpy as np
    import torch

    from paper_2208_01944_gb300 import binding as B
    from paper_2208_01944_gb300 import synth
    from paper_2208_01944_gb300.resnet18 import PalQuantResNet18

    N = args.resnet_batch
    x_np, params = synth.resnet18_inputs(N, seed=0)
    net = PalQuantResNet18(params, N, device=dev)
    xs = [torch.from_numpy(x_np).to(dev)]
    xs.append(torch.flip(xs[0], dims=[0]).contiguous())
    net.calibrate(xs[0])  # step initialisation, untimed
    graphs = [net.capture(x) for x in xs]
    for i in range(3):
        net.replay(graphs[i & 1])
    torch.cuda.synchronize(dev)
    R = args.resnet_reps
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    queue_ahead(net.stream)
    e0.record(net.stream)
    for i in range(R):
        net.replay(graphs[i & 1])
    e1.record(net.stream)
    torch.cuda.synchronize(dev)
    st = B.palquant_sync_check(net.stream)
    assert st == B.PQ_OK, B.strerror(st)
    ms = max_over_ranks(e0.elapsed_time(e1) / R, world, dev)
    out = {"workload": "ResNet-18-shaped PalQuant forward: batch %d, 224x224x3 N(0,1) images, G=2, b=2, per-group widths "
                       "64/128/256/512, fp32 7x7 stem + max pooling and fp32 FC, cyclic shuffle after each block" % N,
           "images_per_s": whole_job_rate(N, world, ms), "ms_per_batch": ms, "batch_per_gpu": N, "reps": R,
           "palquant_body_tops": whole_job_rate(net.body_int_ops(), world, ms) / 1e12,
           "timed": "CUDA-graph replay of the whole forward (stem, pooling, quantiser, 20 PalQuant layers, pooling, FC)",
           "gpu_launches_per_forward": net.launches_per_forward(), "data": "synthetic",
           "code_layout": ("packed FP4 nibbles [N][C/32][H][W][16 B] between layers" if net.fmt == B.PQ_CODES_C32F4
                           else "channel-blocked [N][C/16][H][W][16], one byte per code")}
    # where the time goes: one eager forward with events between its stages
    marks = []
    net.forward(xs[0], marks)
    torch.cuda.synchronize(dev)
    out["stages_ms"] = {name: marks[i - 1][1].elapsed_time(ev) for i, (name, ev) in enumerate(marks) if i > 0}
    del graphs, net
    torch.cuda.empty_cache()
    out["paper_placement"] = measure_resnet18_paper(dev, world, args)
    if not args.no_cpu_baseline and world == 1:
        import time

        import oracle
        import oracle.resnet as OR

        x1, p1 = synth.resnet18_inputs(1, seed=0)
        steps = OR.calibrate(x1, p1, 2, 2)
        t0 = time.perf_counter()
        OR.forward(x1, p1, 2, 2, steps)
        dt = time.perf_counter() - t0
        out["cpu_baseline"] = {"value": 1.0 / dt, "unit": "images/s", "cores": oracle.num_threads(), "kind": "oracle",
                               "sample": f"1 image, forward with given steps, {dt:.2f} s"}
    return out


def measure_unfused_step(dev, stream, c, xs, q, inv_s, wp, d, m_out, m_req, shuf, q_out, K, world):
    """The same step as two launches (the quantiser writing codes, then the layer
    reading them back): K timed steps after 3 warm-up steps, per-kernel events."""
    import torch

    from paper_2208_01944_gb300 import binding as B

    fmt = B.PQ_CODES_C16

    def launch(i):
        B.palquant_quantize_act(xs[i & 1], q, c.N, c.H, c.W, c.G, c.Cin_g, c.bits_a, inv_s, code_format=fmt,
                                stream=stream)
        B.palquant_layer_fused(q, wp, d, m_out, m_req, shuf, None, None, None, q_out, stream=stream)

    with torch.cuda.stream(stream):
        for i in range(3):
            launch(i)
    torch.cuda.synchronize(dev)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    queue_ahead(stream)
    with torch.cuda.stream(stream):
        start.record(stream)
        for i in range(K):
            ev[i][0].record(stream)
            B.palquant_quantize_act(xs[i & 1], q, c.N, c.H, c.W, c.G, c.Cin_g, c.bits_a, inv_s, code_format=fmt,
                                    stream=stream)
            ev[i][1].record(stream)
            B.palquant_layer_fused(q, wp, d, m_out, m_req, shuf, None, None, None, q_out, stream=stream)
            ev[i][2].record(stream)
        stop.record(stream)
    torch.cuda.synchronize(dev)
    st = B.palquant_sync_check(stream)
    assert st == B.PQ_OK, B.strerror(st)
    return {"ms_per_step": max_over_ranks(start.elapsed_time(stop) / K, world, dev),
            "t_quant": sum(e[0].elapsed_time(e[1]) for e in ev) / K,
            "t_conv": sum(e[1].elapsed_time(e[2]) for e in ev) / K}


def unfused_summary(r, c, pk, world):
    """The two-launch step's throughput and the rooflines of its kernels."""
    fp8_peak = 2.0 * pk["bf16_tflops"]
    q_bytes = c.in_elems * 5  # 4-byte read + 1-byte write per element
    conv_bytes = c.in_elems + c.out_elems + c.weight_elems
    quant_gbs = q_bytes / (r["t_quant"] / 1e3) / 1e9
    conv_tops = c.int_ops / (r["t_conv"] / 1e3) / 1e12
    return {
        "value": whole_job_rate(c.int_ops, world, r["ms_per_step"]) / 1e12, "unit": UNIT,
        "ms_per_step": r["ms_per_step"],
        "timed": "quantiser (fp32 NHWC -> codes) + layer (codes -> next-layer codes), two launches",
        "roofline_kernels": [
            {"kernel": "pq_quantize_c16", "bound": "hbm", "achieved": quant_gbs, "peak": pk["hbm_gbs"],
             "unit": "GB/s", "frac": quant_gbs / pk["hbm_gbs"], "traffic": dram_traffic("pq_quantize_c16"),
             "algorithmic_bytes": q_bytes, "avg_launch_ms": r["t_quant"],
             "peak_source": f"{pk['source']} HBM copy bandwidth"},
            {"kernel": "pq_conv_tc_kernel", "bound": "tensor", "achieved": conv_tops, "peak": fp8_peak,
             "unit": "TFLOP/s", "frac": conv_tops / fp8_peak, "traffic": dram_traffic("pq_conv_tc_kernel"),
             "algorithmic_ops": c.int_ops, "algorithmic_bytes": conv_bytes, "avg_launch_ms": r["t_conv"],
             "hbm_frac": conv_bytes / (r["t_conv"] / 1e3) / 1e9 / pk["hbm_gbs"],
             "peak_source": f"{pk['source']} bf16 burst x 2 (dense FP8 E4M3, the exact-integer tensor path)"}],
        "gpu_launches": 2,
    }


def measure_fp4_step(dev, stream, c, xs, inv_s, w_np, inv_sw, m_out, m_req, shuf, K, world):
    """The same step (the quantiser fused into the layer, same steps and
    multipliers) with packed FP4 operands and output codes (PQ_CODES_C32F4, the
    block-scaled FP4 tensor path): K timed steps after 3 warm-up steps, one
    launch each, timed as a region (average launch duration = region / K)."""
    import torch

    from paper_2208_01944_gb300 import binding as B

    fmt = B.PQ_CODES_C32F4
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w, c.bits_out,
                     int(c.relu), code_format=fmt)
    nbytes = B.palquant_packed_weight_bytes(d)
    wp = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    B.palquant_pack_weights(w_np, d, inv_sw, wp, nbytes)
    q_out = torch.empty(c.out_elems // 2, dtype=torch.uint8, device=dev)
    torch.cuda.synchronize(dev)  # the packed weights are in place before the first launch
    # independent batches: each launch may start loading while the previous one finishes
    d_ready = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w,
                           c.bits_out, int(c.relu), code_format=fmt, flags=B.PQ_LAYER_INPUTS_READY)

    def launch(i):
        B.palquant_quantize_layer_fused(xs[i & 1], inv_s, wp, d_ready, m_out, m_req, shuf, None, None, None, q_out,
                                        stream=stream)

    with torch.cuda.stream(stream):
        for i in range(3):
            launch(i)
    torch.cuda.synchronize(dev)
    t = timed_region(dev, stream, launch, K) / K
    st = B.palquant_sync_check(stream)
    assert st == B.PQ_OK, B.strerror(st)
    return {"ms_per_step": max_over_ranks(t, world, dev), "t_step": t}


def fp4_summary(r, c, pk, world):
    """The FP4 step's throughput and the roofline of its one kernel: HBM-bound on
    the fp32 input and the nibble codes out; its tensor instructions are FP4
    (kind::mxf4), whose dense peak is the measured bf16 burst x 6 (nominal 13.5 /
    2.25 PFLOP/s)."""
    fp4_peak = 6.0 * pk["bf16_tflops"]
    step_bytes = c.in_elems * 4 + c.out_elems // 2 + c.weight_elems // 2
    gbs = step_bytes / (r["t_step"] / 1e3) / 1e9
    tops = c.int_ops / (r["t_step"] / 1e3) / 1e12
    return {
        "value": whole_job_rate(c.int_ops, world, r["ms_per_step"]) / 1e12, "unit": UNIT,
        "ms_per_step": r["ms_per_step"],
        "timed": "one launch per step: quantiser fused into the layer, packed FP4 operands and codes; "
                 "independent batches, each launch's loads start while the previous launch finishes",
        "code_layout": "packed FP4 nibbles [N][C/32][H][W][16 B], two 2-bit codes per byte",
        "dtype": "e2m1",
        "dtype_detail": "fp32 activations -> 2-bit codes as FP4 e2m1 x e2m1 weights, block scales 2^-4 -> f32 (exact)",
        "roofline_kernels": [
            {"kernel": "pq_conv_tc_kernel<FP4> (quantise on load)", "bound": "hbm", "achieved": gbs,
             "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": gbs / pk["hbm_gbs"],
             "traffic": dram_traffic("pq_conv_tc_kernel<FP4, quantise-on-load>"), "algorithmic_bytes": step_bytes,
             "algorithmic_ops": c.int_ops, "avg_launch_ms": r["t_step"], "tensor_tops": tops,
             "tensor_frac_fp4": tops / fp4_peak, "peak_source": f"{pk['source']} HBM copy bandwidth"}],
        "gpu_launches": 1,
    }


# ---------------------------------------------------------------------------
# Our arm.
# ---------------------------------------------------------------------------
def run_ours(args, rank, world, local_rank):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2208_01944_gb300 import binding as B

    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    c, x_np, w_np = make_layer_inputs()

    # ---- set-up (untimed): steps from the library's own calibration
    stream = torch.cuda.Stream(device=dev)
    xs = [torch.from_numpy(x_np).to(dev)]
    xs.append(torch.flip(xs[0], dims=[0]).contiguous())  # second input buffer (same values, other order)
    P = c.N * c.H * c.W
    scratch_bytes = B.palquant_act_steps_scratch_bytes(P, c.G)
    scratch = torch.empty(scratch_bytes, dtype=torch.uint8, device=dev)
    s_a = B.palquant_act_steps(xs[0], c.N, c.H, c.W, c.G, c.Cin_g, c.bits_a, scratch, scratch_bytes)
    fmt = B.PQ_CODES_C16
    d = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w, c.bits_out,
                     int(c.relu), code_format=fmt)
    s_w = B.palquant_weight_steps(w_np, d)
    # fl(1 / s) from the library: the requantisation multiplier of s_w = s_a = 1 onto the
    # step s, with no permutation
    ones = np.ones(c.G, dtype=np.float32)
    no_shuffle = B.shuffle(0, 0)
    inv_s = B.palquant_epilogue_scales(c.G, ones, ones, 1.0, s_a, no_shuffle)[1]
    inv_sw = B.palquant_epilogue_scales(c.G, ones, ones, 1.0, s_w, no_shuffle)[1]
    nbytes = B.palquant_packed_weight_bytes(d)
    wp = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    B.palquant_pack_weights(w_np, d, inv_sw, wp, nbytes)
    shuf = B.shuffle(c.shuffle_kind, c.shuffle_shift)
    q = torch.empty((c.N, c.H, c.W, c.G * c.Cin_g), dtype=torch.uint8, device=dev)
    out_shape = (c.N, c.Ho, c.Wo, c.G * c.Cout_g)
    # next layer's steps: calibrated on this layer's rescaled output
    m_out, _ = B.palquant_epilogue_scales(c.G, s_w, s_a, 1.0, None, shuf)
    y = torch.empty(out_shape, dtype=torch.float32, device=dev)
    B.palquant_quantize_act(xs[0], q, c.N, c.H, c.W, c.G, c.Cin_g, c.bits_a, inv_s, code_format=fmt)
    B.palquant_layer_fused(q, wp, d, m_out, m_out, shuf, None, None, y, None)
    s_next = B.palquant_act_steps(y, c.N, c.Ho, c.Wo, c.G, c.Cout_g, c.bits_out, scratch, scratch_bytes)
    m_out, m_req = B.palquant_epilogue_scales(c.G, s_w, s_a, 1.0, s_next, shuf)
    del y
    q_out = torch.empty(out_shape, dtype=torch.uint8, device=dev)
    assert B.palquant_sync_check() == B.PQ_OK
    # Steps are independent batches: no step writes another's input or the weights,
    # so each launch may start loading while the previous one finishes.
    d_ready = B.layer_desc(c.N, c.H, c.W, c.G, c.Cin_g, c.Cout_g, c.k, c.stride, c.pad, c.bits_a, c.bits_w,
                           c.bits_out, int(c.relu), code_format=fmt, flags=B.PQ_LAYER_INPUTS_READY)

    def step(i, s):
        # the whole hot path in one launch: quantise on load, group conv, rescale,
        # ReLU, cyclic remap, requantise
        B.palquant_quantize_layer_fused(xs[i & 1], inv_s, wp, d_ready, m_out, m_req, shuf, None, None, None, q_out,
                                        stream=s)

    # ---- warm-up: at least W steps, and the GPU kept busy until the clock sampler
    # (started first) is running, so the timed region does not start from an idle GPU
    sampler = ClockSampler(local_rank)
    sampler.start()
    t_warm = time.perf_counter()
    n_warm = 0
    while n_warm < args.warmup or time.perf_counter() - t_warm < args.min_warmup_s:
        with torch.cuda.stream(stream):
            for _ in range(min(50, max(1, args.warmup - n_warm)) if args.min_warmup_s <= 0 else 50):
                step(n_warm, stream)
                n_warm += 1
        torch.cuda.synchronize(dev)
    st = B.palquant_sync_check(stream)
    assert st == B.PQ_OK, B.strerror(st)

    # ---- timed region: K steps (one launch each) between two events on the
    # launching stream, queued behind a short spin kernel so that the region holds
    # the K launches back to back (no host launch latency before the first); the
    # step's average launch duration is the region / K, with no events between the
    # launches
    K = args.steps
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    elapsed_ms = timed_region(dev, stream, lambda i: step(i, stream), K)
    st = B.palquant_sync_check(stream)
    assert st == B.PQ_OK, B.strerror(st)
    # per-launch spread, from a separate diagnostic pass (not the timed region)
    spread = launch_spread(dev, stream, lambda i: step(i, stream), max(3, min(K, 200)))
    unfused = measure_unfused_step(dev, stream, c, xs, q, inv_s, wp, d, m_out, m_req, shuf, q_out, K, world)
    fp4 = measure_fp4_step(dev, stream, c, xs, inv_s, w_np, inv_sw, m_out, m_req, shuf, K, world)
    resnet = None if args.no_resnet else measure_resnet18(dev, world, args)
    layers = None if args.no_layers else measure_layer_configs(dev, args)
    clocks = sampler.stop()
    if world > 1:
        dist.barrier()
    t_step = elapsed_ms / K
    elapsed_ms = max_over_ranks(elapsed_ms, world, dev)
    ms_per_step = elapsed_ms / K
    ops_step = c.int_ops
    value = whole_job_rate(ops_step, world, ms_per_step) / 1e12

    # ---- end to end through the public API with host buffers (pinned), per step:
    # H2D copy of the step's fp32 input, the fused quantiser + layer, D2H copy of the
    # step's output codes.  Steps are pipelined over three streams with two device
    # input and output buffers: step i + 1's input copy and step i - 1's output copy
    # run while step i computes (the copy engines move about 210 GB/s each way, so the
    # 205.5 MB input copy sets the pace).
    x_host = torch.from_numpy(x_np).pin_memory()
    out_host = [torch.empty(out_shape, dtype=torch.uint8).pin_memory() for _ in range(2)]
    q_outs = [q_out, torch.empty(out_shape, dtype=torch.uint8, device=dev)]
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_comp = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]

    def e2e_steps(n):
        for i in range(n):
            b = i & 1
            if i >= 2:
                s_in.wait_event(ev_comp[b])  # step i - 2 has read input buffer b
            with torch.cuda.stream(s_in):
                xs[b].copy_(x_host, non_blocking=True)
                ev_in[b].record(s_in)
            stream.wait_event(ev_in[b])
            if i >= 2:
                stream.wait_event(ev_out[b])  # output buffer b has been copied out
            B.palquant_quantize_layer_fused(xs[b], inv_s, wp, d_ready, m_out, m_req, shuf, None, None, None, q_outs[b],
                                            stream=stream)
            ev_comp[b].record(stream)
            s_out.wait_event(ev_comp[b])
            with torch.cuda.stream(s_out):
                out_host[b].copy_(q_outs[b], non_blocking=True)
                ev_out[b].record(s_out)

    E = max(3, min(K, 50))
    e2e_steps(3)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(s_in)
    stream.wait_event(e0)
    s_out.wait_event(e0)
    e2e_steps(E)
    s_in.wait_stream(stream)
    s_in.wait_stream(s_out)
    e1.record(s_in)
    torch.cuda.synchronize(dev)
    st = B.palquant_sync_check(stream)
    assert st == B.PQ_OK, B.strerror(st)
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / E, world, dev)
    e2e_value = whole_job_rate(ops_step, world, e2e_ms) / 1e12

    if rank != 0:
        return
    pk = peaks()
    fp8_peak = 2.0 * pk["bf16_tflops"]  # dense FP8 = 2x dense BF16 (nominal ratio 4.5 / 2.25)
    step_bytes = c.in_elems * 4 + c.out_elems + c.weight_elems  # fp32 in, codes out, weights
    step_gbs = step_bytes / (t_step / 1e3) / 1e9
    step_tops = ops_step / (t_step / 1e3) / 1e12
    roof_step = {"kernel": "pq_conv_tc_kernel (quantise on load)", "bound": "hbm", "achieved": step_gbs,
                 "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": step_gbs / pk["hbm_gbs"],
                 "traffic": dram_traffic("pq_conv_tc_kernel<quantise-on-load>"), "algorithmic_bytes": step_bytes,
                 "algorithmic_ops": ops_step, "avg_launch_ms": t_step, "tensor_tops": step_tops,
                 "tensor_frac": step_tops / fp8_peak, "peak_source": f"{pk['source']} HBM copy bandwidth"}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K, "warmup": args.warmup,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "e4m3", "dtype_detail": "fp32 activations -> u8 codes, e4m3 x e4m3 -> f32 (exact integer)",
        "data": "synthetic",
        "config": {"workload": WORKLOAD, "global_batch": c.N * world, "per_gpu_batch": c.N,
                   "timed": "one launch per step: quantiser fused into the layer (fp32 NHWC -> next-layer codes); "
                            "independent batches, each launch's loads start while the previous launch finishes; "
                            "the K launches are queued behind a 3 ms spin kernel that precedes the start event",
                   "warmup_steps_run": n_warm,
                   "code_layout": "output codes channel-blocked [N][C/16][H][W][16], one byte per code",
                   "l2": "inputs larger than L2 (205.5 MB fp32, two buffers used in turn)",
                   "parallelism": f"replicas x{world}"},
        "images_per_s": whole_job_rate(c.N, world, ms_per_step),
        "pct_dense_int8_peak": 100.0 * value / world / fp8_peak,
        "roofline": roof_step,
        "roofline_kernels": [roof_step],
        "clocks": clocks,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": int(x_np.nbytes),
                "d2h_bytes_per_step": int(np.prod(out_shape)), "ms_per_step": e2e_ms,
                "timed": "pinned host fp32 -> H2D -> fused step -> D2H of the codes, every step; steps "
                         "pipelined over three streams (copies of neighbouring steps overlap the compute)"},
        "gpu_launches": K,
        "launch_spread": spread,
    }
    line["unfused_step"] = unfused_summary(unfused, c, pk, world)
    line["fp4_step"] = fp4_summary(fp4, c, pk, world)
    if resnet is not None:
        line["resnet18"] = resnet
    if layers is not None:
        line["layers"] = layers
    if not args.no_cpu_baseline and world == 1:
        line["cpu_baseline"] = cpu_baseline(c, x_np, w_np, args.cpu_seconds)
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.profile_layer:
        run_profile_layer(args.profile_layer, args.reps, args.profile_format)
        return
    if args.profile_stem:
        run_profile_stem(args.profile_stem, args.reps)
        return
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    run_ours(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
