#!/usr/bin/env python
"""Decode-step benchmark of the KV-COBRA hot path on GB300.

Workload (default): the Llama-3-8B-shaped compressed cache - 32 layers x 8 KV heads x
head_dim 128, 32 query heads, batch 8 x 32768-token contexts, K and V allocated separately
at 1 bpd (KL weights for K).  One step = append-compress the new token's K and V for every
(layer, kv head, sequence) into the packed cache, then decode attention for one query per
query head across all layers (query projection, rank-space scan over the packed codes,
combine + back-projection).

Reported: effective HBM GB/s over the packed cache (packed bytes a step reads / step time),
the scan kernel's roofline fraction against the measured HBM copy bandwidth, an end-to-end
number through host buffers, and the fp64 oracle timed on the host cores on a bounded
sample.  Under torchrun each rank runs its own replica (weak scaling, no collective on the
data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode-attn effective HBM GB/s over packed cache (% of peak); compress tok/s"
FALLBACK_HBM_GBS = 6800.0
PROFILE = os.path.join(ROOT, "profiles", "decode_scan_llama3_8b.txt")
JOINT70B_PROFILE = os.path.join(ROOT, "profiles", "decode_scan_llama3_70b_joint.txt")
SCAN_SOURCES = ["paper_2609_24298_gb300/csrc/decode.cuh", "paper_2609_24298_gb300/csrc/common.cuh"]
CFG = 2
SAMPLE_R, SAMPLE_B = 64, 2  # (r, b) of the oracle sample heads: the most common point at 1 bpd


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="cobra", choices=["cobra", "reference"])
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="oracle sample budget for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--layers", type=int, default=None, help="fewer layers (profiling runs only)")
    ap.add_argument("--no-compress", action="store_true", help="skip the prefill compress measurement")
    ap.add_argument("--compress-only", action="store_true", help="only the prefill compress measurement")
    ap.add_argument("--compress-layers", type=int, default=None, help="fewer layers (profiling runs only)")
    ap.add_argument("--no-measured", action="store_true", help="skip the measured distortion tables (App. E)")
    ap.add_argument("--k-bpd", type=float, default=None, help="K rate of a K+V split (default: the workload's)")
    ap.add_argument("--v-bpd", type=float, default=None, help="V rate of a K+V split (default: the workload's)")
    ap.add_argument("--v-uniform", action="store_true", help="V by the uniform per-head budget (App. vside)")
    ap.add_argument("--measured-only", action="store_true", help="only the measured distortion tables")
    ap.add_argument("--no-calibration", action="store_true", help="skip the device calibration leg")
    ap.add_argument("--calibration-only", action="store_true", help="only the device calibration leg")
    ap.add_argument("--no-rope", action="store_true", help="skip the RoPE decode leg")
    ap.add_argument("--rope-steps", type=int, default=20, help="timed calls of the RoPE decode leg")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the tiny, Llama-3-70B-shaped joint and ragged-sweep decode legs")
    ap.add_argument("--configs-only", default=None,
                    help="only these of those legs, by their ids in synth.CONFIGS (1 tiny, 3 Llama-3-70B-shaped "
                         "joint, 5 ragged sweep), e.g. 1,3,5")
    ap.add_argument("--config-steps", type=int, default=30,
                    help="timed steps of the Llama-3-70B-shaped and ragged-sweep legs")
    return ap.parse_args()


COMPRESS_PROFILE = os.path.join(ROOT, "profiles", "compress_tc_prefill_4bpd.txt")
COMPRESS_SOURCES = ["paper_2609_24298_gb300/csrc/compress_tc.cuh", "paper_2609_24298_gb300/csrc/compress.cuh",
                    "paper_2609_24298_gb300/csrc/common.cuh"]


def source_hash(sources) -> str:
    h = hashlib.sha256()
    for p in sources:
        with open(os.path.join(ROOT, p), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def scan_source_hash() -> str:
    return source_hash(SCAN_SOURCES)


def profiled_traffic(profile=PROFILE, sources=SCAN_SOURCES):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on the current
    kernel source (else None)."""
    try:
        txt = open(profile).read()
    except OSError:
        return None
    m1 = re.search(r"traffic_bytes_per_launch\s*=\s*([0-9.eE+]+)", txt)
    m2 = re.search(r"kernel_source_sha\s*=\s*([0-9a-f]+)", txt)
    if not m1 or not m2 or m2.group(1) != source_hash(sources):
        return None
    return float(m1.group(1))


def hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def max_over_ranks(x: float, world: int, device) -> float:
    """The largest of every rank's x (the slowest replica sets the time); x itself at N = 1."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_gbs(bytes_per_step: int, steps: int, world: int, max_ms: float) -> float:
    """Whole-job GB/s: every rank reads bytes_per_step per step; the job takes max_ms."""
    return bytes_per_step * steps * world / (max_ms * 1e-3) / 1e9


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,"
              "clocks.mem,temperature.gpu")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def has_sample(self) -> bool:
        """Whether nvidia-smi has written its first reading (its first start can take seconds)."""
        try:
            return self.path is not None and os.path.getsize(self.path) > 0
        except OSError:
            return False

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, mem, temp, reasons = [], [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
            try:
                mem.append(float(parts[9]))
                temp.append(float(parts[10]))
            except (IndexError, ValueError):
                pass
        os.unlink(self.path)
        out = {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(smax) if smax else None,
               "samples": len(sm), "reasons": sorted(reasons)}
        if mem:
            out["mem_mhz"] = float(np.median(mem))
        if temp:
            out["gpu_temp_c"] = float(np.median(temp))
        return out


# ---------------------------------------------------------------------------------------
# fp64 oracle on the host cores (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------------------
class OracleSample:
    """One (sequence, layer, kv head) group of the workload run by the oracle: decode
    attention over T tokens of packed codes plus the append-compress of the new token, with
    K and V at (r, b) = (SAMPLE_R, SAMPLE_B).  Setup (calibration, compressing the context) is
    untimed."""

    def __init__(self, head: int, T: int, group: int):
        from oracle import calibrate as ocal
        from oracle import compress as ocomp
        from paper_2609_24298_gb300 import synth

        spec = synth.CONFIGS[CFG]
        self.params, self.codes, self.new = [], [], []
        for side in (0, 1):
            src = synth.HeadSource(CFG, 0, head, side, spec["alpha"])
            cal = ocal.calibrate_head(src.calibration(512))
            p = ocal.head_params(cal, SAMPLE_R, SAMPLE_B, synth.hadamard_signs(*src.key))
            x = src.tokens(T)
            _, c = ocomp.compress(x[:-1], p["W"], p["mu"], p["delta"], SAMPLE_B)
            self.params.append(p)
            self.codes.append(c)
            self.new.append(x[-1:])
        self.q = synth.decode_queries(CFG, 0, head, 1, group)[0].astype(np.float64)
        self.bytes = 2 * ((T * SAMPLE_R * SAMPLE_B + 7) // 8 + 15) // 16 * 16

    def step(self):
        from oracle import attention as oatt
        from oracle import compress as ocomp

        codes = []
        for side in (0, 1):
            p = self.params[side]
            _, c = ocomp.compress(self.new[side], p["W"], p["mu"], p["delta"], SAMPLE_B)
            codes.append(np.concatenate([self.codes[side], c]))
        return oatt.decode(self.q, codes[0], codes[1], self.params[0], self.params[1])


def oracle_rope_rate(seconds: float, T: int, group: int):
    """Packed bytes per second the oracle's RoPE decode (oracle/rope.py) processes over the
    context of OracleSample groups, timed over about `seconds` of work."""
    from oracle import rope as orope

    samples = [OracleSample(h, T, group) for h in range(2)]
    done, nbytes, t0 = 0, 0, time.perf_counter()
    while True:
        s = samples[done % len(samples)]
        orope.decode(s.q, s.codes[0], s.codes[1], s.params[0], s.params[1], T - 2, ROPE_THETA)
        nbytes += s.bytes
        done += 1
        el = time.perf_counter() - t0
        if el >= seconds and done >= 2:
            break
    return nbytes / el / 1e9, done, el


def oracle_rate(seconds: float, T: int, group: int):
    """Packed bytes per second the oracle processes, timed over about `seconds` of work."""
    samples = [OracleSample(h, T, group) for h in range(2)]
    done, nbytes, t0 = 0, 0, time.perf_counter()
    while True:
        s = samples[done % len(samples)]
        s.step()
        nbytes += s.bytes
        done += 1
        el = time.perf_counter() - t0
        if el >= seconds and done >= 2:
            break
    return nbytes / el / 1e9, done, el


def cores_used():
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        if os.environ.get(k, "").isdigit():
            return int(os.environ[k])
    return os.cpu_count()


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2609_24298_gb300 import synth

    spec = synth.CONFIGS[CFG]
    T, group = spec["tokens"], spec["q_heads"] // spec["kv_heads"]
    sample = OracleSample(0, T, group)
    for _ in range(args.warmup):
        sample.step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        sample.step()
    el = time.perf_counter() - t0
    gbs = sample.bytes * args.steps / el / 1e9
    desc = (f"one (seq, layer, kv-head) group per step: decode over {T} tokens with K and V at r={SAMPLE_R}, "
            f"b={SAMPLE_B} + append-compress of the new token (fp64 numpy); a fixed-allocation sample: at 1 bpd "
            "every head stores r b = 128 bits per token, the same bytes as the allocated heads, whose (r, b) vary")
    out = {"metric": METRIC, "value": gbs, "unit": "GB/s", "n_gpus": args.gpus, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
           "config": workload_config(spec),
           "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": cores_used(), "kind": "oracle", "sample": desc},
           "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def workload_config(spec):
    return {"workload": "llama3-8b-shaped decode step: 32 layers x 8 kv heads (GQA 4, head_dim 128) x batch 8 x "
                        "32768-token context, K and V at 1 bpd",
            "layers": spec["layers"], "kv_heads": spec["kv_heads"], "q_heads": spec["q_heads"],
            "batch": spec["seqs"], "context": spec["tokens"], "bpd": spec["bpd"],
            "step": "append K+V of 1 token per (layer, kv head, seq) + decode attention for all layers",
            "l2": "inputs larger than L2 (packed cache of about 2 GiB re-read every step)"}


def split_config(args):
    """The K+V split of a non-default run (Sec. 5 "Joint K+V compression", App. vside)."""
    if args.k_bpd is None and args.v_bpd is None and not args.v_uniform:
        return {}
    return {"workload": "llama3-8b-shaped decode step with a K+V rate split", "k_bpd": args.k_bpd,
            "v_bpd": args.v_bpd, "v_allocation": "uniform per head" if args.v_uniform else "damped"}


# ---------------------------------------------------------------------------------------
# prefill compress (the tensor-core projection path)
# ---------------------------------------------------------------------------------------
COMPRESS_CFG = 4


def run_compress_leg(args, dev, stream, peak):
    """Compress every token of the prefill workload - 32 layers x 8 kv heads x batch 64 x 4096
    tokens of bf16 K and V at 4 bpd - from inputs resident in HBM (about 34 GB, far larger
    than L2), one cobra_compress launch per side covering all layers.  Returns the JSON
    object reported under "compress"."""
    import torch

    from paper_2609_24298_gb300 import cobra, pipeline, synth

    spec = synth.CONFIGS[COMPRESS_CFG]
    L, H, S, T = spec["layers"], spec["kv_heads"], spec["seqs"], spec["tokens"]
    if args.compress_layers:
        L = args.compress_layers
    hp, srcs = pipeline.build_params(COMPRESS_CFG, L, spec["bpd"], joint=False)
    rows = -(-T // 128)
    dp = pipeline.DeviceParams(hp, S * rows, device=dev)
    xs = []
    for side in (0, 1):
        x = torch.empty((L, S, T, H, 128), dtype=torch.bfloat16, device=dev)
        for l in range(L):
            x[l] = pipeline.device_tokens([srcs[side * L * H + l * H + h] for h in range(H)], S, T,
                                          seed=COMPRESS_CFG * 1000003 + 2 * l + side, device=dev)
        xs.append(x)
    descs = [cobra.compress_desc(head0=side * L * H, layer_stride=H, n_layers=L, n_kv_heads=H, side=side, n_seqs=S,
                                 rows_per_seq=rows, x_stride_layer=S * T * H * 128, x_stride_seq=T * H * 128,
                                 x_stride_tok=H * 128, x_stride_head=128) for side in (0, 1)]

    def one_pass():
        for side in (0, 1):
            cobra.cobra_compress(dp.block, descs[side], xs[side], 0, T, dp.cache, None, stream)

    # the clock sampler's first reading can take seconds: it starts with the warm-up, which keeps
    # the GPU busy until that reading is in (at most 10 s), so its samples are all under load
    clocks = ClockSampler(torch.device(dev).index or 0)
    clocks.start()
    t_start = time.time()
    n_warm = 0
    while n_warm < 3 or (time.time() - t_start < 10.0 and (time.time() - t_start < 1.0 or not clocks.has_sample())):
        one_pass()
        torch.cuda.synchronize()
        n_warm += 1
    if cobra.cobra_check(stream) != cobra.COBRA_OK:
        clocks.stop()
        raise RuntimeError("device status after compress warm-up")
    K = max(5, min(50, args.steps // 40))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(K):
        one_pass()
    e1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if cobra.cobra_check(stream) != cobra.COBRA_OK:
        raise RuntimeError("device status after the compress timed region")
    ms = e0.elapsed_time(e1) / K
    traffic = profiled_traffic(COMPRESS_PROFILE, COMPRESS_SOURCES)
    in_bytes = 2 * L * S * T * H * 128 * 2
    out_bytes = int(sum(16 * int(r) * int(b) for r, b in zip(hp.r, hp.b) if r > 0)) * S * rows
    flops = 2 * 128 * int(sum(int(r) for r in hp.r)) * S * T  # algorithmic y = W^T x per token-head
    gbs = (in_bytes + out_bytes) / (ms * 1e-3) / 1e9
    tokens = S * T
    del xs
    return {
        "metric": "compress tok/s", "value": tokens / (ms * 1e-3), "unit": "tok/s",
        "workload": f"prefill compress: {L} layers x {H} kv heads x batch {S} x {T} tokens of bf16 K and V "
                    f"(head_dim 128) at {spec['bpd']:g} bpd, inputs resident in HBM",
        "tokens_per_pass": tokens, "head_tokens_per_s": tokens * L * H * 2 / (ms * 1e-3), "ms_per_pass": ms,
        "passes": K, "launches": 2 * K, "gbs": gbs,
        "roofline": {"bound": "hbm", "kernel": "compress_tc_kernel", "achieved": gbs, "peak": peak, "unit": "GB/s",
                     "frac": gbs / peak, "algorithmic_bytes_per_pass": in_bytes + out_bytes,
                     "traffic_per_launch": traffic if L == 32 else None,
                     "tensor_tflops_algorithmic": flops / (ms * 1e-3) / 1e12},
        "l2": f"inputs larger than L2 ({in_bytes / 1e9:.1f} GB of bf16 K/V read every pass)",
        "clocks": clk,
    }


MEASURE_PROFILE = os.path.join(ROOT, "profiles", "measure_tables_llama3_8b.txt")
MEASURE_SOURCES = ["paper_2609_24298_gb300/csrc/measure.cuh", "paper_2609_24298_gb300/csrc/common.cuh"]
ISSUE_PEAK = 152 * 4 * 2.07e9  # warp-instructions per second: 152 SMs x 4 schedulers at 2070 MHz


def profiled_instructions(profile=MEASURE_PROFILE, sources=MEASURE_SOURCES):
    """Warp-instructions per call from a committed ncu summary taken on the current source."""
    try:
        txt = open(profile).read()
    except OSError:
        return None
    m1 = re.search(r"warp_instructions_per_call\s*=\s*([0-9.eE+]+)", txt)
    m2 = re.search(r"kernel_source_sha\s*=\s*([0-9a-f]+)", txt)
    if not m1 or not m2 or m2.group(1) != source_hash(sources):
        return None
    return float(m1.group(1))


CALIB_PROFILE = os.path.join(ROOT, "profiles", "calibrate_heads_llama3_8b.txt")
CALIB_SOURCES = ["paper_2609_24298_gb300/csrc/calib.cuh", "paper_2609_24298_gb300/csrc/common.cuh"]
FP64_NOMINAL_TFLOPS = 1.25  # GB300's fp64 rate (nominal; no measured figure on this machine)


def profiled_value(key, profile, sources):
    """A per-call figure from a committed ncu summary taken on the current source."""
    try:
        txt = open(profile).read()
    except OSError:
        return None
    m1 = re.search(key + r"\s*=\s*([0-9.eE+]+)", txt)
    m2 = re.search(r"kernel_source_sha\s*=\s*([0-9a-f]+)", txt)
    if not m1 or not m2 or m2.group(1) != source_hash(sources):
        return None
    return float(m1.group(1))


def run_calibration_leg(args, dev, stream, srcs, cpu_baseline: bool):
    """Table alg:kvrobin steps 1-2 for the decode workload's model on the device: 512 heads x
    512 calibration vectors (the 256 K heads with their groups' 2048 calibration queries,
    attention-KL weights; the 256 V heads with MSE weights), two cobra_calibrate_heads calls.
    Returns the JSON object reported under "calibration"."""
    import torch

    from paper_2609_24298_gb300 import cobra, pipeline, synth

    spec = synth.CONFIGS[CFG]
    G = spec["q_heads"] // spec["kv_heads"]
    xs = [s.calibration(512) for s in srcs]
    qs = [synth.calibration_queries(CFG, s.key[1], s.key[2], G, 512, spec["alpha"]) if s.key[3] == 0 else None
          for s in srcs]
    calls = []
    for kl in (True, False):
        idx = [i for i, q in enumerate(qs) if (q is not None) == kl]
        x = torch.tensor(np.stack([np.asarray(xs[i], np.float32) for i in idx]), device=dev).contiguous()
        q = torch.tensor(np.stack([np.asarray(qs[i], np.float32).reshape(-1, 128) for i in idx]),
                         device=dev).contiguous() if kl else None
        outs = [torch.empty((len(idx), n), dtype=torch.float64, device=dev) for n in (128, 128, 128 * 128, 128)]
        calls.append((x, q, outs))

    def call():
        for x, q, (mu, lam, U, w) in calls:
            cobra.cobra_calibrate_heads(x, q, mu, lam, U, w, stream)

    call()
    torch.cuda.synchronize()
    K = 3
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(K):
        call()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / K
    t0 = time.time()
    pipeline.calibrate_heads(xs, qs)
    host_ms = (time.time() - t0) * 1e3
    flops = profiled_value("fp64_flops_per_call", CALIB_PROFILE, CALIB_SOURCES)
    out = {
        "metric": "calibration steps 1-2 (covariance, eigen-decomposition, KL weights and order)", "value": ms,
        "unit": "ms for all heads", "higher_is_better": False,
        "workload": f"{len(srcs)} heads (32 layers x 8 kv heads x K/V) x 512 calibration vectors; K heads with "
                    f"{G * 512} calibration queries each",
        "calls": K, "launches": 2 * K,
        "host_library_ms": host_ms, "host_library_threads": pipeline._threads(),
        "roofline": {"bound": "fp64", "kernel": "calib_kernel", "unit": "TFLOP/s", "peak": FP64_NOMINAL_TFLOPS,
                     "peak_kind": "nominal", "fp64_flops_per_call": flops,
                     "achieved": flops / (ms * 1e-3) / 1e12 if flops else None,
                     "frac": flops / (ms * 1e-3) / 1e12 / FP64_NOMINAL_TFLOPS if flops else None},
    }
    if cpu_baseline:
        from oracle import calibrate as ocal

        t0 = time.time()
        ocal.calibrate_head(np.asarray(xs[0], np.float64), qs[0])
        el = time.time() - t0
        out["cpu_baseline"] = {"value": el * len(srcs) * 1e3, "unit": "ms for all heads", "cores": cores_used(),
                               "kind": "oracle", "sample": f"one K head ({el * 1e3:.1f} ms of fp64 numpy), "
                                                          f"extrapolated to {len(srcs)} heads"}
    del calls
    return out


def run_measured_leg(args, dev, stream, cals, srcs, cpu_baseline: bool):
    """App. E's measured distortion tables for every (layer, kv head, side) of the decode
    workload's model: 512 heads x 512 calibration tokens through the deployed quantizer at
    every candidate (r, b) of the allocator's grid (65 ranks x 8 widths), one
    cobra_measure_distortion call.  Returns the JSON object reported under "measured"."""
    import torch

    from paper_2609_24298_gb300 import cobra, synth

    n = len(cals)
    xs = np.stack([s.calibration(512) for s in srcs]).astype(np.float32)
    f32 = lambda a: torch.tensor(np.asarray(a, np.float32), device=dev).contiguous()
    x = f32(xs)
    U = f32(np.stack([c["U"].T.reshape(-1) for c in cals]))
    lam = torch.tensor(np.stack([c["lam"] for c in cals]), dtype=torch.float64, device=dev).contiguous()
    w = torch.tensor(np.stack([c["w"] for c in cals]), dtype=torch.float64, device=dev).contiguous()
    mu = f32(np.stack([c["mu"] for c in cals]))
    signs = torch.tensor(np.stack([synth.hadamard_signs(*s.key) for s in srcs]), dtype=torch.int8,
                         device=dev).contiguous()
    rg, bg = list(range(0, 129, 2)), list(range(1, 9))
    coords = torch.empty((n, 512, 128), dtype=torch.float32, device=dev)
    D = torch.empty((n, len(rg), len(bg)), dtype=torch.float64, device=dev)

    def call():
        cobra.cobra_measure_distortion(x, U, lam, w, mu, signs, rg, bg, coords, D, stream)

    for _ in range(2):
        call()
    torch.cuda.synchronize()
    K = 5
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(K):
        call()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / K
    evals = n * len(rg) * len(bg) * 512  # (head, r, b, calibration token) evaluations
    out = {
        "metric": "measured distortion tables (App. E)", "value": ms, "unit": "ms per table set",
        "higher_is_better": False,
        "workload": f"{n} heads (32 layers x 8 kv heads x K/V) x 512 calibration tokens x {len(rg)} ranks x "
                    f"{len(bg)} bit widths, inputs resident on the device",
        "evaluations_per_s": evals / (ms * 1e-3), "calls": K, "launches": 2 * K,
    }
    instr = profiled_instructions()
    out["roofline"] = {"bound": "issue", "kernel": "coords_kernel + measure_kernel", "unit": "warp-instr/s",
                       "peak": ISSUE_PEAK, "warp_instructions_per_call": instr,
                       "achieved": instr / (ms * 1e-3) if instr else None,
                       "frac": instr / (ms * 1e-3) / ISSUE_PEAK if instr else None}
    if cpu_baseline:
        # the oracle's fp64 tables for one head over the same grid, extrapolated to all heads
        from oracle import calibrate as ocal
        from oracle import measured as omeas

        cal = ocal.calibrate_head(xs[0].astype(np.float64))
        t0 = time.time()
        omeas.measured_table(xs[0].astype(np.float64), cal, np.ones(128), synth.hadamard_signs(*srcs[0].key), rg, bg)
        el = time.time() - t0
        out["cpu_baseline"] = {"value": el * n * 1e3, "unit": "ms per table set", "cores": cores_used(),
                               "kind": "oracle", "sample": f"one head's full table ({el:.1f} s of fp64 numpy), "
                                                          f"extrapolated to {n} heads"}
    del x, U, lam, w, mu, signs, coords, D
    return out


# ---------------------------------------------------------------------------------------
# the CUDA path
# ---------------------------------------------------------------------------------------
ROPE_THETA = 500000.0  # Llama-3-8B's rotary base
ROPE_SOURCES = ["paper_2609_24298_gb300/csrc/rope.cuh", "paper_2609_24298_gb300/csrc/decode.cuh",
                "paper_2609_24298_gb300/csrc/common.cuh"]
ROPE_PROFILE = os.path.join(ROOT, "profiles", "rope_decode_llama3_8b.txt")


def bf16_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except (OSError, KeyError, ValueError):
        return 1900.0, "fallback"


def run_rope_leg(args, dev, stream, hp, wl, desc, ws, info, q, lens, out, cpu_baseline: bool):
    """Decode attention for a model with the rotary embedding (K compressed before it, Sec. 5
    "Scope"): the same compressed cache, plan and queries as the main step, each key rebuilt,
    turned to its position and scored (cobra_decode_rope_attn, three launches).  The rebuild is
    a dense contraction, so the leg is measured against the tensor roofline: algorithmic
    FLOPs per call = sum over (seq, layer, kv head) of T (2 d r_K + 2 d G + 2 r_V G).
    Returns the JSON object reported under "rope"."""
    import torch

    from paper_2609_24298_gb300 import cobra, pipeline

    L, H, S, G = wl.layers, wl.kv, wl.seqs, wl.group
    T = int(np.max(wl.tokens))
    cpu = None
    if cpu_baseline:
        gbs, n, el = oracle_rope_rate(min(args.cpu_seconds, 10.0), T, G)
        cpu = {"value": gbs, "unit": "GB/s", "cores": cores_used(), "kind": "oracle",
               "sample": f"{n} (seq, layer, kv-head) RoPE decodes over {T - 1} tokens with K and V at "
                         f"r={SAMPLE_R}, b={SAMPLE_B} ({el:.1f} s of fp64 numpy)"}
    tb = cobra.cobra_rope_table_bytes(T)
    table = torch.empty(tb // 4, dtype=torch.float32, device=dev)
    cobra.cobra_rope_table(ROPE_THETA, T, table, tb, stream)
    nws = ws.numel()

    def call():
        cobra.cobra_decode_rope_attn(wl.dev.block, desc, info, q, None, table, T, wl.dev.cache, lens, None, out, ws,
                                     nws, stream)

    for _ in range(3):
        call()
    torch.cuda.synchronize()
    if cobra.cobra_check(stream) != cobra.COBRA_OK:
        raise RuntimeError("device status after the RoPE warm-up")
    K = max(3, args.rope_steps)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(K):
        call()
    e1.record(stream)
    torch.cuda.synchronize()
    if cobra.cobra_check(stream) != cobra.COBRA_OK:
        raise RuntimeError("device status after the RoPE timed region")
    ms = e0.elapsed_time(e1) / K
    n = L * H
    rk = np.asarray(hp.r[:n], np.float64)
    rv = np.asarray(hp.r[n:2 * n], np.float64)
    flops = float(S * T * np.sum(2 * 128 * rk + 2 * 128 * G + 2 * rv * G))
    bytes_call = pipeline.packed_bytes_read(wl)
    peak, kind = bf16_peak()
    achieved = flops / (ms * 1e-3) / 1e12
    return {"metric": "packed KV bytes decoded per second with RoPE", "value": bytes_call / (ms * 1e-3) / 1e9,
            "unit": "GB/s", "ms_per_call": ms, "calls": K, "theta": ROPE_THETA,
            "workload": f"the main step's cache and queries: {L} layers x {H} kv heads x {S} seqs x {T} tokens, "
                        "query at position T - 1",
            "roofline": {"bound": "tensor", "kernel": "rope_scan_kernel (timed with its query rotation and "
                                                      "combine launches)",
                         "achieved": achieved, "peak": peak, "peak_kind": kind + " bf16 burst", "unit": "TFLOP/s",
                         "frac": achieved / peak, "algorithmic_flops_per_call": flops,
                         "traffic": profiled_value("traffic_bytes_per_launch", ROPE_PROFILE, ROPE_SOURCES)},
            "cpu_baseline": cpu,
            "gpu_launches": 3 * K}


# ---------------------------------------------------------------------------------------
# the other decode workloads (tiny, Llama-3-70B-shaped joint, ragged sweep), measured after the headline
# ---------------------------------------------------------------------------------------
def allocated_params(cfg: int, layers: int, bpd: float, base=None):
    """Per-head parameters of a config at `bpd`: calibration (reused from `base` when given:
    the rate sweep re-allocates the same calibrated heads) and the library's allocation."""
    from paper_2609_24298_gb300 import cobra, pipeline, synth

    spec = synth.CONFIGS[cfg]
    if base is None:
        return pipeline.build_params(cfg, layers, bpd, joint=spec["joint"])
    hp0, srcs = base
    w = hp0.alloc["w"]
    if spec["joint"]:
        res = cobra.cobra_allocate(w, bpd)
        r, b = res["r"], res["b"]
    else:
        n = len(w) // 2
        rk, rv = cobra.cobra_allocate(w[:n], bpd), cobra.cobra_allocate(w[n:], bpd)
        r, b = np.concatenate([rk["r"], rv["r"]]), np.concatenate([rk["b"], rv["b"]])
    hp = pipeline.fuse_heads(hp0.cals, r, b, [synth.hadamard_signs(*x.key) for x in srcs])
    hp.cals, hp.alloc = hp0.cals, hp0.alloc
    return hp, srcs


class StepWorkload:
    """A decode workload on the device: the cache filled by cobra_compress with T - 1 tokens per
    sequence, the plan, and the inputs of one decode step (append of the new K and V token at
    position T - 1, query projection, scan, combine; cobra_decode_step)."""

    def __init__(self, dev, cfg: int, layers: int, hp, srcs, lens, paged: bool, seed: int):
        import torch

        from paper_2609_24298_gb300 import cobra, pipeline, synth

        spec = synth.CONFIGS[cfg]
        H = spec["kv_heads"]
        G = spec["q_heads"] // H
        L, S = layers, len(lens)
        lens = np.asarray(lens, np.int64)
        rows = int(-(-lens.max() // 128))
        wl = pipeline.Workload(cfg=cfg, layers=L, kv=H, group=G, seqs=S, tokens=lens - 1, bpd=0.0, joint=False)
        if paged:
            pps = -(-rows // 2)
            wl.pages_per_seq = pps
            wl.page_table = torch.tensor(synth.shuffled_pages(cfg, S * pps), dtype=torch.int32, device=dev)
            n_slots = 2 * S * pps
        else:
            wl.rows_per_seq = rows
            n_slots = S * rows
        wl.dev = pipeline.DeviceParams(hp, n_slots, device=dev)
        pipeline.fill_cache(wl, srcs, device=dev)
        wl.tokens = lens
        self.desc, self.ws, self.info = pipeline.decode_setup(wl, device=dev)
        gen = torch.Generator(device=dev)
        gen.manual_seed(seed)
        self.xk = torch.randn((L, S, H, 128), generator=gen, device=dev).to(torch.bfloat16)
        self.xv = torch.randn((L, S, H, 128), generator=gen, device=dev).to(torch.bfloat16)
        self.q = torch.randn((L, S, H * G, 128), generator=gen, device=dev).to(torch.bfloat16)
        self.out = torch.empty((L, S, H * G, 128), dtype=torch.float32, device=dev)
        self.pos = torch.tensor(lens - 1, dtype=torch.int32, device=dev)
        self.lens = torch.tensor(lens, dtype=torch.int32, device=dev)
        self.adesc = [cobra.compress_desc(head0=side * L * H, layer_stride=H, n_layers=L, n_kv_heads=H, side=side,
                                          n_seqs=S, rows_per_seq=wl.rows_per_seq, pages_per_seq=wl.pages_per_seq,
                                          x_stride_layer=S * H * 128, x_stride_seq=H * 128, x_stride_tok=0,
                                          x_stride_head=128) for side in (0, 1)]
        self.wl, self.hp, self.G = wl, hp, G
        self.bytes = pipeline.packed_bytes_read(wl)

    def step(self, stream):
        from paper_2609_24298_gb300 import cobra

        wl = self.wl
        cobra.cobra_decode_step(wl.dev.block, self.desc, self.info, self.adesc[0], self.adesc[1], self.xk, self.xv,
                                self.pos, self.q, wl.dev.cache, self.lens, wl.page_table, self.out, self.ws,
                                self.ws.numel(), stream)

    def scan(self, stream):
        from paper_2609_24298_gb300 import cobra

        wl = self.wl
        cobra.cobra_decode_scan(wl.dev.block, self.desc, self.info, wl.dev.cache, self.lens, wl.page_table, self.ws,
                                self.ws.numel(), stream)

    def timed(self, stream, steps: int, warmup: int):
        """(ms per step, ms per scan): K steps with events at the two ends only, then the scan
        alone between events (the q~ blocks of the last step stay in the workspace)."""
        import torch

        from paper_2609_24298_gb300 import cobra

        for _ in range(warmup):
            self.step(stream)
        torch.cuda.synchronize()
        if cobra.cobra_check(stream) != cobra.COBRA_OK:
            raise RuntimeError("device status after warm-up")
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        ev[0].record(stream)
        for _ in range(steps):
            self.step(stream)
        ev[1].record(stream)
        ev[2].record(stream)
        for _ in range(steps):
            self.scan(stream)
        ev[3].record(stream)
        torch.cuda.synchronize()
        if cobra.cobra_check(stream) != cobra.COBRA_OK:
            raise RuntimeError("device status after the timed steps")
        return ev[0].elapsed_time(ev[1]) / steps, ev[2].elapsed_time(ev[3]) / steps

    def release(self):
        del self.wl, self.ws, self.xk, self.xv, self.q, self.out


def oracle_group_rate(hp, srcs, cfg: int, layers: int, T: int, G: int, seconds: float):
    """The fp64 oracle's decode of one (layer 0, kv head 0) group of a leg's workload over T
    tokens, with that group's allocated (r, b) (compressing its context is setup, not timed),
    repeated for about `seconds`.  Returns (GB/s of packed codes, groups done, seconds)."""
    from oracle import attention as oatt
    from oracle import compress as ocomp
    from paper_2609_24298_gb300 import synth

    spec = synth.CONFIGS[cfg]
    H = spec["kv_heads"]
    n = layers * H
    ps, codes, nbytes = [], [], 0
    for idx in (0, n):  # K and V head of (layer 0, kv head 0)
        r, b = int(hp.r[idx]), int(hp.b[idx]) if hp.r[idx] else 1
        p = {"r": r, "b": b, "W": np.asarray(hp.W[idx], np.float32), "delta": np.float32(hp.delta[idx]),
             "mu": np.asarray(hp.mu[idx], np.float32)}
        if r:
            _, c = ocomp.compress(srcs[idx].tokens(T), p["W"], p["mu"], p["delta"], b)
        else:
            c = np.zeros((T, 0), np.int64)
        ps.append(p)
        codes.append(c)
        nbytes += ((T * r * (b if r else 0) + 7) // 8 + 15) // 16 * 16
    q = synth.decode_queries(cfg, 0, 0, 1, G)[0].astype(np.float64)
    done, t0 = 0, time.perf_counter()
    while True:
        oatt.decode(q, codes[0], codes[1], ps[0], ps[1])
        done += 1
        el = time.perf_counter() - t0
        if el >= seconds and done >= 1:
            break
    return nbytes * done / el / 1e9, done, el


def workload_leg(args, dev, stream, cfg: int, bpd: float, lens, paged: bool, steps: int, cpu_baseline: bool,
                 base=None, label: str = ""):
    """One decode workload measured like the headline (cobra_decode_step, events at the ends of
    the timed steps; the scan alone for its roofline).  Returns (JSON object, (hp, srcs))."""
    from paper_2609_24298_gb300 import synth

    spec = synth.CONFIGS[cfg]
    H = spec["kv_heads"]
    G = spec["q_heads"] // H
    L = spec["layers"]
    hp, srcs = allocated_params(cfg, L, bpd, base)
    wlk = StepWorkload(dev, cfg, L, hp, srcs, lens, paged, seed=cfg * 7919 + int(bpd * 8))
    ms, scan_ms = wlk.timed(stream, steps, args.warmup)
    peak, kind = hbm_peak()
    achieved = wlk.bytes / (scan_ms * 1e-3) / 1e9
    out = {"workload": label, "bpd": bpd, "value": wlk.bytes / (ms * 1e-3) / 1e9, "unit": "GB/s",
           "ms_per_step": ms, "steps": steps, "packed_bytes_per_step": wlk.bytes,
           "roofline": {"bound": "hbm", "kernel": "decode_kernel (rank-space scan)", "achieved": achieved,
                        "peak": peak, "peak_kind": kind, "unit": "GB/s", "frac": achieved / peak,
                        "scan_ms": scan_ms},
           "gpu_launches": 3 * steps + steps}  # the timed steps (3 launches each) and scans
    wlk.release()
    if cpu_baseline:
        gbs, n, el = oracle_group_rate(hp, srcs, cfg, L, int(np.asarray(lens)[0]), G, args.cpu_seconds / 3)
        out["cpu_baseline"] = {"value": gbs, "unit": "GB/s", "cores": cores_used(), "kind": "oracle",
                               "sample": f"{n} decode(s) of one (layer 0, kv head 0) group over "
                                         f"{int(np.asarray(lens)[0])} tokens with its allocated (r_K, b_K) = "
                                         f"({int(hp.r[0])}, {int(hp.b[0])}), (r_V, b_V) = "
                                         f"({int(hp.r[L * H])}, {int(hp.b[L * H])}) ({el:.1f} s of fp64 numpy)"}
    return out, (hp, srcs)


def run_llama3_70b_joint_leg(args, dev, stream, cpu_baseline: bool):
    """Llama-3-70B-shaped joint K+V at 0.5 bpd: 80 layers x 8 kv heads, GQA 8, one 131072-token
    sequence; the step appends the new token and decodes over all layers."""
    from paper_2609_24298_gb300 import synth

    spec = synth.CONFIGS[3]
    out, _ = workload_leg(args, dev, stream, 3, spec["bpd"], [spec["tokens"]], False, args.config_steps,
                          cpu_baseline, label="llama3-70b-shaped decode step: 80 layers x 8 kv heads (GQA 8) x 1 "
                                              "sequence x 131072 tokens, K and V allocated jointly at 0.5 bpd")
    out["roofline"]["traffic"] = profiled_traffic(JOINT70B_PROFILE, SCAN_SOURCES)
    return out


def run_ragged_sweep_leg(args, dev, stream, cpu_baseline: bool):
    """Ragged paged rate sweep: 32 layers x 8 kv heads x 32 sequences of lengths uniform in
    [1024, 65536] in 256-token pages (shuffled), every bpd point re-allocated."""
    from paper_2609_24298_gb300 import synth

    spec = synth.CONFIGS[5]
    lens = synth.ragged_lengths(5, spec["seqs"], *spec["tokens"])
    points, base = [], None
    for i, bpd in enumerate(spec["bpd"]):
        o, base = workload_leg(args, dev, stream, 5, bpd, lens, True, args.config_steps, cpu_baseline and i == 1,
                               base=base, label=f"ragged paged sweep point: 32 layers x 8 kv heads x 32 sequences "
                                                f"(lengths in [1024, 65536], sum {int(lens.sum())}), 256-token "
                                                f"pages, K and V at {bpd} bpd")
        points.append(o)
    return {"workload": "ragged paged rate sweep: 32 layers x 8 kv heads x 32 sequences of 1024-65536 tokens, "
                        "256-token pages, 0.5 to 4 bpd", "points": points}


def run_tiny_leg(args, dev, stream, cpu_baseline: bool):
    """The tiny single-layer case: 8 kv heads, GQA 4, one 2048-token sequence at 2 bpd; the
    decode step's latency."""
    from paper_2609_24298_gb300 import synth

    spec = synth.CONFIGS[1]
    out, _ = workload_leg(args, dev, stream, 1, spec["bpd"], [spec["tokens"]], False, 200, cpu_baseline,
                          label="tiny decode step: 1 layer x 8 kv heads (GQA 4) x 1 sequence x 2048 tokens, "
                                "K and V at 2 bpd")
    out["latency_us"] = out["ms_per_step"] * 1e3
    out["note"] = "latency-bound: the packed bytes (1 MB) fit L2 and the step is three short launches"
    return out


class AuxLegs:
    """Runs the legs measured after the headline.  A leg that fails is reported in its place as
    {"error": ...}.  After a device-side failure (a CUDA error, or a library status of
    COBRA_ECUDA / COBRA_ETIMEOUT, which can leave the context unusable) the remaining GPU legs are
    not run on that context: each reports {"error": "skipped after ..."} naming the first cause.
    Every leg ends with a synchronisation and a status check, so a failure is charged to the leg
    that caused it."""

    def __init__(self, stream):
        self.stream = stream
        self.device_error = None

    def _is_device_error(self, e) -> bool:
        from paper_2609_24298_gb300 import cobra

        if isinstance(e, cobra.CobraError):
            return e.status in (cobra.COBRA_ECUDA, cobra.COBRA_ETIMEOUT)
        msg = str(e)
        return "CUDA" in msg or "cuda" in msg or "device-side" in msg

    def run(self, fn, *a):
        import torch

        from paper_2609_24298_gb300 import cobra

        if self.device_error:
            return {"error": f"skipped after {self.device_error}"[:400]}
        try:
            res = fn(*a)
            torch.cuda.synchronize()
            st = cobra.cobra_check(self.stream)
            if st != cobra.COBRA_OK:
                raise cobra.CobraError("cobra_check after " + fn.__name__, st)
            return res
        except Exception as e:  # the headline line is printed either way
            msg = f"{fn.__name__}: {type(e).__name__}: {e}"[:400]
            if self._is_device_error(e):
                self.device_error = msg
            return {"error": msg}


def run_cobra(args):
    import torch
    import torch.distributed as dist

    from paper_2609_24298_gb300 import cobra, pipeline, synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    spec = synth.CONFIGS[CFG]
    L, H, S, T = spec["layers"], spec["kv_heads"], spec["seqs"], spec["tokens"]
    if args.layers:
        L = args.layers
    G = spec["q_heads"] // H
    Hq = H * G
    cobra.lib()
    if args.compress_only:
        print(json.dumps(run_compress_leg(args, dev, torch.cuda.current_stream(), hbm_peak()[0])), flush=True)
        return
    if args.calibration_only:
        srcs = [synth.HeadSource(CFG, l, h, side, spec["alpha"]) for side in (0, 1) for l in range(L) for h in range(H)]
        print(json.dumps(run_calibration_leg(args, dev, torch.cuda.current_stream(), srcs,
                                             not args.no_cpu_baseline)), flush=True)
        return
    if args.configs_only:
        legs = AuxLegs(torch.cuda.current_stream())
        st, cb = torch.cuda.current_stream(), not args.no_cpu_baseline
        todo = {int(x) for x in args.configs_only.split(",")}
        fns = {1: ("tiny_2bpd", run_tiny_leg), 3: ("llama3_70b_joint_0p5bpd", run_llama3_70b_joint_leg),
               5: ("ragged_paged_sweep", run_ragged_sweep_leg)}
        print(json.dumps({name: legs.run(fn, args, dev, st, cb) for c, (name, fn) in fns.items() if c in todo}),
              flush=True)
        return
    if args.measured_only:
        hp, srcs = pipeline.build_params(CFG, L, spec["bpd"], joint=False)
        print(json.dumps(run_measured_leg(args, dev, torch.cuda.current_stream(), hp.cals, srcs,
                                          not args.no_cpu_baseline)), flush=True)
        return

    # cpu baseline first, before any GPU work (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        gbs, n, el = oracle_rate(args.cpu_seconds, T, G)
        cpu = {"value": gbs, "unit": "GB/s", "cores": cores_used(), "kind": "oracle",
               "sample": f"{n} (seq, layer, kv-head) decode steps over {T} tokens with K and V at r={SAMPLE_R}, "
                         f"b={SAMPLE_B} incl. append-compress ({el:.1f} s of fp64 numpy); a fixed-allocation sample: at "
                         "1 bpd every head stores r b = 128 bits per token, the same bytes as the allocated heads, "
                         "whose (r, b) vary"}

    k_bpd = args.k_bpd if args.k_bpd is not None else spec["bpd"]
    v_opts = cobra.alloc_opts(mode=cobra.ALLOC_UNIFORM) if args.v_uniform else None
    hp, srcs = pipeline.build_params(CFG, L, k_bpd, joint=False, v_bpd=args.v_bpd, v_opts=v_opts)
    rows = -(-T // 128)
    wl = pipeline.Workload(cfg=CFG, layers=L, kv=H, group=G, seqs=S, tokens=np.full(S, T - 1, np.int64),
                           bpd=spec["bpd"], joint=False, rows_per_seq=rows)
    wl.dev = pipeline.DeviceParams(hp, S * rows, device=dev)
    pipeline.fill_cache(wl, srcs, device=dev)
    wl.tokens = np.full(S, T, np.int64)
    desc, ws, info = pipeline.decode_setup(wl, device=dev)
    nbytes_ws = ws.numel()
    stream = torch.cuda.current_stream()

    # per-step inputs: the new token's K and V for every (layer, kv head, seq); the queries
    gen = torch.Generator(device=dev)
    gen.manual_seed(2609 + rank)
    # the step's inputs (new K and V tokens, queries) in one device buffer, so that the
    # end-to-end leg moves them with one host-to-device copy
    n_kv, n_q = L * S * H * 128, L * S * Hq * 128
    din = torch.empty(2 * n_kv + n_q, dtype=torch.bfloat16, device=dev)
    xk, xv, q = (din[:n_kv].view(L, S, H, 128), din[n_kv:2 * n_kv].view(L, S, H, 128),
                 din[2 * n_kv:].view(L, S, Hq, 128))
    xk.copy_(torch.randn((L, S, H, 128), generator=gen, device=dev))
    xv.copy_(torch.randn((L, S, H, 128), generator=gen, device=dev))
    q.copy_(torch.randn((L, S, Hq, 128), generator=gen, device=dev))
    out = torch.empty((L, S, Hq, 128), dtype=torch.float32, device=dev)
    pos = torch.full((S,), T - 1, dtype=torch.int32, device=dev)
    lens = torch.full((S,), T, dtype=torch.int32, device=dev)
    adesc = [cobra.compress_desc(head0=side * L * H, layer_stride=H, n_layers=L, n_kv_heads=H, side=side, n_seqs=S,
                                 rows_per_seq=rows, x_stride_layer=S * H * 128, x_stride_seq=H * 128, x_stride_tok=0,
                                 x_stride_head=128) for side in (0, 1)]
    block, cache = wl.dev.block, wl.dev.cache

    stages = ("append_v", "qproj_append_k", "scan", "combine")

    def step():
        # one decode step through the public entry point: the query projection fused with the K
        # and V appends (one launch), scan, combine
        cobra.cobra_decode_step(block, desc, info, adesc[0], adesc[1], xk, xv, pos, q, cache, lens, None, out, ws,
                                nbytes_ws, stream)

    def staged_step(ev):
        # the step's work as separate calls, with events between them (they serialise the
        # launches, so this pass only gives the per-stage breakdown; the V append is its own
        # launch here)
        ev[0].record(stream)
        cobra.cobra_append(block, adesc[1], xv, pos, cache, None, stream)
        ev[1].record(stream)
        cobra.cobra_decode_qproj_append(block, desc, info, q, adesc[0], xk, pos, cache, None, ws, nbytes_ws, stream)
        ev[2].record(stream)
        cobra.cobra_decode_scan(block, desc, info, cache, lens, None, ws, nbytes_ws, stream)
        ev[3].record(stream)
        cobra.cobra_decode_combine(block, desc, info, lens, out, ws, nbytes_ws, stream)
        ev[4].record(stream)

    launches_per_step = 3  # query projection with both appends, scan, combine
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    st = cobra.cobra_check(stream)
    if st != cobra.COBRA_OK:
        raise RuntimeError(f"device status {st} after warm-up")

    # timed region: K whole steps, events only at its two ends (on the launch stream)
    K = args.steps
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    t_start.record(stream)
    for k in range(K):
        step()
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    total_ms = t_start.elapsed_time(t_end)
    # per-launch breakdown in a separate pass (events between the launches serialise them, so
    # the timed region above has none)
    KB = min(K, 200)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(stages) + 1)] for _ in range(KB)]
    for k in range(KB):
        staged_step(ev[k])
    torch.cuda.synchronize()
    stage_ms = {name: float(np.mean([e[i].elapsed_time(e[i + 1]) for e in ev])) for i, name in enumerate(stages)}
    scan_ms = stage_ms["scan"]
    total_ms = max_over_ranks(total_ms, world, dev)
    st = cobra.cobra_check(stream)
    if st != cobra.COBRA_OK:
        raise RuntimeError(f"device status {st} after the timed region")

    bytes_step = pipeline.packed_bytes_read(wl)
    value = weak_scaling_gbs(bytes_step, K, world, total_ms)

    # end to end through the public API: pinned host inputs in, host output out, every step
    hin = torch.empty_like(din, device="cpu").pin_memory()
    hout = torch.empty_like(out, device="cpu").pin_memory()
    hin.copy_(din.cpu())
    Ke = max(10, K // 4)

    # the step's inputs and output in pinned host memory; GB300's coherent NVLink-C2C lets the
    # kernels read the new tokens and queries from it and write the output into it directly
    hk, hv, hq = (hin[:n_kv].view(L, S, H, 128), hin[n_kv:2 * n_kv].view(L, S, H, 128),
                  hin[2 * n_kv:].view(L, S, Hq, 128))

    def e2e_step_direct():
        cobra.cobra_decode_step(block, desc, info, adesc[0], adesc[1], hk, hv, pos, hq, cache, lens, None, hout, ws,
                                nbytes_ws, stream)

    # the same with staging copies (one host-to-device copy of the inputs, one device-to-host
    # copy of the output)
    def e2e_step_staged():
        din.copy_(hin, non_blocking=True)
        cobra.cobra_decode_step(block, desc, info, adesc[0], adesc[1], xk, xv, pos, q, cache, lens, None, out, ws,
                                nbytes_ws, stream)
        hout.copy_(out, non_blocking=True)

    def time_e2e(fn):
        for _ in range(5):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(Ke):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return max_over_ranks(e0.elapsed_time(e1) / Ke, world, dev)

    e2e_staged_ms = time_e2e(e2e_step_staged)
    ref_out = hout.clone()
    e2e_ms = time_e2e(e2e_step_direct)
    if not torch.equal(hout, ref_out):
        raise RuntimeError("the step through host buffers differs from the staged step")
    h2d = din.numel() * 2
    d2h = out.numel() * 4

    peak, peak_kind = hbm_peak()
    achieved = bytes_step / (scan_ms * 1e-3) / 1e9
    # the legs below are measured after the headline: a failure in one is reported in its place
    legs = AuxLegs(stream)
    calibration = None
    if not args.no_calibration and rank == 0:
        calibration = legs.run(run_calibration_leg, args, dev, stream, srcs, not args.no_cpu_baseline and world == 1)
    measured = None
    if not args.no_measured and rank == 0:
        measured = legs.run(run_measured_leg, args, dev, stream, hp.cals, srcs, not args.no_cpu_baseline and world == 1)
    rope = None
    if not args.no_rope and rank == 0:
        rope = legs.run(run_rope_leg, args, dev, stream, hp, wl, desc, ws, info, q, lens, out,
                        not args.no_cpu_baseline and world == 1)
    configs = None
    if not args.no_configs and rank == 0:
        cb = not args.no_cpu_baseline and world == 1
        configs = {"tiny_2bpd": legs.run(run_tiny_leg, args, dev, stream, cb),
                   "llama3_70b_joint_0p5bpd": legs.run(run_llama3_70b_joint_leg, args, dev, stream, cb),
                   "ragged_paged_sweep": legs.run(run_ragged_sweep_leg, args, dev, stream, cb)}
    compress = None
    if not args.no_compress:
        del hin, hout
        compress = legs.run(run_compress_leg, args, dev, stream, peak)
    traffic = profiled_traffic()
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": K, "warmup": args.warmup,
            "ms_per_step": total_ms / K, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "fp16-mma/fp32-acc on 1-8 bit codes", "data": "synthetic", "impl": "cobra",
            "config": workload_config(spec) | split_config(args) | {"parallelism": f"replicas x{world}", "layers": L,
                                               "packed_bytes_per_step": bytes_step},
            "roofline": {"bound": "hbm", "kernel": "decode_kernel (rank-space scan)", "achieved": achieved,
                         "peak": peak, "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "scan_ms": scan_ms,
                         "algorithmic_bytes_per_launch": bytes_step, "frac_of_nominal_8TBs": achieved / 8000.0},
            "compress": compress,
            "other_decode_workloads": configs,
            "rope": rope,
            "measured": measured,
            "calibration": calibration,
            "cpu_baseline": cpu,
            "e2e": {"value": weak_scaling_gbs(bytes_step, 1, world, e2e_ms), "unit": "GB/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
                    "transfer": "cobra_decode_step on pinned host buffers: the kernels read the new K/V tokens "
                                "and queries from host memory and write the output there over NVLink-C2C",
                    "staged_copies": {"value": weak_scaling_gbs(bytes_step, 1, world, e2e_staged_ms),
                                      "ms_per_step": e2e_staged_ms,
                                      "transfer": "one cudaMemcpyAsync of the inputs in and one of the output "
                                                  "out, around the same call on device buffers"}},
            "stage_ms": stage_ms,
            "gpu_launches": launches_per_step * K,
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_cobra(args)


if __name__ == "__main__":
    main()
