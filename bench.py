#!/usr/bin/env python
"""Streaming-decode benchmark of the GB300 FlashDecoder library.

One step = one 480p stream of 16 latent chunks decoded through the C ABI (fd_reset, then 16 x
fd_decode_chunk), i.e. 64 output frames (r_t = 4 per chunk), the paper's FPS definition: total
decoded frames / total decode time (Sec. 4.1 "Evaluation Metrics"). Inputs are synthetic,
seeded latents shaped like Wan2.1 480p latents (16 x 60 x 104, PixelUnshuffle 2 -> 1560 tokens)
and random-init bf16 weights of the 24-block, D = 1024 decoder; they are resident in HBM
before the timed region. The weights alone (585 MB) exceed L2 (129 MB) and are re-read every
chunk, so no L2 flush is needed between steps.

Prints one JSON line (rank 0). --impl reference times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decoded frames/s and p50 per-chunk latency at 480p/720p; % bf16 TC peak"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="480p")
    ap.add_argument("--multi", default="batch", choices=["batch", "concurrent"],
                    help="several streams per GPU: stacked GEMMs (fd_decode_batch) or one "
                         "forked CUDA stream per decoder (fd_decode_chunks)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-secondary", action="store_true",
                    help="skip the other configurations (720p, 480p x 8, 720p wide, XL 480p)")
    ap.add_argument("--no-training", action="store_true", help="skip the training-step line")
    ap.add_argument("--training-only", action="store_true",
                    help="run only the training-step line (one GPU; for profiling it alone)")
    return ap.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            p = json.load(fh)
        return p["bf16_tflops"], p["bf16_tflops_sustained"], p["hbm_gbs"], "measured"
    except Exception:
        return 1900.0, 1700.0, 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu = gpu_id
        self.proc = None
        self.file = None

    def __enter__(self):
        try:
            self.file = tempfile.TemporaryFile(mode="w+")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.file, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None:
            return None
        self.file.seek(0)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.file:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


def source_hash(*names: str) -> str:
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_2607_14898_gb300", "csrc", n), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def ncu_traffic(kernel_file: str, workload: str, launch: str):
    """DRAM bytes of one launch of a kernel (launch = which of its launches was captured) from
    the committed ncu summary, if the kernel source (its file and the PTX primitives it
    includes) has not changed since the counters were taken (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    cur = source_hash(kernel_file, "fd_ptx.cuh")
    with open(path) as fh:
        for line in fh:
            f = line.split()
            if (len(f) >= 5 and f[0] == kernel_file and f[1] == workload and f[2] == cur
                    and f[4] == launch):
                return float(f[3])
    return None


def attention_traffic(workload: str, prof: dict):
    """DRAM bytes per attention launch, averaged over the same launches as the achieved rate:
    the backbone and refinement captures weighted by how many of each were profiled."""
    tb = ncu_traffic("fd_attn.cu", workload, "backbone")
    tr = ncu_traffic("fd_attn.cu", workload, "refine")
    nb, nr = prof["attn_backbone"][0], prof["attn_refine"][0]
    if tb is None or tr is None or nb + nr == 0:
        return None
    return round((tb * nb + tr * nr) / (nb + nr))


def kernel_profile(cfg, prof: dict, chunks: int, steps: int, sustained: float) -> dict:
    """Per-kernel-kind times of `steps` profiled streams of `chunks` chunks (CUDA events around
    each launch on its stream) against the kinds' algorithmic FLOPs and bytes."""
    from paper_2607_14898_gb300 import costs
    kflops, kbytes = {}, {}
    for t in range(chunks):
        for k, v in costs.chunk_flops(cfg, t).items():
            kflops[k] = kflops.get(k, 0) + v * steps
        for k, v in costs.chunk_bytes(cfg, t).items():
            kbytes[k] = kbytes.get(k, 0) + v * steps
    kernels = {}
    for k, (n, ms) in prof.items():
        if n == 0:
            continue
        e = {"launches": n, "ms_total": round(ms, 3), "us_per_launch": round(1e3 * ms / n, 2)}
        if k in kflops:
            e["tflops"] = round(kflops[k] / (ms * 1e-3) / 1e12, 1)
        if k in kbytes:
            e["gbs"] = round(kbytes[k] / (ms * 1e-3) / 1e9, 1)
        kernels[k] = e
    att_ms = prof["attn_backbone"][1] + prof["attn_refine"][1]
    att_n = prof["attn_backbone"][0] + prof["attn_refine"][0]
    att_flops = kflops["attn_backbone"] + kflops["attn_refine"]
    gemm_kinds = ["embed", "qkv", "out", "mlp1", "mlp2", "tup", "head1", "head2"]
    gemm_ms = sum(prof[k][1] for k in gemm_kinds)
    # fraction of the tensor-core roofline of the GEMMs; FP8 MLP products are held to the e4m3
    # peak, taken as the measured bf16 peak x the nominal e4m3 / bf16 ratio (2)
    fp8 = bool(getattr(cfg, "mlp_fp8", False))
    gemm_peak_time = sum(kflops[k] / (sustained * (2.0 if fp8 and k in ("mlp1", "mlp2") else 1.0))
                         for k in gemm_kinds) / 1e12
    return {"kernels": kernels, "att_ms": att_ms, "att_n": att_n, "att_flops": att_flops,
            "att_tflops": att_flops / (att_ms * 1e-3) / 1e12,
            "gemm_tflops": sum(kflops[k] for k in gemm_kinds) / (gemm_ms * 1e-3) / 1e12,
            "gemm_frac": gemm_peak_time / (gemm_ms * 1e-3),
            "ms_step": sum(ms for _, ms in prof.values()) / steps}


# ---------------------------------------------------------------------------------- GPU arm
def run_ours(args, rank: int, world: int):
    import numpy as np
    import torch

    import synth
    from paper_2607_14898_gb300 import costs
    from paper_2607_14898_gb300 import flashdec as fdp
    from paper_2607_14898_gb300.replicas import RankGroup, rank_env, stream_seeds

    local = rank_env().local_rank
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    group = RankGroup(dist, "cuda")

    cfg = synth.PRESETS[args.workload]
    chunks = cfg.chunks
    S = cfg.streams  # independent streams on this GPU (480p x 8: 8)
    frames_per_step = S * chunks * cfg.r_t
    w = synth.make_weights(cfg)
    blob = fdp.pack_blob(cfg, w)
    weights = fdp.Weights(cfg, blob)
    decs = [fdp.Decoder(cfg, weights) for _ in range(S)]
    dec = decs[0]
    # replicas: rank r decodes its own streams (latent seeds r*S .. r*S + S - 1)
    seeds = stream_seeds(cfg.latent_seed, rank, S)
    zs = [torch.from_numpy(synth.make_latents(cfg, seed=sd)).cuda() for sd in seeds]
    z = zs[0]
    out_dtype = torch.uint8 if cfg.out_u8 else torch.float32
    pixs = [[torch.empty(cfg.out_channels, cfg.r_t, cfg.out_h, cfg.out_w, dtype=out_dtype,
                         device="cuda") for _ in range(chunks)] for _ in range(S)]
    pix = pixs[0]
    stream = torch.cuda.Stream()
    batch = fdp.Batch(cfg, weights, S) if S > 1 and args.multi == "batch" else None

    def step(events=None):
        for d in decs:
            d.reset()
        for t in range(chunks):
            if events is not None:
                events[t][0].record(stream)
            if S == 1:
                dec.decode_chunk(z[t], pix[t], stream)
            elif batch is not None:  # chunk t of every stream, GEMMs stacked (fd_decode_batch)
                batch.decode(decs, [zz[t] for zz in zs], [pp[t] for pp in pixs], stream)
            else:  # chunk t of every stream, concurrently (fd_decode_chunks)
                fdp.decode_chunks(decs, [zz[t] for zz in zs], [pp[t] for pp in pixs], stream)
            if events is not None:
                events[t][1].record(stream)

    def step_single():  # stream 0 alone, for the per-kernel profile
        dec.reset()
        for t in range(chunks):
            dec.decode_chunk(z[t], pix[t], stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    torch.cuda.synchronize()
    if dec.sync_status() != fdp.FD_OK:
        raise RuntimeError("device error during warm-up")

    # ---------------------------------------------------------------- timed region
    ev = [[[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(chunks)]
          for _ in range(args.steps)]
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    launches0 = sum(d.launch_count for d in decs)
    group.barrier()
    torch.cuda.synchronize()
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(local).uuid)
    except Exception:
        gpu_id = str(local)
    with ClockSampler(gpu_id) as clocks:
        with torch.cuda.stream(stream):
            t0.record(stream)
            for k in range(args.steps):
                step(ev[k])
            t1.record(stream)
        torch.cuda.synchronize()
    group.barrier()
    gpu_launches = sum(d.launch_count for d in decs) - launches0
    ms_total = t0.elapsed_time(t1)
    value, frames_all, ms_max = group.throughput(frames_per_step * args.steps, ms_total)
    lat = [ev[k][t][0].elapsed_time(ev[k][t][1]) for k in range(args.steps) for t in range(chunks)]
    lat_steady = [ev[k][t][0].elapsed_time(ev[k][t][1]) for k in range(args.steps)
                  for t in range(cfg.window - 1, chunks)]
    if any(d.sync_status() != fdp.FD_OK for d in decs):
        raise RuntimeError("device error in the timed region")
    flops_step = S * costs.stream_flops(cfg, chunks)

    # ---------------------------------------------------------------- per-kernel profile
    dec.profile(True)
    with torch.cuda.stream(stream):
        for _ in range(args.steps):
            step_single()
    torch.cuda.synchronize()
    prof = dec.profile_collect()
    dec.profile(False)
    burst, sustained, hbm, peak_src = peaks()
    kp = kernel_profile(cfg, prof, chunks, args.steps, sustained)
    kernels, att_tflops, att_flops, att_ms, att_n = (kp["kernels"], kp["att_tflops"],
                                                     kp["att_flops"], kp["att_ms"], kp["att_n"])
    gemm_tflops, gemm_frac, prof_ms_step = kp["gemm_tflops"], kp["gemm_frac"], kp["ms_step"]
    fp8 = bool(getattr(cfg, "mlp_fp8", False))

    # ---------------------------------------------------------------- end to end (host buffers)
    lat_host = [torch.from_numpy(synth.make_latents(cfg, seed=sd)).pin_memory() for sd in seeds]
    pix_host = [[torch.empty(pix[0].shape, dtype=out_dtype).pin_memory() for _ in range(chunks)]
                for _ in range(S)]

    def step_host():
        for d in decs:
            d.reset()
        if S == 1:  # the whole stream in one overlapped host-buffer call
            dec.decode_sequence_host(list(lat_host[0]), pix_host[0], stream)
            return
        for t in range(chunks):  # streams one after another through the per-chunk call
            for i, d in enumerate(decs):
                d.decode_chunk_host(lat_host[i][t], pix_host[i][t], stream)

    with torch.cuda.stream(stream):
        step_host()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    group.barrier()
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(args.steps):
            step_host()
        e1.record(stream)
    torch.cuda.synchronize()
    group.barrier()
    e2e_value, _, _ = group.throughput(frames_per_step * args.steps, e0.elapsed_time(e1))
    latent_bytes = cfg.latent_channels * cfg.latent_h * cfg.latent_w * 4
    pixel_bytes = pix[0].numel() * pix[0].element_size()

    line = {
        "metric": METRIC,
        "value": round(value, 2),
        "unit": "frames/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(ms_max / args.steps, 3),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16 (block MLPs e4m3)" if fp8 else "bf16",
        "data": "synthetic (seeded N(0,1) latents, random-init N(0,0.02) bf16 weights)",
        "config": {
            "workload": f"{cfg.name} {S} stream{'s' if S > 1 else ''} per GPU: latent "
                        f"{cfg.latent_channels}x{cfg.latent_h}x{cfg.latent_w}, patch {cfg.patch} "
                        f"({cfg.tokens} tokens/chunk), {chunks} chunks per step, "
                        f"{cfg.n_blocks}+{cfg.n_refine} blocks, D={cfg.hidden}, "
                        f"{cfg.heads} heads / {cfg.kv_groups} KV groups, "
                        f"{'gated-SiLU' if cfg.mlp_gated else 'GELU'} MLP"
                        f"{' (FP8 e4m3, static scales)' if fp8 else ''}, W={cfg.window}, r_t="
                        f"{cfg.r_t}, output {cfg.out_h}x{cfg.out_w} "
                        f"{'uint8' if cfg.out_u8 else 'fp32'}",
            "frames_per_step": frames_per_step,
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "streams": ("single" if S == 1 else "fd_decode_batch (stacked GEMMs)"
                        if batch is not None else "fd_decode_chunks (forked CUDA streams)"),
            "l2": "no flush: per-chunk working set (585 MB bf16 weights) > 129 MB L2",
        },
        "latency_ms": {"p50": round(statistics.median(lat), 3),
                       "p99": round(sorted(lat)[max(0, int(0.99 * len(lat)) - 1)], 3),
                       "steady_p50": round(statistics.median(lat_steady), 3),
                       "steady_frames_per_s": round(S * cfg.r_t / (statistics.median(lat_steady)
                                                               * 1e-3), 2)},
        "tensor_tflops_step": round(flops_step * args.steps / (ms_total * 1e-3) / 1e12, 1),
        "tensor_frac_step": round(flops_step * args.steps / (ms_total * 1e-3) / 1e12
                                  / sustained, 3),
        "clocks": clocks.summary(),
        "e2e": {"value": round(e2e_value, 2), "unit": "frames/s",
                "h2d_bytes_per_step": S * chunks * latent_bytes,
                "d2h_bytes_per_step": S * chunks * pixel_bytes,
                "call": ("fd_decode_sequence_host (pinned host latents / pixels; copies "
                         "overlapped with the decoding on a library-owned copy stream)"
                         if S == 1 else "fd_decode_chunk_host per chunk (pinned host latents / "
                         "pixels, copies on the stream)")},
        "gpu_launches": int(gpu_launches),
        "roofline": {"kernel": "attention (attn_kernel, backbone + refinement launches)",
                     "bound": "tensor", "achieved": round(att_tflops, 1),
                     "peak": sustained, "unit": "TFLOP/s",
                     "frac": round(att_tflops / sustained, 3),
                     "peak_source": f"bf16_tflops_sustained ({peak_src}); kernel timed inside "
                                    "a long step",
                     "traffic": attention_traffic(cfg.name, prof),
                     "traffic_launch": "ncu DRAM read+write bytes per attention launch: one "
                                       "steady-state backbone and one refinement capture "
                                       "(profiles/traffic.txt), weighted by the launches "
                                       "profiled",
                     "flops_per_launch": round(att_flops / att_n),
                     "us_per_launch": round(1e3 * att_ms / att_n, 2),
                     "measured_over": f"{args.steps} profiled steps of the same workload "
                                      "(CUDA events around each launch on its stream)",
                     "gemm_tflops": round(gemm_tflops, 1),
                     "gemm_frac": round(gemm_frac, 3),
                     "gemm_peak": ("bf16 sustained; the FP8 MLP products against 2x that (e4m3)"
                                   if fp8 else "bf16 sustained"),
                     "profiled_ms_per_step": round(prof_ms_step, 3)},
        "kernels": kernels,
    }
    if rank == 0 and world == 1 and not args.no_secondary and cfg.name == "480p":
        line["secondary"] = {n: secondary_line(args, stream, n, blob) for n in SECONDARY}
    if rank == 0 and world == 1 and not args.no_training and cfg.name == "480p":
        line["training"] = training_line(args, stream, blob)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg, w)
    if batch is not None:
        batch.close()
    for d in decs:
        d.close()
    weights.close()
    if dist is not None:
        dist.destroy_process_group()
    return line


# further configurations of the benchmark, each timed like the headline in the same run
SECONDARY = ("720p", "480p_x8", "720p_wide", "xl_480p")


def secondary_line(args, stream, name, blob480):
    """One more configuration: warm-up streams, then one timed stream (CUDA events around each
    chunk on the launching stream), then its own per-kernel profile (stream 0 decoded alone,
    events around every launch) with the attention's roofline. Configurations with the 480p
    model's weight layout (720p, 480p x 8) reuse its blob; the others draw their own weights.
    Several streams per GPU (480p x 8) decode through fd_decode_batch, as the headline does."""
    import statistics as st

    import torch

    import synth
    from paper_2607_14898_gb300 import costs
    from paper_2607_14898_gb300 import flashdec as fdp

    cfg = synth.PRESETS[name]
    chunks, S = cfg.chunks, cfg.streams
    base = synth.PRESETS["480p"]
    same = (synth.weight_layout(cfg) == synth.weight_layout(base)
            and cfg.mlp_gated == base.mlp_gated and cfg.mlp_fp8 == base.mlp_fp8)
    blob = blob480 if same else fdp.pack_blob(cfg, synth.make_weights(cfg))
    weights = fdp.Weights(cfg, blob)
    decs = [fdp.Decoder(cfg, weights) for _ in range(S)]
    batch = fdp.Batch(cfg, weights, S) if S > 1 else None
    zs = [torch.from_numpy(synth.make_latents(cfg, chunks=chunks, seed=sd)).cuda()
          for sd in range(cfg.latent_seed, cfg.latent_seed + S)]
    dt = torch.uint8 if cfg.out_u8 else torch.float32
    pixs = [[torch.empty(cfg.out_channels, cfg.r_t, cfg.out_h, cfg.out_w, dtype=dt,
                         device="cuda") for _ in range(chunks)] for _ in range(S)]
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(chunks)]

    def step(record):
        for d in decs:
            d.reset()
        for t in range(chunks):
            if record:
                ev[t][0].record(stream)
            if batch is None:
                decs[0].decode_chunk(zs[0][t], pixs[0][t], stream)
            else:
                batch.decode(decs, [z[t] for z in zs], [p[t] for p in pixs], stream)
            if record:
                ev[t][1].record(stream)

    def step_single():
        decs[0].reset()
        for t in range(chunks):
            decs[0].decode_chunk(zs[0][t], pixs[0][t], stream)

    warm = 1 if chunks * cfg.tokens > 16 * 3600 else max(1, args.warmup)
    with torch.cuda.stream(stream):
        for _ in range(warm):
            step(False)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        step(True)
        b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b)
    lat = [ev[t][0].elapsed_time(ev[t][1]) for t in range(chunks)]
    steady = lat[cfg.window - 1:]
    ok = all(d.sync_status() == fdp.FD_OK for d in decs)
    decs[0].profile(True)
    with torch.cuda.stream(stream):
        step_single()
    torch.cuda.synchronize()
    prof = decs[0].profile_collect()
    decs[0].profile(False)
    _, sustained, _, peak_src = peaks()
    kp = kernel_profile(cfg, prof, chunks, 1, sustained)
    if batch is not None:
        batch.close()
    for d in decs:
        d.close()
    weights.close()
    flops = S * costs.stream_flops(cfg, chunks)
    fp8 = bool(cfg.mlp_fp8)
    return {"workload": f"{name}: {S} stream{'s' if S > 1 else ''} of {chunks} chunks, latent "
                        f"{cfg.latent_channels}x{cfg.latent_h}x{cfg.latent_w}, patch {cfg.patch} "
                        f"({cfg.tokens} tokens/chunk), {cfg.n_blocks}+{cfg.n_refine} blocks, "
                        f"D={cfg.hidden}, {cfg.heads} heads / {cfg.kv_groups} KV groups, "
                        f"{'gated-SiLU' if cfg.mlp_gated else 'GELU'} MLP, W={cfg.window}, "
                        f"{'uint8' if cfg.out_u8 else 'fp32'} pixels, "
                        f"{'AR(1)' if cfg.latent_mode == 'ar1' else 'N(0,1)'} latents"
                        + (", fd_decode_batch (stacked GEMMs)" if S > 1 else ""),
            "frames_per_s": round(S * chunks * cfg.r_t / (ms * 1e-3), 2),
            "warmup_streams": warm,
            "p50_ms": round(st.median(lat), 3), "steady_p50_ms": round(st.median(steady), 3),
            "p99_ms": round(sorted(lat)[max(0, int(0.99 * len(lat)) - 1)], 3),
            "tensor_frac_step": round(flops / (ms * 1e-3) / 1e12 / sustained, 3),
            "roofline": {"kernel": "attention (attn_kernel, backbone + refinement launches)"
                                   + (", stream 0 alone" if S > 1 else ""),
                         "bound": "tensor", "achieved": round(kp["att_tflops"], 1),
                         "peak": sustained, "unit": "TFLOP/s",
                         "frac": round(kp["att_tflops"] / sustained, 3),
                         "peak_source": f"bf16_tflops_sustained ({peak_src})",
                         "flops_per_launch": round(kp["att_flops"] / kp["att_n"]),
                         "us_per_launch": round(1e3 * kp["att_ms"] / kp["att_n"], 2),
                         "gemm_tflops": round(kp["gemm_tflops"], 1),
                         "gemm_frac": round(kp["gemm_frac"], 3),
                         "gemm_peak": ("bf16 sustained; the FP8 MLP products against 2x that"
                                       if fp8 else "bf16 sustained"),
                         "measured_over": "1 profiled stream (CUDA events around each launch)"},
            "kernels": kp["kernels"], "device_ok": ok}


TRAIN_CHUNKS = 2


def training_line(args, stream, blob):
    """Streaming training step of the 480p model (fd_train_step) over a clip of TRAIN_CHUNKS
    latent chunks: forward with every activation kept, L1 loss against the target pixels, every
    parameter's gradient. Synthetic latents and targets, the bench's random-init weights; inputs
    resident in HBM. Steps timed with CUDA events on the launching stream; then one profiled
    step (events around every launch) for the per-kind times and the dominant kind's roofline."""
    import numpy as np
    import torch

    import synth
    from paper_2607_14898_gb300 import costs
    from paper_2607_14898_gb300 import flashdec as fdp

    cfg = synth.PRESETS["480p"]
    T = TRAIN_CHUNKS
    weights = fdp.Weights(cfg, blob)
    tr = fdp.Trainer(cfg, weights, T)
    lat = torch.from_numpy(synth.make_latents(cfg, chunks=T)).cuda()
    tgt = torch.from_numpy(np.ascontiguousarray(
        np.stack(synth.make_target_pixels(cfg, chunks=T, min_abs=0.3)))).cuda()
    loss = torch.zeros(1, device="cuda")
    grads = torch.zeros(tr.grad_elems, device="cuda")
    for _ in range(max(3, args.warmup)):
        tr.step(lat, tgt, loss, grads, stream)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = max(1, args.steps)
    a.record(stream)
    for _ in range(steps):
        tr.step(lat, tgt, loss, grads, stream)
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / steps
    ok = tr.status(stream) == fdp.FD_OK
    tr.profile(True)
    tr.step(lat, tgt, loss, grads, stream)
    prof = tr.profile_collect()
    tr.profile(False)
    tr.close()
    weights.close()
    _, sustained, hbm, peak_src = peaks()
    fl = costs.training_kind_flops(cfg, T)
    total = sum(fl.values())
    kinds = {}
    for k, (n, kms) in prof.items():
        e = {"launches": n, "ms": round(kms, 3)}
        if k in fl and kms > 0:
            e["tflops"] = round(fl[k] / (kms * 1e-3) / 1e12, 1)
        kinds[k] = e
    top = max(prof, key=lambda k: prof[k][1])
    dom = {"kernel": f"{top} (the kind with the most device time in the profiled step)"}
    if top in fl:
        ach = fl[top] / (prof[top][1] * 1e-3) / 1e12
        dom.update({"bound": "tensor", "achieved": round(ach, 1), "peak": sustained,
                    "unit": "TFLOP/s", "frac": round(ach / sustained, 3),
                    "peak_source": f"bf16_tflops_sustained ({peak_src})",
                    "work": "algorithmic FLOPs of the kind (costs.training_kind_flops)"})
    return {"workload": f"480p model (24 + 2 blocks, D 1024), streaming training step over a "
                        f"clip of {T} latent chunks ({T * cfg.r_t} frames): forward with the "
                        "activations kept, L1 loss, every parameter's gradient",
            "ms_per_step": round(ms, 3), "steps": steps,
            "frames_per_s": round(T * cfg.r_t / (ms * 1e-3), 2),
            "tflops": round(total / (ms * 1e-3) / 1e12, 1),
            "tensor_frac_step": round(total / (ms * 1e-3) / 1e12 / sustained, 3),
            "roofline": dom, "kinds": kinds,
            "profiled_ms": round(sum(v[1] for v in prof.values()), 3), "device_ok": ok}


def cpu_model() -> str:
    """The host CPU's model name (lscpu / /proc/cpuinfo), for the baseline's record."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() in ("Model name", "Model"):
                name = line.split(":", 1)[1].strip()
                if name and not name.isdigit():
                    return name
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as fh:
            for line in fh:
                if line.lower().startswith(("model name", "cpu part")):
                    return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


class SteadyOracle:
    """The CPU oracle decoding one stream (fp64 PyTorch, as it stands): the first W - 1 chunks
    fill its cache untimed, so every timed chunk attends over a full window of W chunks (the
    steady state of the stream, where per-chunk cost stays constant)."""

    def __init__(self, cfg, w, threads: int, chunks: int):
        import torch

        import oracle
        import synth
        torch.set_num_threads(threads)
        self.z = synth.make_latents(cfg, chunks=chunks + cfg.window - 1)
        self.dec = oracle.StreamingDecoder(cfg, w)
        self.t = 0
        for _ in range(cfg.window - 1):
            self.dec.decode_chunk(self.z[self.t])
            self.t += 1

    def timed_chunk(self) -> float:
        t0 = time.perf_counter()
        self.dec.decode_chunk(self.z[self.t])
        sec = time.perf_counter() - t0
        self.t += 1
        return sec


def steady_sample(cfg) -> str:
    return (f"steady-state chunk of the {cfg.name} stream (chunk t >= W-1 = {cfg.window - 1}: "
            f"the cache holds W = {cfg.window} chunks; the first W-1 chunks decoded untimed), "
            f"full {cfg.n_blocks}+{cfg.n_refine}-block model, fp64 PyTorch CPU oracle")


def cpu_baseline(cfg, w):
    """The oracle's steady-state rate: after the cache fill, one steady-state chunk untimed
    (first-touch costs of its larger attention buffers), then one timed."""
    threads = os.cpu_count() or 1
    ref = SteadyOracle(cfg, w, threads, 2)
    ref.timed_chunk()
    sec = ref.timed_chunk()
    return {"value": round(cfg.r_t / sec, 4), "unit": "frames/s", "cores": threads,
            "cpu": cpu_model(), "kind": "oracle",
            "sample": f"one {steady_sample(cfg)} (the second steady-state chunk), {sec:.1f} s "
                      f"for {cfg.r_t} frames"}


# ---------------------------------------------------------------------------- reference arm
def run_reference(args):
    """The oracle (there is no reference implementation: the reference is a paper), on the
    host cores. A steady-state chunk of the 480p stream takes about 43 s there (16 cores), so
    that W + K steps end within a few minutes each step is a smaller sample of the same
    stream: chunk 0 after a reset (the cache holds that one chunk). The steady-state rate is
    the cpu_baseline of the GPU arm's line."""
    import torch

    import oracle
    import synth
    cfg = synth.PRESETS[args.workload]
    w = synth.make_weights(cfg)
    threads = os.cpu_count() or 1
    torch.set_num_threads(threads)
    z = synth.make_latents(cfg, chunks=1)

    def chunk0() -> float:
        dec = oracle.StreamingDecoder(cfg, w)
        t0 = time.perf_counter()
        dec.decode_chunk(z[0])
        return time.perf_counter() - t0

    for _ in range(args.warmup):
        chunk0()
    secs = [chunk0() for _ in range(args.steps)]
    total = sum(secs)
    value = cfg.r_t * args.steps / total
    sample = (f"per step: chunk 0 of the {cfg.name} stream after a reset (the cache holds 1 of "
              f"W = {cfg.window} chunks), full {cfg.n_blocks}+{cfg.n_refine}-block model, fp64 "
              f"PyTorch CPU oracle")
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": "frames/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * total / args.steps, 1), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{cfg.name} single stream (oracle sample)", "sample": sample},
        "cpu_baseline": {"value": round(value, 4), "unit": "frames/s", "cores": threads,
                         "cpu": cpu_model(), "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "frames/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main():
    args = parse()
    from paper_2607_14898_gb300.replicas import rank_env
    env = rank_env()
    rank, world = env.rank, env.world
    if args.impl == "reference":
        if rank != 0:
            return
        print(json.dumps(run_reference(args)), flush=True)
        return
    if args.training_only:
        import torch

        import synth
        from paper_2607_14898_gb300 import flashdec as fdp
        cfg = synth.PRESETS["480p"]
        torch.cuda.set_device(0)
        stream = torch.cuda.Stream()
        line = {"training": training_line(args, stream,
                                          fdp.pack_blob(cfg, synth.make_weights(cfg)))}
        print(json.dumps(line), flush=True)
        return
    line = run_ours(args, rank, world)
    if rank == 0:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
