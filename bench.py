"""Benchmark: incremental ViT encode of a streaming camera feed on one GB300 (or N
replicas under torchrun).

A step is one ``ivit_encode_incremental`` call on the next frame of a seeded synthetic
stream (the whole hot path: embed, score, select, gather, every block on the updated
rows, final-token scatter).  Default workload: SigLIP-So400m-shaped encoder, 224x224
frames (256 tokens), one camera, about 10% dynamic patches per frame.

Printed JSON line (rank 0): frames/s of the incremental path with the frames already
resident in HBM (``value``), ms per frame, the same library's full re-encode on the
same frames and the speedup over it, the end-to-end number through the C ABI with host
buffers (``e2e``), the GEMM kernel family's achieved HBM bandwidth against the measured
peak, timed inside the replayed CUDA graph by the library's kernel timeline, with every
family's time per step and the call-level fraction of the HBM roofline (``roofline``),
the oracle's CPU throughput (``cpu_baseline``) and the SM clocks sampled during the
timed region.

``--impl reference`` times the oracle (the plain CPU restatement the library is checked
against) on the same workload instead.
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
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_12287_gb300 import synth  # noqa: E402

METRIC = "ms/frame and frames/s incremental ViT encode at 10% dynamic tokens; x vs full encode"
DEFAULT_WORKLOAD = "so400m_224_1view"


def describe(wl) -> dict:
    s = wl.shape
    return {
        "workload": wl.name,
        "encoder": (f"{s.img_h}x{s.img_w} px, patch {s.patch} ({s.n_tokens} tokens/view), dim {s.dim}, "
                    f"{s.depth} layers, {s.heads} heads, MLP {s.mlp_dim}, pre-LN, "
                    f"{'tanh' if s.gelu == 0 else 'erf'} GELU, seeded random-init bf16 weights"),
        "views": wl.sv,
        "selection": ("threshold sim<%.2f" % wl.threshold) if wl.select_mode == 0 else f"top-{wl.topk}",
        "scene": wl.scene,
    }


def read_peaks() -> dict:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d.get("hbm_gbs"), "bf16_tflops": d.get("bf16_tflops"),
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained") or d.get("bf16_tflops"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


L2_BYTES = 129e6  # GB300 L2


def weight_matrix_bytes(shape) -> float:
    """bf16 bytes of the weight matrices every call streams (patch embedding, QKV,
    out-proj, MLP) -- the weights term of the algorithmic bytes."""
    D, F, L = shape.dim, shape.mlp_dim, shape.depth
    kp = shape.patch * shape.patch * 3
    return 2.0 * (D * kp + L * (3 * D * D + D * D + 2 * D * F))


def algorithmic_bytes_per_step(wl, rows_per_step: float) -> float:
    """Bytes one incremental call must move at least: the weights once, every view's
    cached K/V of every layer read by attention, the frames, the patch embeddings
    written and scored against the reference (fp32, read twice), and the updated rows'
    K/V and output tokens written."""
    s = wl.shape
    N, D, L, sv = s.n_tokens, s.dim, s.depth, wl.sv
    kv = 2.0 * 2 * L * sv * N * D
    frames = sv * s.img_h * s.img_w * 3
    embed = 3 * 4.0 * sv * N * D
    writes = rows_per_step * (2 * 2 * L * D + 2 * D)
    return weight_matrix_bytes(s) + kv + frames + embed + writes


def ideal_ms_per_step(wl, rows_per_step: float, full: bool, peaks: dict) -> dict:
    """Roofline time of one call: the larger of its algorithmic bytes at the measured HBM
    copy bandwidth and its FLOPs at the measured sustained bf16 tensor throughput.  A
    full encode runs every block on all SV*N tokens and writes every cached K/V; an
    incremental call runs them on ``rows_per_step`` updated tokens and reads every cached
    K/V (Sec. III-B, Eq. 4-5).  Both stream the weights once and embed every patch."""
    s = wl.shape
    N, D, F, L, sv = s.n_tokens, s.dim, s.mlp_dim, s.depth, wl.sv
    kp = s.patch * s.patch * 3
    rows = float(sv * N) if full else float(rows_per_step)
    flops = 2.0 * sv * N * D * kp + L * (rows * 2.0 * (4 * D * D + 2 * D * F) + 4.0 * rows * N * D)
    kv_all = 2.0 * 2 * L * sv * N * D
    if full:
        byts = weight_matrix_bytes(s) + kv_all + sv * s.img_h * s.img_w * 3 + 3 * 4.0 * sv * N * D
    else:
        byts = algorithmic_bytes_per_step(wl, rows)
    t_mem = byts / (peaks["hbm_gbs"] * 1e9)
    t_mma = flops / (peaks["bf16_tflops_sustained"] * 1e12)
    return {"ms": 1e3 * max(t_mem, t_mma), "bound": "hbm" if t_mem >= t_mma else "tensor", "bytes": byts,
            "flops": flops}


def gemm_traffic_ratio():
    """DRAM bytes / algorithmic bytes of the GEMM from the committed ncu summary, or None
    when the kernel source changed since that capture."""
    summ = os.path.join(ROOT, "profiles", "gemm_tc_kernel_so400m_224_1view.md")
    if not os.path.exists(summ):
        return None
    text = open(summ).read()
    m = re.search(r"traffic_to_algorithmic_ratio:\s*([0-9.eE+]+)", text)
    h = re.search(r"gemm_tc_kernel_source_sha256:\s*([0-9a-f]{64})", text)
    if not m or not h:
        return None
    # the profiled kernel and everything it uses sit above the warp-specialised form
    src = open(os.path.join(ROOT, "paper_2607_12287_gb300", "csrc", "gemm.cu")).read()
    cut = src.find("// Many-tile form")
    if cut < 0 or hashlib.sha256(src[:cut].encode()).hexdigest() != h.group(1):
        return None
    return float(m.group(1))


class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return None
        rows = []
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
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, flags in rows for i, f in enumerate(flags) if f == "Active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "samples": len(rows), "reasons": reasons}


def make_frames(wl, n: int):
    return [np.ascontiguousarray(f) for f in wl.frames(n)]


def replica_workload(wl, rank: int):
    """Weak scaling: every rank encodes its own camera streams (the same scene recipe
    with its own seed); ranks exchange nothing on the data path."""
    import dataclasses
    return dataclasses.replace(wl, seed=wl.seed + 1000 * rank) if rank else wl


def max_over_ranks(value: float, dist, device=None) -> float:
    """The slowest rank's time (the job finishes when every replica has)."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def cpu_baseline(wl, weights, frames, budget_s: float = 20.0) -> dict:
    """The oracle as it stands, on this host's cores: an untimed full encode of frame 0,
    then incremental frames timed until ``budget_s`` is spent (at least one)."""
    import oracle
    orc = oracle.Oracle.for_workload(wl, weights)
    orc.encode_full(frames[0])
    done, t0 = 0, time.perf_counter()
    while done + 3 < len(frames):  # keeps two frames for the single-thread leg
        orc.encode_incremental(frames[done + 1])
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    el = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0))
    # the same oracle state continued on one thread (bounded to a few frames)
    single = None
    if done + 1 < len(frames):
        oracle.set_threads(1)
        n1, t1 = 0, time.perf_counter()
        while done + 1 + n1 < len(frames):
            orc.encode_incremental(frames[done + 1 + n1])
            n1 += 1
            if time.perf_counter() - t1 > budget_s / 2:
                break
        el1 = time.perf_counter() - t1
        oracle.set_threads(cores)
        single = {"value": n1 * wl.sv / el1, "unit": "frames/s", "cores": 1,
                  "sample": f"frames {done + 1}..{done + n1} of the same stream ({el1:.1f} s)"}
    orc.close()
    return {"value": done * wl.sv / el, "unit": "frames/s", "cores": cores, "kind": "oracle",
            "sample": (f"oracle incremental encode of frames 1..{done} of the {wl.name} stream after an "
                       f"untimed full encode of frame 0 ({el:.1f} s, OpenMP over {cores} cores)"),
            "single_thread": single}


def run_reference(args, wl, rank: int) -> None:
    if rank != 0:
        return
    weights = synth.make_weights(wl.shape, 0)
    frames = make_frames(wl, 1 + args.warmup + args.steps)
    import oracle
    orc = oracle.Oracle.for_workload(wl, weights)
    orc.encode_full(frames[0])
    for t in range(args.warmup):
        orc.encode_incremental(frames[1 + t])
    t0 = time.perf_counter()
    for t in range(args.steps):
        orc.encode_incremental(frames[1 + args.warmup + t])
    el = time.perf_counter() - t0
    orc.close()
    fps = args.steps * wl.sv / el
    cores = len(os.sched_getaffinity(0))
    line = {
        "impl": "reference", "metric": METRIC, "value": fps, "unit": "frames/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "config": describe(wl),
        "cpu_baseline": {"value": fps, "unit": "frames/s", "cores": cores, "kind": "oracle",
                         "sample": f"{args.steps} incremental frames after a full encode and "
                                   f"{args.warmup} warm-up frames, OpenMP over {cores} cores"},
        "e2e": {"value": fps, "unit": "frames/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ivit", choices=["ivit", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--streams", type=int, default=0,
                    help="run the workload with this many camera streams (its first ones)")
    ap.add_argument("--lean", action="store_true",
                    help="time the incremental and full steps only (one handle: for profiler captures)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.workload in synth.WORKLOADS:
        wl = synth.WORKLOADS[args.workload]
    elif args.workload.startswith("so400m_224_sweep_"):
        wl = synth.sweep_workload(int(args.workload.rsplit("_", 1)[1].rstrip("pct")) / 100.0)
    else:
        ap.error(f"unknown workload {args.workload}")
    if args.streams > 0:
        import dataclasses
        sv = args.streams * wl.n_views
        views = wl.views[:sv] if len(wl.views) >= sv else wl.views
        wl = dataclasses.replace(wl, name=f"{wl.name}_{args.streams}streams", n_streams=args.streams, views=views)

    if args.impl == "reference":
        run_reference(args, wl, rank)
        return

    import torch
    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")

    import paper_2607_12287_gb300 as pkg
    dev = torch.device("cuda", local_rank)
    wl = replica_workload(wl, rank)
    weights = synth.make_weights(wl.shape, 0)
    n_frames = 1 + args.warmup + args.steps
    frames = make_frames(wl, n_frames)
    frames_dev = [torch.from_numpy(f).to(dev) for f in frames]
    enc = pkg.IncrementalViT.for_workload(wl, weights)
    stream = torch.cuda.current_stream(dev)
    out = enc.tokens_buffer()
    counts = torch.zeros((n_frames, wl.sv), dtype=torch.int32, device=dev)

    def barrier():
        torch.cuda.synchronize(dev)
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize(dev)

    host_ms = {}

    step_ms = {}

    def timed(fn_step, label, encoder=None):
        """Full encode of frame 0, warm-up frames, then K timed steps (CUDA events on the
        launch stream, one after every step for the per-step distribution)."""
        (encoder or enc).encode_full(frames_dev[0], out)
        for t in range(args.warmup):
            fn_step(1 + t)
        barrier()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
        ev[0].record(stream)
        h0 = time.perf_counter()
        for t in range(args.steps):
            fn_step(1 + args.warmup + t)
            ev[t + 1].record(stream)
        host_ms[label] = 1e3 * (time.perf_counter() - h0) / args.steps
        ev[-1].synchronize()
        ms = ev[0].elapsed_time(ev[-1])
        per = np.array([ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)])
        step_ms[label] = {"median": float(np.median(per)), "p10": float(np.percentile(per, 10)),
                          "p90": float(np.percentile(per, 90))}
        barrier()
        return max_over_ranks(ms, dist, dev)

    def inc_step(t):
        pkg.ivit_encode_incremental(enc.h, frames_dev[t], out, counts[t], stream)

    def full_step(t):
        pkg.ivit_encode_full(enc.h, frames_dev[t], out, stream)

    peaks = read_peaks()
    with ClockSampler(local_rank) as clk:
        inc_ms = timed(inc_step, "incremental")
    clocks = clk.summary()
    launches_per_step = pkg.ivit_last_launch_count(enc.h)
    changed = counts[1 + args.warmup:].float().sum(1).cpu().numpy()
    full_ms = timed(full_step, "full")
    if args.lean:  # profiler captures: the two timed passes only
        if rank == 0:
            print(json.dumps({"metric": METRIC, "lean": True, "config": describe(wl),
                              "ms_per_step": inc_ms / args.steps, "full_encode_ms_per_step": full_ms / args.steps,
                              "device_status": enc.device_status(), "clocks": clocks}), flush=True)
        enc.close()
        if dist is not None:
            dist.barrier()
            dist.destroy_process_group()
        return

    # e2e: host frames (pinned) -> device, encode through the C ABI, tokens + counts -> host
    host_in = [torch.from_numpy(f).pin_memory() for f in frames]
    host_out = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    host_cnt = torch.empty(wl.sv, dtype=torch.int32).pin_memory()
    dev_in = torch.empty_like(frames_dev[0])
    cnt_dev = torch.empty(wl.sv, dtype=torch.int32, device=dev)

    def e2e_step(t):
        dev_in.copy_(host_in[t], non_blocking=True)
        pkg.ivit_encode_incremental(enc.h, dev_in, out, cnt_dev, stream)
        host_out.copy_(out, non_blocking=True)
        host_cnt.copy_(cnt_dev, non_blocking=True)

    e2e_ms = timed(e2e_step, "e2e")

    # Kernel timeline inside the replayed graph: every launch of a step records its CTAs'
    # start (after the wait on the previous kernel) and end times (the graph is captured
    # again with the recording in it); per-family time per step is the sum over its
    # launches of (last end - first start).
    pkg.ivit_timeline(enc.h, True)
    enc.encode_full(frames_dev[0], out)
    fam_ms = {f: 0.0 for f in pkg.TIMELINE_FAMILIES}
    fam_n = {f: 0 for f in pkg.TIMELINE_FAMILIES}
    tl_bytes = tl_span = 0.0
    for t in range(args.steps):
        inc_step(1 + args.warmup + t)
        r = pkg.ivit_timeline_read(enc.h, stream)
        if t < 2:  # the first calls capture the graph again
            continue
        for f in fam_ms:
            fam_ms[f] += r["ms"][f]
            fam_n[f] += r["launches"][f]
        tl_bytes += r["gemm_bytes"]
        tl_span += r["span_ms"]
    tl_steps = max(1, args.steps - 2)
    pkg.ivit_timeline(enc.h, False)
    status = enc.device_status()

    # Approximation quality (a diagnostic, not gated): per-token cosine between the
    # incremental output and a full re-encode of the same frame, over a few frames.
    ref_enc = pkg.IncrementalViT.for_workload(wl, weights)

    def quality(encoder, n=8):
        n = min(n, n_frames - 1)
        encoder.encode_full(frames_dev[0], out)
        means, low = [], 1.0
        for t in range(1, 1 + n):
            a, _ = encoder.encode_incremental(frames_dev[t])
            b = ref_enc.encode_full(frames_dev[t])
            c = torch.nn.functional.cosine_similarity(a.float(), b.float(), dim=-1)
            means.append(float(c.mean()))
            low = min(low, float(c.min()))
        return {"frames": n, "mean_token_cosine": float(np.mean(means)), "min_token_cosine": low}

    quality_default = quality(enc)
    # The paper's alternating chunks (Sec. III-B) through the library's schedule option:
    # every other call is a full encode.
    import dataclasses
    enc_oe = pkg.IncrementalViT.for_workload(dataclasses.replace(wl, schedule=synth.SCHED_ODD_EVEN), weights)
    oe_ms = timed(lambda t: pkg.ivit_encode_incremental(enc_oe.h, frames_dev[t], out, counts[t], stream),
                  "odd_even", enc_oe)
    enc_oe.close()
    # The other reading of Sec. III-B: attention on the updated tokens, MLP on every token.
    enc_all = pkg.IncrementalViT.for_workload(dataclasses.replace(wl, mlp_tokens=1), weights)
    all_ms = timed(lambda t: pkg.ivit_encode_incremental(enc_all.h, frames_dev[t], out, counts[t], stream),
                   "mlp_all_tokens", enc_all)
    mlp_all = {"ms_per_step": all_ms / args.steps, "speedup_vs_full": full_ms / all_ms,
               "quality_vs_full": quality(enc_all), "device_status": enc_all.device_status()}
    enc_all.close()
    ref_enc.close()

    frames_total = args.steps * wl.sv * world
    value = frames_total / (inc_ms / 1e3)
    ms_step = inc_ms / args.steps
    gemm_launches = fam_n["gemm"] / tl_steps
    gemm_ms_step = fam_ms["gemm"] / tl_steps
    gemm_bytes_step = tl_bytes / tl_steps
    achieved = gemm_bytes_step / (gemm_ms_step / 1e3) / 1e9 if gemm_ms_step > 0 else None
    ratio = gemm_traffic_ratio()
    traffic = ratio * gemm_bytes_step / gemm_launches if (ratio is not None and gemm_launches) else None
    rows_step = float(changed.mean())
    call_bytes = algorithmic_bytes_per_step(wl, rows_step)
    ideal_inc = ideal_ms_per_step(wl, rows_step, False, peaks)
    ideal_full = ideal_ms_per_step(wl, rows_step, True, peaks)
    wbytes = weight_matrix_bytes(wl.shape)
    line = {
        "metric": METRIC, "value": value, "unit": "frames/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": inc_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": dict(describe(wl), **{
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
            "l2": ("no flush: the weight matrices (%.0f MB bf16) exceed the 129 MB L2 and are streamed "
                   "from HBM every step" % (wbytes / 1e6)) if wbytes > L2_BYTES else
                  ("no flush: the weight matrices (%.1f MB bf16) fit in the 129 MB L2 and stay resident "
                   "across steps (the streaming workload as it runs)" % (wbytes / 1e6)),
            "changed_tokens_per_frame_mean": float(changed.mean()) / wl.sv,
            "dynamic_fraction_mean": float(changed.mean()) / (wl.sv * wl.shape.n_tokens),
        }),
        "ms_per_frame": inc_ms / args.steps / wl.sv,
        "timesteps_per_s": args.steps * world / (inc_ms / 1e3),
        "ms_per_step_distribution": step_ms,
        "full_encode_ms_per_step": full_ms / args.steps,
        "full_encode_frames_per_s": frames_total / (full_ms / 1e3),
        "speedup_vs_full": full_ms / inc_ms,
        # the same ratio at the roofline (measured peaks): what a perfect implementation of
        # both calls would show on this workload
        "ideal_speedup_vs_full": ideal_full["ms"] / ideal_inc["ms"],
        "ideal_ms_per_step": {"incremental": ideal_inc, "full": ideal_full,
                              "frac_incremental": ideal_inc["ms"] / ms_step,
                              "frac_full": ideal_full["ms"] / (full_ms / args.steps)},
        "odd_even_ms_per_step": oe_ms / args.steps,  # Sec. III-B alternating full / incremental calls
        "quality_vs_full": quality_default,
        "mlp_all_tokens": mlp_all,
        "e2e": {"value": frames_total / (e2e_ms / 1e3), "unit": "frames/s",
                "ms_per_step": e2e_ms / args.steps,
                "h2d_bytes_per_step": int(frames[0].nbytes),
                "d2h_bytes_per_step": int(out.numel() * out.element_size() + wl.sv * 4)},
        "roofline": {"kernel": "gemm_tc_kernel (every QKV/out-proj/MLP/embed launch of a step)", "bound": "hbm",
                     "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": (achieved / peaks["hbm_gbs"]) if achieved else None,
                     "peak_source": peaks["source"] + " (copy bandwidth, MEASURED_PEAKS.json)",
                     "traffic": traffic,
                     "traffic_source": ("ncu dram__bytes ratio of the committed GEMM summary x algorithmic bytes"
                                        if traffic is not None else
                                        "null: gemm.cu changed since the committed ncu capture"),
                     "timing": ("in-graph kernel timeline: per launch, last CTA end - first CTA start after the "
                                "wait on the previous kernel (globaltimer), summed over the step's launches; "
                                "%d steps after two graph captures" % tl_steps),
                     "launches_per_step": gemm_launches,
                     "avg_launch_us": 1e3 * gemm_ms_step / gemm_launches if gemm_launches else None,
                     "algorithmic_bytes_per_launch": gemm_bytes_step / gemm_launches if gemm_launches else None,
                     "families_ms_per_step": {f: fam_ms[f] / tl_steps for f in fam_ms},
                     "families_launches_per_step": {f: fam_n[f] / tl_steps for f in fam_n},
                     "kernel_span_ms_per_step": tl_span / tl_steps,
                     "call_level": {"algorithmic_bytes_per_step": call_bytes,
                                    "achieved": call_bytes / (ms_step / 1e3) / 1e9,
                                    "frac": call_bytes / (ms_step / 1e3) / 1e9 / peaks["hbm_gbs"],
                                    "what": "weights + cached K/V of every layer + frames + embeddings + "
                                            "updated rows' K/V and tokens, / ms_per_step"}},
        "host_enqueue_ms_per_step": host_ms,
        "gpu_launches": int(launches_per_step * args.steps),
        "launches_per_step": int(launches_per_step),
        "device_status": status,
        "clocks": clocks,
    }
    if rank == 0 and not args.no_cpu:
        line["cpu_baseline"] = cpu_baseline(wl, weights, frames)
    if rank == 0:
        print(json.dumps(line), flush=True)
    enc.close()
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
