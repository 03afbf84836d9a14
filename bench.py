"""Benchmark: streaming chunk-causal attention on the 1080p-shaped workload.

One step streams a whole synthetic 1080p-shaped video through the library:
15 chunks of 2 latent frames x 8160 tokens, 12 heads, d = 128, each chunk one
KV-cache append plus one chunk-causal attention forward over every earlier
chunk (Sec. 3.1 with an unbounded window).  The metric is attention TFLOP/s
counted on visible (query, key) pairs only, 4*B*H*Lq*Lk*d per chunk.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Under torchrun (N > 1) every rank streams its own video (weak scaling: the
videos are independent units, no data-path collective); the timed region is
bracketed by a barrier and CUDA synchronisation and the max over ranks is
reported.  `--impl reference` times the CPU oracle on this host's cores on a
bounded sample of the same workload (no GPU work).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

HOST_CORES = len(os.sched_getaffinity(0))
os.environ.setdefault("OPENBLAS_NUM_THREADS", str(HOST_CORES))
os.environ.setdefault("OMP_NUM_THREADS", str(HOST_CORES))

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2609_36757_gb300 import workloads as WL  # noqa: E402

METRIC = "chunk-causal attn TFLOP/s and % of GB300 bf16 peak; ms per 1080p chunk"
UNIT = "TFLOP/s"
WORKLOAD = WL.W1080P


def chunk_flops(w: WL.Workload, visible_tokens: int, c: int) -> float:
    """QK^T plus PV over visible pairs: 4 * B * H * Lq * Lk * d."""
    lq = w.frames_in_chunk(c) * w.tokens_per_frame
    return 4.0 * w.batch * w.heads * lq * visible_tokens * w.head_dim


def visible_tokens_per_chunk(w: WL.Workload):
    """Lk of each chunk from the library's own visibility plan (host only)."""
    from paper_2609_36757_gb300 import fastvr as FV
    cfg = FV.config_from_workload(w)
    plan = FV.fastvr_attn_plan(cfg, 1 << 40, FV.fastvr_kv_cache_bytes(cfg))
    out = []
    try:
        for c in range(w.num_chunks):
            FV.fastvr_plan_set_state(plan, c + 1, w.frames_in_chunk(c))
            out.append(FV.fastvr_plan_visible(plan)[1])
    finally:
        FV.fastvr_plan_destroy(plan)
    return out


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0,
            "bf16_tflops_sustained": 1700.0}, "fallback"


def load_profile(kernel: str):
    """The key=value lines of a committed ncu summary
    (profiles/<kernel>_traffic.txt), when that summary was taken on the
    current kernel source (else None)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"{kernel}_traffic.txt")
    if not os.path.exists(path):
        return None
    kv = {}
    for line in open(path):
        if "=" in line and not line.startswith("#"):
            k, v = line.strip().split("=", 1)
            kv[k.strip()] = v.strip()
    src = os.path.join(ROOT, "paper_2609_36757_gb300", "csrc", kv.get("source", ""))
    if not os.path.exists(src):
        return None
    digest = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    if digest != kv.get("source_sha256_16"):
        return None
    return kv


def load_traffic(kernel: str):
    """DRAM bytes per average launch from a committed ncu summary taken on
    the current kernel source (else None)."""
    kv = load_profile(kernel)
    return None if kv is None else float(kv["dram_bytes_per_avg_launch"])


def append_dram(peaks):
    """What DRAM saw during one 1080p kv_append launch (ncu), beside the
    event-timed rate that counts every byte the append reads and writes."""
    kv = load_profile("kv_append_1080p")
    if kv is None:
        return None
    rd = float(kv["dram_read_bytes"])
    wr = float(kv["dram_write_bytes_during_launch"])
    t = float(kv["ncu_time_ns"]) * 1e-9
    return {"read_bytes": rd, "write_bytes_during_launch": wr,
            "algorithmic_bytes": float(kv["algorithmic_read_bytes"]) +
            float(kv["algorithmic_write_bytes"]),
            "ncu_us": t * 1e6, "dram_gbs_during_launch": (rd + wr) / t / 1e9,
            "dram_frac_of_hbm": (rd + wr) / t / 1e9 / peaks["hbm_gbs"],
            "source": "profiles/kv_append_1080p_traffic.txt (ncu)"}


# ------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        self.device_index = device_index

    def start(self):
        try:
            ident = str(self.device_index)
            try:
                ident = "GPU-" + str(torch.cuda.get_device_properties(
                    self.device_index).uuid)
            except Exception:
                pass
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", ident, f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            return None
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx = float(parts[1])
            except ValueError:
                continue
            for n, val in zip(names, parts[4:8]):
                if val.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx,
                "samples": len(sm), "reasons": sorted(reasons)}


# ------------------------------------------------------------- CPU oracle
class OracleSample:
    """The oracle timed on the last chunk of a workload (its largest visible
    window), head 0 of batch 0, in blocks of query rows."""

    def __init__(self, w: WL.Workload, chunks, rows_per_block: int = 256):
        from oracle import attention as OA
        self.OA, self.w, self.rows = OA, w, rows_per_block
        self.c = len(chunks) - 1
        vis = OA.visible_chunks(self.c, w.window_chunks)
        self.k = np.concatenate([chunks[j][1][0, :, 0].float().numpy()
                                 for j in vis]).astype(np.float64)
        self.v = np.concatenate([chunks[j][2][0, :, 0].float().numpy()
                                 for j in vis]).astype(np.float64)
        self.q = chunks[self.c][0][0, :, 0].float().numpy().astype(np.float64)
        self.next_row = 0

    def run(self, seconds: float, max_blocks: int):
        """Returns (TFLOP/s, description)."""
        lk = self.k.shape[0]
        flops, blocks = 0.0, 0
        t0 = time.perf_counter()
        while blocks < max_blocks:
            r0 = self.next_row
            qb = self.q[r0:r0 + self.rows]
            self.next_row = (r0 + self.rows) % self.q.shape[0]
            self.OA.softmax_attention(qb, self.k, self.v, self.w.softmax_scale)
            flops += 4.0 * qb.shape[0] * lk * self.w.head_dim
            blocks += 1
            if time.perf_counter() - t0 >= seconds:
                break
        dt = time.perf_counter() - t0
        desc = (f"oracle fp64 (numpy) on chunk {self.c} of {self.w.name}: "
                f"{blocks} block(s) of {self.rows} query rows x Lk={lk} keys, "
                f"head 0, {dt:.2f} s")
        return flops / dt / 1e12, desc


def host_chunks(w: WL.Workload, seed_offset: int = 0):
    if seed_offset:
        import dataclasses
        w = dataclasses.replace(w, seed=w.seed + seed_offset)
    return [(q, k, v) for _, q, k, v in WL.chunk_stream(w)]


# ------------------------------------------------------------- arms
def run_reference(args, rank: int, world: int) -> None:
    if rank != 0:
        return
    w = WORKLOAD
    sample = OracleSample(w, host_chunks(w))
    for _ in range(args.warmup):
        sample.run(0.0, 1)
    vals = []
    for _ in range(args.steps):
        v, desc = sample.run(0.0, 1)
        vals.append(v)
    value = statistics.median(vals)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic (seeded N(0,1) bf16 inputs)",
        "config": {"workload": w.name, "batch": w.batch, "heads": w.heads,
                   "head_dim": w.head_dim, "tokens_per_frame": w.tokens_per_frame,
                   "frames_per_chunk": w.frames_per_chunk,
                   "chunks": w.num_chunks, "window_chunks": w.window_chunks},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": HOST_CORES,
                         "kind": "oracle", "sample": desc},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_gpu(args, rank: int, world: int, local_rank: int) -> None:
    from paper_2609_36757_gb300 import fastvr as FV
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = WORKLOAD
    lk = visible_tokens_per_chunk(w)
    flops = [chunk_flops(w, lk[c], c) for c in range(w.num_chunks)]
    step_flops = sum(flops)

    chunks = host_chunks(w, seed_offset=rank)
    dq = [q.to(dev) for q, _, _ in chunks]
    dk = [k.to(dev) for _, k, _ in chunks]
    dv = [v.to(dev) for _, _, v in chunks]
    att = FV.StreamingAttention(FV.config_from_workload(w), dev)
    t = time_stream(att, w, dq, dk, dv, args.steps, args.warmup, dev,
                    local_rank if rank == 0 else None, world)
    fwd_ms, app_ms, launches = t["fwd_ms"], t["app_ms"], t["launches"]
    clock_info = t["clocks"]
    max_ms = reduce_max(t["elapsed_ms"], world)
    value = world * step_flops * args.steps / (max_ms / 1e3) / 1e12

    e2e = (None if args.skip_e2e else
           run_e2e(args, w, chunks, att, dev, step_flops, world))
    one_step = measure_one_step(dev)
    del dq, dk, dv, att
    per_workload = None
    if args.per_workload and world == 1:
        peaks, _ = load_peaks()
        per_workload = {name: measure_workload(WL.WORKLOADS[name], dev,
                                               peaks, local_rank)
                        for name in PER_WORKLOADS}
        per_workload[TRAIN_LEG] = measure_train_leg(WL.WORKLOADS[TRAIN_LEG],
                                                    dev, peaks, local_rank)

    if rank != 0:
        return
    peaks, peak_kind = load_peaks()
    fwd_total_ms = sum(map(sum, fwd_ms))
    attn_tflops = step_flops * args.steps / (fwd_total_ms / 1e3) / 1e12
    app_total_ms = sum(map(sum, app_ms))
    # K and V (bf16) read once and written once: read + write bytes, the
    # same accounting as the measured HBM copy peak
    app_bytes = sum(2 * 2 * 2 * w.batch * w.heads * w.frames_in_chunk(c) *
                    w.tokens_per_frame * w.head_dim for c in range(w.num_chunks))
    app_gbs = app_bytes * args.steps / (app_total_ms / 1e3) / 1e9
    per_chunk_fwd = [statistics.median(fwd_ms[s][c] for s in range(args.steps))
                     for c in range(w.num_chunks)]
    peak = peaks["bf16_tflops_sustained"]
    traffic = (load_traffic("chunk_attn_fwd_1080p") if w.name == "1080p"
               else None)
    kv_row = 2 * w.batch * w.heads * w.head_dim * 2  # K+V bytes per token
    qkv_step = sum(3 * w.batch * w.heads * w.head_dim * 2 *
                   w.frames_in_chunk(c) * w.tokens_per_frame
                   for c in range(w.num_chunks))
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": max_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) bf16 Q/K/V, one video per GPU)",
        "config": {"workload": w.name, "batch": w.batch, "heads": w.heads,
                   "head_dim": w.head_dim, "tokens_per_frame": w.tokens_per_frame,
                   "frames_per_chunk": w.frames_per_chunk,
                   "chunks": w.num_chunks, "window_chunks": w.window_chunks,
                   "step": f"reset + {w.num_chunks} x (kv_append + "
                           "chunk_attn_fwd)",
                   "l2": f"inputs larger than L2 (visible K/V per chunk "
                         f"{min(lk) * kv_row / 1e9:.2f}-"
                         f"{max(lk) * kv_row / 1e9:.2f} GB, "
                         f"{qkv_step / 1e9:.2f} GB of Q/K/V per step)",
                   "parallelism": f"replicas x{world} (one video per GPU)"},
        "ms_per_chunk": {"mean_fwd": statistics.mean(per_chunk_fwd),
                         "last_fwd": per_chunk_fwd[-1],
                         "mean_append": app_total_ms / args.steps / w.num_chunks},
        "latent_frames_per_s": world * w.num_frames * args.steps / (max_ms / 1e3),
        "attn_kernel_tflops": attn_tflops,
        "frac_of_burst_peak": attn_tflops / peaks["bf16_tflops"],
        "append_gbs": app_gbs,
        "append_frac_of_hbm": app_gbs / peaks["hbm_gbs"],
        "append_dram": append_dram(peaks) if w.name == "1080p" else None,
        "roofline": {"bound": "tensor", "achieved": attn_tflops, "peak": peak,
                     "unit": "TFLOP/s", "frac": attn_tflops / peak,
                     "peak_kind": f"{peak_kind} bf16 sustained",
                     "kernel": "chunk_attn_fwd (attention + split merge)",
                     "traffic": traffic},
        "gpu_launches": launches,
        "one_step_update": dict(one_step,
                                frac_of_hbm=one_step["gbs"] / peaks["hbm_gbs"]),
        "clocks": clock_info,
        "e2e": e2e,
    }
    if per_workload is not None:
        line["per_workload"] = per_workload
    if world == 1 and args.cpu_seconds > 0:
        cpu_v, desc = OracleSample(w, chunks).run(args.cpu_seconds, 10 ** 6)
        line["cpu_baseline"] = {"value": cpu_v, "unit": UNIT,
                                "cores": HOST_CORES, "kind": "oracle",
                                "sample": desc}
    print(json.dumps(line), flush=True)


def time_stream(att, w, dq, dk, dv, steps, warmup, dev, clock_index, world):
    """Stream w's chunks (device tensors dq/dk/dv) through `att`: `warmup`
    untimed steps, then `steps` timed ones, each reset + per chunk (append,
    forward), with CUDA events on the launching stream around every launch
    and around the whole timed region (bracketed by a barrier and device
    synchronisation).  Clocks are sampled during the timed region when
    clock_index is a device index."""
    from paper_2609_36757_gb300 import fastvr as FV
    douts = [torch.empty_like(q) for q in dq]
    stream = torch.cuda.current_stream(dev)

    def step(ev=None):
        att.reset()
        for c in range(w.num_chunks):
            if ev is not None:
                ev[c][0].record(stream)
            att.append(dk[c], dv[c])
            if ev is not None:
                ev[c][1].record(stream)
            att.forward(dq[c], out=douts[c])
            if ev is not None:
                ev[c][2].record(stream)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize(dev)
    if att.status() != FV.FASTVR_OK:
        raise RuntimeError("device-side failure during warm-up")

    evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(3)]
            for _ in range(w.num_chunks)] for _ in range(steps)]
    clocks = ClockSampler(clock_index) if clock_index is not None else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize(dev)
    launches_before = att.launch_count()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for s in range(steps):
        step(evs[s])
    t_end.record(stream)
    launches = att.launch_count() - launches_before
    torch.cuda.synchronize(dev)
    barrier(world)
    clock_info = clocks.stop() if clocks else None
    if att.status() != FV.FASTVR_OK:
        raise RuntimeError("device-side failure in the timed region")
    return {
        "elapsed_ms": t_start.elapsed_time(t_end),
        "fwd_ms": [[evs[s][c][1].elapsed_time(evs[s][c][2])
                    for c in range(w.num_chunks)] for s in range(steps)],
        "app_ms": [[evs[s][c][0].elapsed_time(evs[s][c][1])
                    for c in range(w.num_chunks)] for s in range(steps)],
        "launches": launches, "clocks": clock_info,
    }


# The other streams of the metric (480p, 720p peaked, windowed 1080p) and the
# paper's own inference shape (k = 3, W = 1, six 64 x 64 latent tiles on B).
PER_WORKLOADS = ("480p", "720p-peaked", "1080p-windowed", "paper-tiles-64x64")


def measure_workload(w, dev, peaks, clock_index, steps: int = 3,
                     warmup: int = 3):
    """One stream's numbers with the headline's method: inputs drawn on the
    device with the workload's recipe (resident in HBM), path TFLOP/s over
    the whole timed region, kernel TFLOP/s over the attention launches'
    events, per-chunk ms, latent frames/s, and the clocks of this leg."""
    from paper_2609_36757_gb300 import fastvr as FV
    lk = visible_tokens_per_chunk(w)
    flops = [chunk_flops(w, lk[c], c) for c in range(w.num_chunks)]
    data = [(q, k, v) for _, q, k, v in WL.chunk_stream(w, device=str(dev))]
    dq, dk, dv = ([x[i] for x in data] for i in range(3))
    att = FV.StreamingAttention(FV.config_from_workload(w), dev)
    t = time_stream(att, w, dq, dk, dv, steps, warmup, dev, clock_index, 1)
    del data, dq, dk, dv, att
    torch.cuda.empty_cache()
    path = sum(flops) * steps / (t["elapsed_ms"] / 1e3) / 1e12
    kernel = sum(flops) * steps / (sum(map(sum, t["fwd_ms"])) / 1e3) / 1e12
    per_chunk = [statistics.median(t["fwd_ms"][s][c] for s in range(steps))
                 for c in range(w.num_chunks)]
    return {
        "steps": steps, "warmup": warmup,
        "shape": {"batch": w.batch, "heads": w.heads, "head_dim": w.head_dim,
                  "tokens_per_frame": w.tokens_per_frame,
                  "frames_per_chunk": w.frames_per_chunk,
                  "chunks": w.num_chunks, "window_chunks": w.window_chunks,
                  "last_chunk_frames": w.last_chunk_frames or
                  w.frames_per_chunk, "peaked": w.peaked},
        "flops_per_step": sum(flops),
        "path_tflops": path, "kernel_tflops": kernel,
        "ms_per_chunk": {"mean_fwd": statistics.mean(per_chunk),
                         "last_fwd": per_chunk[-1],
                         "mean_step_per_chunk": t["elapsed_ms"] / steps /
                         w.num_chunks},
        "latent_frames_per_s": w.num_frames * steps / (t["elapsed_ms"] / 1e3),
        "kernel_frac_of_sustained": kernel / peaks["bf16_tflops_sustained"],
        "kernel_frac_of_burst": kernel / peaks["bf16_tflops"],
        "gpu_launches": t["launches"], "clocks": t["clocks"],
    }


def measure_one_step(dev, sets: int = 8, rounds: int = 3):
    """The one-step update z_hat = z_LQ - sigma v (Eq. one_step, outside the
    attention step) on 1080p-sized latents: 48 channels x 30 latent frames x
    68 x 120, bf16.  Successive calls rotate over `sets` distinct latents
    (8 x 70 MB, larger than L2), timed with CUDA events; bytes = read z and
    v, write z_hat."""
    from paper_2609_36757_gb300 import fastvr as FV
    n = 48 * 30 * 68 * 120
    bufs = [(torch.randn(n, device=dev).to(torch.bfloat16),
             torch.randn(n, device=dev).to(torch.bfloat16),
             torch.empty(n, device=dev, dtype=torch.bfloat16))
            for _ in range(sets)]
    for z, v, out in bufs:
        FV.one_step_update(z, v, 0.8, out=out)
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record()
    for _ in range(rounds):
        for z, v, out in bufs:
            FV.one_step_update(z, v, 0.8, out=out)
    end.record()
    torch.cuda.synchronize(dev)
    us = start.elapsed_time(end) * 1e3 / (rounds * sets)
    return {"elements": n, "us": us, "gbs": 3 * 2 * n / (us * 1e-6) / 1e9,
            "l2": f"{sets} distinct latents rotated ({sets * 6 * n / 1e6:.0f} MB)"}


def measure_oneshot(w, q, k, v, dev, steps: int, warmup: int, clock_index,
                    world: int = 1, train: bool = True):
    """Median CUDA-event times of the one-shot forward and (train) backward
    over `steps` timed calls on resident inputs [B, L, H, d], after
    `warmup` untimed ones, with the clocks sampled meanwhile.  dO is drawn
    on the device from a generator seeded with the workload's seed."""
    from paper_2609_36757_gb300 import fastvr as FV
    g = torch.Generator(device=dev)
    g.manual_seed(w.seed + 1)
    do = torch.randn(q.shape, generator=g, device=dev).to(torch.bfloat16)
    cfg = FV.config_from_workload(w)
    stream = torch.cuda.current_stream(dev)

    def step(ev):
        ev[0].record(stream)
        o, lse = FV.blockcausal_attention(cfg, q, k, v, want_lse=True)
        ev[1].record(stream)
        if train:
            FV.blockcausal_attention_bwd(cfg, q, k, v, o, do, lse)
        ev[2].record(stream)

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)]
           for _ in range(warmup + steps)]
    for i in range(warmup):
        step(evs[i])
    torch.cuda.synchronize(dev)
    clocks = ClockSampler(clock_index) if clock_index is not None else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    barrier(world)
    for i in range(warmup, warmup + steps):
        step(evs[i])
    torch.cuda.synchronize(dev)
    barrier(world)
    clock_info = clocks.stop() if clocks else None
    timed = evs[warmup:]
    return {"fwd_ms": statistics.median(e[0].elapsed_time(e[1]) for e in timed),
            "bwd_ms": statistics.median(e[1].elapsed_time(e[2]) for e in timed),
            "clocks": clock_info}


def oneshot_flops(w) -> float:
    """Forward FLOPs of the one-shot form: 4 B H d x visible pairs."""
    lk = visible_tokens_per_chunk(w)
    return sum(chunk_flops(w, lk[c], c) for c in range(w.num_chunks))


# The training form in the default line: forward + backward of the training
# clip (one shot, Eq. 1 with W = 1).
TRAIN_LEG = "train-1024-clip"


def measure_train_leg(w, dev, peaks, clock_index, steps: int = 5,
                      warmup: int = 3):
    """Forward and backward TFLOP/s of the one-shot form on `w`, inputs drawn
    on the device with the workload's recipe; the backward counted as 2.5 x
    the forward FLOPs (the five products a backward needs)."""
    data = [(q, k, v) for _, q, k, v in WL.chunk_stream(w, device=str(dev))]
    q, k, v = (torch.cat([x[i] for x in data], 1) for i in range(3))
    del data
    t = measure_oneshot(w, q, k, v, dev, steps, warmup, clock_index)
    del q, k, v
    torch.cuda.empty_cache()
    f = oneshot_flops(w)
    fwd = f / (t["fwd_ms"] / 1e3) / 1e12
    bwd = 2.5 * f / (t["bwd_ms"] / 1e3) / 1e12
    return {
        "steps": steps, "warmup": warmup,
        "shape": {"batch": w.batch, "heads": w.heads, "head_dim": w.head_dim,
                  "tokens": w.num_tokens, "frames_per_chunk": w.frames_per_chunk,
                  "window_chunks": w.window_chunks},
        "fwd_flops": f, "bwd_flops": 2.5 * f,
        "fwd_ms": t["fwd_ms"], "bwd_ms": t["bwd_ms"],
        "fwd_tflops": fwd, "bwd_tflops": bwd,
        "fwd_frac_of_burst": fwd / peaks["bf16_tflops"],
        "bwd_frac_of_burst": bwd / peaks["bf16_tflops"],
        "clocks": t["clocks"],
    }


def run_oneshot(args, rank: int, world: int, local_rank: int) -> None:
    """One-shot (training) form over a whole sequence: forward, and in
    `train` mode the backward too.  FLOPs: forward 4 B H d x visible pairs;
    backward 2.5 x that (five products of the same size: S recomputed, dP,
    dV, dQ, dK; the kernels compute two more to avoid atomics, not counted)."""
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = WORKLOAD
    fwd_flops = oneshot_flops(w)
    chunks = host_chunks(w, seed_offset=rank)
    q, k, v = (torch.cat([c[i] for c in chunks], 1).to(dev) for i in range(3))
    train = args.mode == "train"
    t = measure_oneshot(w, q, k, v, dev, args.steps, args.warmup,
                        local_rank if rank == 0 else None, world, train)
    fwd_ms, bwd_ms, clock_info = t["fwd_ms"], t["bwd_ms"], t["clocks"]
    step_ms = reduce_max(fwd_ms + bwd_ms, world)
    if rank != 0:
        return
    peaks, peak_kind = load_peaks()
    total = fwd_flops * (3.5 if train else 1.0)
    value = world * total / (step_ms / 1e3) / 1e12
    line = {
        "metric": ("one-shot chunk-causal attn fwd+bwd TFLOP/s" if train else
                   "one-shot chunk-causal attn fwd TFLOP/s"),
        "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (seeded N(0,1) bf16 Q/K/V/dO)",
        "config": {"workload": w.name, "batch": w.batch, "heads": w.heads,
                   "head_dim": w.head_dim, "tokens": w.num_tokens,
                   "frames_per_chunk": w.frames_per_chunk,
                   "window_chunks": w.window_chunks, "mode": args.mode},
        "clocks": clock_info,
        "fwd_ms": fwd_ms, "fwd_tflops": fwd_flops / (fwd_ms / 1e3) / 1e12,
        "fwd_frac_of_burst_peak": fwd_flops / (fwd_ms / 1e3) / 1e12 /
                                  peaks["bf16_tflops"],
    }
    if train:
        line["bwd_ms"] = bwd_ms
        line["bwd_tflops"] = 2.5 * fwd_flops / (bwd_ms / 1e3) / 1e12
        line["bwd_frac_of_burst_peak"] = line["bwd_tflops"] / peaks["bf16_tflops"]
    print(json.dumps(line), flush=True)


def run_e2e(args, w, chunks, att, dev, step_flops, world):
    """The same metric through the public API from pinned host buffers: every
    step copies each chunk's Q/K/V host->device and each output device->host,
    on two side streams, through a ring of three device slots, so that a
    chunk's inputs load while the previous chunk computes; the ring and its
    events carry over from one step to the next, so the next step's first
    chunk also loads while this step's last one computes."""
    kSlots = 3
    pq = [q.pin_memory() for q, _, _ in chunks]
    pk = [k.pin_memory() for _, k, _ in chunks]
    pv = [v.pin_memory() for _, _, v in chunks]
    po = [torch.empty_like(q).pin_memory() for q in pq]
    slots = [[torch.empty_like(pq[0], device=dev) for _ in range(3)]
             for _ in range(kSlots)]
    outs = [torch.empty_like(pq[0], device=dev) for _ in range(kSlots)]
    compute = torch.cuda.current_stream(dev)
    h2d = torch.cuda.Stream(dev)
    d2h = torch.cuda.Stream(dev)
    h2d_bytes = sum(t.numel() * 2 for t in pq + pk + pv)
    d2h_bytes = sum(t.numel() * 2 for t in po)
    # free[s]: the slot's inputs are consumed; out_free[s]: its output is out
    free = [torch.cuda.Event() for _ in range(kSlots)]
    out_free = [torch.cuda.Event() for _ in range(kSlots)]
    for e in free + out_free:
        e.record(compute)
    used = [0]

    def step():
        att.reset()
        for c in range(w.num_chunks):
            s = used[0] % kSlots
            used[0] += 1
            L = pq[c].shape[1]
            sq, sk, sv = (x[:, :L] for x in slots[s])
            with torch.cuda.stream(h2d):
                h2d.wait_event(free[s])
                sq.copy_(pq[c], non_blocking=True)
                sk.copy_(pk[c], non_blocking=True)
                sv.copy_(pv[c], non_blocking=True)
                ready = torch.cuda.Event()
                ready.record(h2d)
            compute.wait_event(ready)
            compute.wait_event(out_free[s])
            att.append(sk, sv)
            o = outs[s][:, :L]
            att.forward(sq, out=o)
            free[s].record(compute)
            done = torch.cuda.Event()
            done.record(compute)
            with torch.cuda.stream(d2h):
                d2h.wait_event(done)
                po[c].copy_(o, non_blocking=True)
                out_free[s].record(d2h)

    for _ in range(max(1, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    rank0 = int(os.environ.get("RANK", "0")) == 0
    clocks = ClockSampler(dev.index) if rank0 and dev.index is not None else None
    if clocks:
        clocks.start()
        time.sleep(0.3)
    barrier(world)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    torch.cuda.synchronize(dev)
    barrier(world)
    dt = reduce_max(time.perf_counter() - t0, world)
    clock_info = clocks.stop() if clocks else None
    return {"value": world * step_flops * args.steps / dt / 1e12, "unit": UNIT,
            "h2d_bytes_per_step": h2d_bytes, "d2h_bytes_per_step": d2h_bytes,
            "clocks": clock_info}


# ------------------------------------------------------------- distributed
def barrier(world: int) -> None:
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def reduce_max(x: float, world: int) -> float:
    if world <= 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def main(argv=None):
    global WORKLOAD
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="fastvr", choices=["fastvr", "reference"])
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="CPU-baseline sample length (0 skips it)")
    ap.add_argument("--workload", default=WORKLOAD.name,
                    choices=sorted(WL.WORKLOADS),
                    help="workload to stream (the metric is quoted on 1080p)")
    ap.add_argument("--chunks", type=int, default=0,
                    help="stream only the first N chunks (small profiling "
                         "cases); 0 = the whole workload")
    ap.add_argument("--mode", default="stream",
                    choices=["stream", "oneshot", "train"],
                    help="stream: the streaming metric (default); oneshot / "
                         "train: the whole sequence at once, forward / "
                         "forward + backward (extra measurements)")
    ap.add_argument("--skip-e2e", action="store_true",
                    help="omit the end-to-end leg (profiling cases)")
    ap.add_argument("--no-per-workload", dest="per_workload",
                    action="store_false",
                    help="omit the per-workload legs (480p, 720p peaked, "
                         "windowed 1080p, paper tiles) run after the "
                         "headline at N = 1")
    args = ap.parse_args(argv)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    WORKLOAD = WL.WORKLOADS[args.workload]
    if args.chunks:
        import dataclasses
        WORKLOAD = dataclasses.replace(WORKLOAD, num_chunks=args.chunks,
                                       name=f"{WORKLOAD.name}-first{args.chunks}")
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    try:
        if args.mode == "stream":
            run_gpu(args, rank, world, local_rank)
        else:
            run_oneshot(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
