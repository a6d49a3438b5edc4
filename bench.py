"""Benchmark of the action-expert tick (one step = one tick of the whole hot
path: embed, 32 x [RMSNorm+QKV, Eq. 1 attention, W_o, RMSNorm+SwiGLU, W_d],
head) on synthetic seeded inputs, printed as one JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl fsx|reference]

Default workload: bf16_b128_ragged, the largest single-GPU configuration: 128
vehicles with ragged caches L_b ~ U[64, 2048] (the seeded draw holds 129,767
cached tokens per layer, 68 GB over 32 layers), bf16 weights / cache / frames.
value = vehicle-ticks/s over all ranks (weak scaling: every rank runs its own
vehicles; the path has no cross-vehicle exchange). The same line carries, under
"workloads", the B = 1 paper-shaped tick (bf16_b1_l224), the history-length
sweep at B = 1 (L = 224 ... 4096) and the 16-vehicle batch, each with its
us/tick and its fraction of the max(HBM, tensor) tick roofline. Inputs are
resident in HBM when the timed region starts; weights (675 MB) plus cache
exceed the 129 MB L2, so no flush is needed between ticks.

The workload `clip_j40_delta1` times the staleness-masked forward over a 40-frame
clip (Sec. 3.2: every frame block over the cache prefix ending one frame earlier,
all blocks in one tick over explicit row ranges); value = frame-blocks/s.
The workload `fastslow_b1_l224` paces one vehicle's ticks (every 12.5 ms) with a cache
append before every 4th tick through an fsx session (Sec. 3.3) and reports the tick
latency distribution in the serial and the concurrent schedule.
The workload `paper_b1_l224` times the paper's own ten-token layout (state token,
four visual tokens, five queries, two-layer head; Sec. 3.1) at B = 1, L = 224.
The workload `append_b1_l224` instead times the backbone's incremental cache
append (one call = n_new = 4 tokens through the 32-layer, 4096-wide backbone
for one vehicle with 224 cached tokens); value = vehicle-appends/s.

Without torchrun (WORLD_SIZE unset), --gpus N > 1 starts N ranks itself, one
per GPU, and rank 0 prints the line.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "vehicle-ticks/s (1e6 / us-per-tick x B) of the action-expert tick"
UNIT = "vehicle-ticks/s"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_TENSOR_TFS = 1700.0      # dense bf16 / fp16, sustained (one earlier GB300 measurement)
NOMINAL_HBM_GBS = 8000.0          # the HBM3e figure the tick roofline is stated against
NOMINAL_TENSOR_TFS = 2250.0       # dense bf16 / fp16 tensor peak, nominal
KCLASS_NAMES = ["qkv", "attention", "out_proj", "gate_up", "down", "persistent"]
DEFAULT_WORKLOAD = "bf16_b128_ragged"
# timed beside the headline with the same handle: the B = 1 paper-shaped tick, the
# history-length sweep and the 16-vehicle batch
EXTRA_WORKLOADS = ["bf16_b1_l224", "bf16_b1_l512", "bf16_b1_l1024", "bf16_b1_l2048", "bf16_b1_l4096",
                   "bf16_b16_ragged"]

# DRAM bytes (read + write) of one launch of the timed kernel, from one ncu capture, with the
# SHA-256 prefix of the kernel's source file at capture time: a figure whose source has
# changed since is reported as null (traffic_stale).
NCU_TRAFFIC = {
    ("attention", "bf16_b128_ragged"): (2258.315e6 + 39.520768e6, "attention_tc.cu", "d912fb0f53ded610"),
}


def traffic_for(kclass, workload):
    """(bytes, stale) of the timed kernel's last ncu capture, (None, False) when none exists."""
    import hashlib
    entry = NCU_TRAFFIC.get((kclass, workload))
    if entry is None:
        return None, False
    nbytes, src, sha = entry
    path = os.path.join(ROOT, "paper_2607_15621_gb300", "csrc", src)
    try:
        with open(path, "rb") as fh:
            cur = hashlib.sha256(fh.read()).hexdigest()[:16]
    except OSError:
        return None, True
    return (nbytes, False) if cur == sha else (None, True)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", default="fsx", choices=["fsx", "reference"])
    ap.add_argument("--kernel-class", default=None, choices=KCLASS_NAMES,
                    help="kernel timed for the roofline (default: the dominant one, i.e. the persistent tick "
                         "for one vehicle and attention for a batch)")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="time only the named workload (no B = 1, sweep and B = 16 entries)")
    ap.add_argument("--layers", type=int, default=None,
                    help="expert layers (default: the workload's 32); fewer layers keep a profiling run's cache small")
    return ap.parse_args()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value: float, device=None) -> float:
    """Largest `value` over the ranks of the default process group (the value itself
    when no group is initialised): the job's time is its slowest rank's time."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def peaks():
    """HBM copy GB/s and sustained dense bf16 TF/s of this GPU (fp16 runs at the bf16 rate)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            p = json.load(fh)
        hbm = float(p["hbm_gbs"])
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_TENSOR_TFS, "fallback"
    tfs = p.get("bf16_tflops_sustained", p.get("bf16_tflops"))
    return hbm, float(tfs) if tfs else FALLBACK_TENSOR_TFS, "measured"


def workload_info(name):
    from paper_2607_15621_gb300 import synth
    spec = synth.WORKLOADS[name]
    lengths = synth.cache_lengths(name, 0)
    return spec, lengths


def algorithmic_bytes(dims, lengths, cache_dtype, weight_bytes):
    """Per tick: expert weights once + every vehicle's cache rows once at every layer."""
    elem = 2 if cache_dtype == "bf16" else 4
    kv = int(np.sum(lengths)) * dims.n_layers * 2 * dims.hd * elem
    return weight_bytes + kv, kv


def tick_flops(dims, lengths):
    """Per tick: the projection GEMMs (2 flop per weight per token) of every layer plus
    Eq. 1 (Q K^T and P V over the cache and own keys: 4 T D flop per key, head and layer)."""
    T, d, hd, f = dims.n_tok, dims.d_model, dims.hd, dims.d_ff
    B = len(lengths)
    per_layer_w = 3 * hd * d + d * hd + 2 * f * d + d * f
    gemm = 2 * B * T * per_layer_w * dims.n_layers
    keys = int(np.sum(lengths)) + B * T
    attn = 4 * T * dims.head_dim * dims.n_heads * keys * dims.n_layers
    return gemm + attn


def clock_dir():
    """Where the raw nvidia-smi samples of the timed region go (FSX_CLOCKS_DIR, else a
    temporary directory); the JSON line carries their summary."""
    import tempfile
    return os.environ.get("FSX_CLOCKS_DIR") or tempfile.gettempdir()


def start_clock_sampler(path, index):
    try:
        fh = open(path, "w")
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        proc = subprocess.Popen(["nvidia-smi", f"--id={index}", f"--query-gpu={q}", "--format=csv,noheader,nounits",
                                 "-lms", "200"], stdout=fh, stderr=subprocess.DEVNULL)
        return proc, fh
    except Exception:
        return None, None


def stop_clock_sampler(proc, fh, path):
    if proc is None:
        return None
    proc.terminate()
    try:
        proc.wait(timeout=5)
    except Exception:
        proc.kill()
    fh.close()
    sm, smax, reasons = [], [], set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    with open(path) as f:
        for line in f:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
    if not sm:
        return None
    return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
            "samples": len(sm)}


def baseline_vehicles(lengths, n=8):
    """The vehicles the CPU baseline runs: for one vehicle that one; for a batch, n of
    them spread over the length order, the shortest and the longest included."""
    lengths = np.asarray(lengths)
    if len(lengths) == 1:
        return [0]
    order = np.argsort(lengths, kind="stable")
    picks = np.unique(np.round(np.linspace(0, len(order) - 1, min(n, len(order)))).astype(int))
    return [int(order[i]) for i in picks]


def cpu_baseline(name, seconds):
    """The fp64 oracle as it stands, on the host cores. One vehicle: vehicle 0's tick
    repeated for `seconds`. A batch: one tick of each of 8 vehicles spread over the
    length order (shortest and longest included), each over its own seeded draw of a
    cache of its length (the batch's 68 GB cache is not copied to the host), stopping
    early only past 4 x `seconds`; vehicles are independent, so the rate is per
    vehicle-tick of that mix."""
    from oracle import fsx_oracle
    from paper_2607_15621_gb300 import synth
    spec, lengths = workload_info(name)
    dims = synth.EXPERT
    w = synth.make_weights(dims, 0, spec["dtype"])
    picks = baseline_vehicles(lengths)

    def inputs(b):
        k, v, off = synth.make_cache(dims, [int(lengths[b])], 1000 + b, spec["dtype"])
        fr = synth.make_frames(dims, 1, 1000 + b, spec["dtype"]).double().numpy()
        return [t.float().numpy() for t in k], [t.float().numpy() for t in v], off, fr

    n, done, t0 = 0, [], time.perf_counter()
    if len(picks) == 1:
        kn, vn, off, fr = inputs(0)
        t0 = time.perf_counter()
        while True:
            fsx_oracle.expert_tick(w, kn, vn, off, fr, dims.n_heads, dims.head_dim, dims.n_waypoints)
            n += 1
            el = time.perf_counter() - t0
            if el >= seconds or n >= 1000:
                break
        sample = f"{n} full 32-layer fp64 ticks of vehicle 0 of {name} (L={int(lengths[0])}) in {el:.1f} s"
    else:
        el = 0.0
        for b in picks:
            kn, vn, off, fr = inputs(b)
            t1 = time.perf_counter()
            fsx_oracle.expert_tick(w, kn, vn, off, fr, dims.n_heads, dims.head_dim, dims.n_waypoints)
            el += time.perf_counter() - t1
            n += 1
            done.append(int(lengths[b]))
            if el >= 4 * seconds:
                break
        sample = (f"one full 32-layer fp64 tick of each of {n} vehicles of {name} spread over the length order "
                  f"(L = {done}), each over its own seeded cache draw, {el:.1f} s of oracle time")
    return {"value": n / el, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle", "sample": sample}


APPEND_METRIC = "vehicle-appends/s (1e6 / us-per-append x B) of the backbone's incremental cache append"
APPEND_UNIT = "vehicle-appends/s"


def append_inputs(args, device):
    """Backbone dims, weights, per-layer caches (cached rows then room for the new
    rows), offsets, destination rows and new-token embeddings of an append workload."""
    import torch
    from paper_2607_15621_gb300 import synth
    spec = synth.APPEND_WORKLOADS[args.workload]
    dims = synth.BACKBONE if args.layers is None else dataclasses.replace(synth.BACKBONE, n_layers=args.layers)
    B, L, n = spec["batch"], spec["length"], dims.n_new
    w = synth.make_backbone_weights(dims, 0, "bf16")
    cache_dims = synth.Dims(n_layers=dims.n_layers, n_heads=dims.n_heads, head_dim=dims.head_dim)
    k, v, off = synth.make_cache(cache_dims, [L] * B, 0, "bf16", device=device)
    rows = B * (L + n)
    kc, vc = [], []
    for kl, vl in zip(k, v):
        kt = torch.zeros(rows, dims.n_heads, dims.head_dim, dtype=torch.bfloat16, device=device)
        vt = torch.zeros_like(kt)
        kt[:B * L] = kl
        vt[:B * L] = vl
        kc.append(kt)
        vc.append(vt)
    dst = np.array([B * L + n * b for b in range(B)], dtype=np.int64)
    x = synth.make_append_tokens(dims, B, 0, device=device)
    return dims, w, kc, vc, off, dst, x, B, L


def append_cpu_baseline(args, dims, w, kc, vc, off, x, seconds):
    """The fp64 append oracle as it stands, on the host cores: vehicle 0's append."""
    from oracle import append_oracle
    lo, hi = int(off[0]), int(off[1])
    kn = [t[lo:hi].float().cpu().numpy() for t in kc]
    vn = [t[lo:hi].float().cpu().numpy() for t in vc]
    xn = x[:1].float().cpu().numpy()
    n, t0 = 0, time.perf_counter()
    while True:
        append_oracle.backbone_append(w, kn, vn, np.array([0, hi - lo]), xn, dims.n_heads, dims.head_dim)
        n += 1
        el = time.perf_counter() - t0
        if el >= seconds or n >= 1000:
            break
    return {"value": n / el, "unit": APPEND_UNIT, "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{n} full {dims.n_layers}-layer fp64 appends of vehicle 0 of {args.workload} "
                      f"(L={hi - lo}) in {el:.1f} s"}


def run_append_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    dims, w, kc, vc, off, dst, x, B, L = append_inputs(args, "cpu")
    cb = append_cpu_baseline(args, dims, w, kc, vc, off, x, max(1.0, min(args.cpu_seconds, 60.0)))
    line = {"impl": "reference", "metric": APPEND_METRIC, "value": cb["value"], "unit": APPEND_UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 / cb["value"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)",
            "config": {"workload": args.workload, "B": B, "cache_len": L, "layers": dims.n_layers,
                       "d_model": dims.d_model, "new_tokens": dims.n_new, "parallelism": f"replicas x{world}",
                       "sample": "vehicle 0 per step; vehicles are independent"},
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": APPEND_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def run_append(args):
    """The cache append on the GPU: CUDA events around K calls, inputs resident in HBM."""
    import torch
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_15621_gb300 import fsx
    dims, w, kc, vc, off, dst, x, B, L = append_inputs(args, dev)
    rows = kc[0].shape[0]
    offsets = torch.as_tensor(off, device=dev)
    dst_t = torch.as_tensor(dst, device=dev)
    hidden = torch.empty(B, dims.n_new, dims.d_model, device=dev)
    ap = fsx.Append(dims, w, B, rows, device=local)
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    # every call writes the same destination rows, so each timed call is a full append
    for _ in range(max(args.warmup, 3)):
        ap.append(kc, vc, offsets, dst_t, x, hidden, stream)
    torch.cuda.synchronize()
    if ap.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during warm-up")
    clock_path = os.path.join(clock_dir(), f"clocks_rank{rank}.csv")
    os.makedirs(os.path.dirname(clock_path), exist_ok=True)
    proc, fh = start_clock_sampler(clock_path, local)
    time.sleep(0.5)
    barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        ap.append(kc, vc, offsets, dst_t, x, hidden, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms = max_over_ranks(e0.elapsed_time(e1), dev)
    clocks = stop_clock_sampler(proc, fh, clock_path)
    if ap.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during the timed region")
    ms_per_step = ms / args.steps

    # end to end: new-token embeddings in from pinned host memory, hidden states back
    x_h = x.cpu().pin_memory()
    hid_h = torch.empty(B, dims.n_new, dims.d_model).pin_memory()
    e2e_steps = max(1, args.steps // 2)
    barrier()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        x.copy_(x_h, non_blocking=True)
        ap.append(kc, vc, offsets, dst_t, x, hidden, stream)
        hid_h.copy_(hidden, non_blocking=True)
        stream.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, dev)

    hbm, tensor_tfs, peak_kind = peaks()
    hd = dims.hd
    per_layer_w = 3 * hd * dims.d_model + dims.d_model * hd + 3 * dims.d_ff * dims.d_model
    cache_bytes = B * (L + dims.n_new) * dims.n_layers * 2 * hd * 2   # cached rows read + new rows written
    call_bytes = ap.weight_bytes() + cache_bytes
    flops = (2 * B * dims.n_new * per_layer_w + 4 * B * dims.n_new * hd * (L + dims.n_new)) * dims.n_layers
    achieved = call_bytes / (ms_per_step / 1e3) / 1e9
    rl_us = max(call_bytes / (hbm * 1e9), flops / (tensor_tfs * 1e12)) * 1e6
    line = {
        "metric": APPEND_METRIC, "value": world * B / (ms_per_step / 1e3), "unit": APPEND_UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step,
        "us_per_append": ms_per_step * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f16 (fp32 accumulate)", "data": "synthetic (seeded N(0,1/fan_in) weights, N(0,1) cache and tokens)",
        "config": {"workload": args.workload, "B": B, "cache_len": L, "layers": dims.n_layers,
                   "d_model": dims.d_model, "new_tokens": dims.n_new,
                   "l2": "inputs larger than L2 (the backbone weights exceed 129 MB)",
                   "parallelism": f"replicas x{world}"},
        "gpu_launches": (1 + 7 * dims.n_layers) * args.steps,
        "roofline": {"bound": "hbm", "kernel": "append (whole call)", "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": achieved / hbm, "traffic": None, "peak_source": peak_kind,
                     "bytes_per_launch": call_bytes, "launch_us": ms_per_step * 1e3,
                     "flops_per_call": flops, "roofline_us": rl_us},
        "e2e": {"value": world * B * e2e_steps / e2e_s, "unit": APPEND_UNIT,
                "h2d_bytes_per_step": int(x_h.numel() * x_h.element_size()),
                "d2h_bytes_per_step": int(hid_h.numel() * hid_h.element_size())},
        "clocks": clocks,
    }
    ap.close()
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = append_cpu_baseline(args, dims, w, kc, vc, off, x, args.cpu_seconds)
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


CLIP_METRIC = "frame-blocks/s of the staleness-masked clip forward (all frames of a clip in one tick)"
CLIP_UNIT = "frame-blocks/s"


def clip_inputs(args, device):
    """Expert dims and weights, the clip's cache (one buffer), the blocks' prefix lengths
    as offsets, zero start rows and the blocks' frame tokens."""
    from paper_2607_15621_gb300 import synth
    c = synth.CLIP_WORKLOADS[args.workload]
    dims = synth.EXPERT if args.layers is None else dataclasses.replace(synth.EXPERT, n_layers=args.layers)
    prefix = synth.clip_prefixes(args.workload)
    rows = c["text"] + c["tokens_per_frame"] * c["frames"]
    w = synth.make_weights(dims, 0, "bf16")
    k, v, _ = synth.make_cache(dims, [rows], 0, "bf16", device=device)
    off = np.concatenate([[0], np.cumsum(prefix)]).astype(np.int64)
    frames = synth.make_frames(dims, c["frames"], 0, "bf16", device=device)
    return dims, w, k, v, off, prefix, frames, rows, c


def run_clip_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    from oracle import fsx_oracle, staleness_oracle
    dims, w, k, v, off, prefix, frames, rows, c = clip_inputs(args, "cpu")
    kn = [t.float().numpy() for t in k]
    vn = [t.float().numpy() for t in v]
    fr = frames.double().numpy()
    seconds = max(1.0, min(args.cpu_seconds, 60.0))
    # a bounded sample: frame blocks spread evenly over the clip (every stride-th block, so
    # the sampled prefix lengths follow the clip's own mix), each one fp64 tick over the
    # prefix the staleness rule gives it; the per-block rate scales to the whole clip
    J = c["frames"]
    stride = 4
    order = list(range(0, J, stride)) + [j for j in range(J) if j % stride]
    n_blocks, t0 = 0, time.perf_counter()
    for j in order:
        pj = staleness_oracle.visible_prefix(j, c["delta"], c["text"], c["tokens_per_frame"])
        fsx_oracle.expert_tick(w, [t[:pj] for t in kn], [t[:pj] for t in vn], np.array([0, pj]), fr[j:j + 1],
                               dims.n_heads, dims.head_dim, dims.n_waypoints)
        n_blocks += 1
        if time.perf_counter() - t0 >= seconds:
            break
    el = time.perf_counter() - t0
    cb = {"value": n_blocks / el, "unit": CLIP_UNIT, "cores": os.cpu_count(), "kind": "oracle",
          "sample": f"{n_blocks} of {J} frame blocks of {args.workload} (every {stride}th block first, each over "
                    f"its staleness prefix), fp64, in {el:.1f} s; one clip = {J} blocks"}
    line = {"impl": "reference", "metric": CLIP_METRIC, "value": cb["value"], "unit": CLIP_UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * J / cb["value"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)",
            "config": {"workload": args.workload, "frames": J, "text": c["text"], "delta": c["delta"],
                       "layers": dims.n_layers, "parallelism": f"replicas x{world}"},
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": CLIP_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def run_clip(args):
    """All frame blocks of one clip in one ranged tick on the GPU (CUDA events over K ticks)."""
    import torch
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_15621_gb300 import fsx
    dims, w, k, v, off, prefix, frames, rows, c = clip_inputs(args, dev)
    J = c["frames"]
    offsets = torch.as_tensor(off, device=dev)
    starts = torch.zeros(J, dtype=torch.int64, device=dev)
    out = torch.empty(J, dims.n_waypoints, 2, device=dev)
    ex = fsx.Expert(dims, w, J, rows, "bf16", "bf16", device=local)
    weight_bytes = ex.weight_bytes()
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    for _ in range(max(args.warmup, 3)):
        ex.tick(k, v, offsets, frames, out, stream, starts=starts)
    torch.cuda.synchronize()
    if ex.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during warm-up")
    clock_path = os.path.join(clock_dir(), f"clocks_rank{rank}.csv")
    os.makedirs(os.path.dirname(clock_path), exist_ok=True)
    proc, fh = start_clock_sampler(clock_path, local)
    time.sleep(0.5)
    barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        ex.tick(k, v, offsets, frames, out, stream, starts=starts)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms = max_over_ranks(e0.elapsed_time(e1), dev)
    clocks = stop_clock_sampler(proc, fh, clock_path)
    if ex.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during the timed region")
    ms_per_step = ms / args.steps

    # end to end: the blocks' frame tokens in from pinned host memory, waypoints back
    fr_h = frames.cpu().pin_memory()
    out_h = torch.empty(J, dims.n_waypoints, 2).pin_memory()
    e2e_steps = max(1, args.steps // 2)
    barrier()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        frames.copy_(fr_h, non_blocking=True)
        ex.tick(k, v, offsets, frames, out, stream, starts=starts)
        out_h.copy_(out, non_blocking=True)
        stream.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, dev)

    hbm, tensor_tfs, peak_kind = peaks()
    # HBM bytes: the expert weights once plus the distinct cache rows the blocks read (the
    # longest prefix) once per layer; the blocks' overlapping prefixes are L2 re-reads of
    # those rows, reported separately as logical bytes
    tick_bytes, _ = algorithmic_bytes(dims, [int(np.max(prefix))], "bf16", weight_bytes)
    logical_bytes, _ = algorithmic_bytes(dims, prefix, "bf16", weight_bytes)
    flops = tick_flops(dims, prefix)
    achieved = tick_bytes / (ms_per_step / 1e3) / 1e9
    rl_us = max(tick_bytes / (hbm * 1e9), flops / (tensor_tfs * 1e12)) * 1e6
    line = {
        "metric": CLIP_METRIC, "value": world * J / (ms_per_step / 1e3), "unit": CLIP_UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step,
        "us_per_clip": ms_per_step * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f16 (fp32 accumulate)", "data": "synthetic (seeded N(0,1) cache/frames, N(0,1/fan_in) weights)",
        "config": {"workload": args.workload, "frames": J, "text": c["text"], "delta": c["delta"],
                   "layers": dims.n_layers, "cache_rows": rows,
                   "l2": "inputs larger than L2 (the expert weights exceed 129 MB)",
                   "parallelism": f"replicas x{world}"},
        "gpu_launches": ex.launches(J) * args.steps,
        "roofline": {"bound": "hbm", "kernel": "clip tick (whole graph)", "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": achieved / hbm, "traffic": None, "peak_source": peak_kind,
                     "bytes_per_launch": tick_bytes, "logical_bytes_per_launch": logical_bytes,
                     "launch_us": ms_per_step * 1e3, "flops_per_tick": flops, "roofline_us": rl_us},
        "e2e": {"value": world * J * e2e_steps / e2e_s, "unit": CLIP_UNIT,
                "h2d_bytes_per_step": int(fr_h.numel() * fr_h.element_size()),
                "d2h_bytes_per_step": int(out_h.numel() * out_h.element_size())},
        "clocks": clocks,
    }
    ex.close()
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


PAPER_METRIC = "vehicle-ticks/s (1e6 / us-per-tick x B) of the ten-token expert tick (state token, 4 visual, 5 queries)"


def paper_inputs(args, device):
    from paper_2607_15621_gb300 import synth
    spec = synth.PAPER_WORKLOADS[args.workload]
    dims = dataclasses.replace(synth.EXPERT, n_action=5, n_frame=5)
    if args.layers is not None:
        dims = dataclasses.replace(dims, n_layers=args.layers)
    B, L = spec["batch"], spec["length"]
    w = synth.make_paper_weights(dims, 0, "bf16")
    k, v, off = synth.make_cache(dims, [L] * B, 0, "bf16", device=device)
    visual, state = synth.make_paper_inputs(dims, B, 0, "bf16", device=device)
    return dims, w, k, v, off, visual, state, B, L


def run_paper_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    from oracle import paper_tokens_oracle
    dims, w, k, v, off, visual, state, B, L = paper_inputs(args, "cpu")
    kn = [t.float().numpy() for t in k]
    vn = [t.float().numpy() for t in v]
    vis = visual[:1].double().numpy()
    st = state[:1].double().numpy()
    lo, hi = int(off[0]), int(off[1])
    seconds = max(1.0, min(args.cpu_seconds, 60.0))
    n, t0 = 0, time.perf_counter()
    while True:
        paper_tokens_oracle.expert_tick_paper_tokens(w, [t[lo:hi] for t in kn], [t[lo:hi] for t in vn],
                                                     np.array([0, hi - lo]), vis, st, dims.n_heads, dims.head_dim)
        n += 1
        el = time.perf_counter() - t0
        if el >= seconds or n >= 1000:
            break
    cb = {"value": n / el, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
          "sample": f"{n} full {dims.n_layers}-layer fp64 ten-token ticks of vehicle 0 of {args.workload} (L={L}) "
                    f"in {el:.1f} s"}
    line = {"impl": "reference", "metric": PAPER_METRIC, "value": cb["value"], "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * B / cb["value"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)",
            "config": {"workload": args.workload, "B": B, "cache_len": L, "layers": dims.n_layers,
                       "tokens_per_vehicle": 10, "parallelism": f"replicas x{world}",
                       "sample": "vehicle 0 per step; vehicles are independent"},
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def run_paper(args):
    """The ten-token tick on the GPU: CUDA events around K ticks (state MLP, layer stack,
    two-layer head), inputs resident in HBM; e2e with the visual tokens and ego state
    copied in from pinned host memory and the waypoints read back every tick."""
    import torch
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_15621_gb300 import fsx
    dims, w, k, v, off, visual, state, B, L = paper_inputs(args, dev)
    offsets = torch.as_tensor(off, device=dev)
    out = torch.empty(B, 5, 2, device=dev)
    ex = fsx.PaperExpert(dims, w, B, int(off[-1]), "bf16", "bf16", device=local)
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    for _ in range(max(args.warmup, 3)):
        ex.paper_tick(k, v, offsets, visual, state, out, stream)
    torch.cuda.synchronize()
    if ex.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during warm-up")
    clock_path = os.path.join(clock_dir(), f"clocks_rank{rank}.csv")
    os.makedirs(os.path.dirname(clock_path), exist_ok=True)
    proc, fh = start_clock_sampler(clock_path, local)
    time.sleep(0.5)
    barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        ex.paper_tick(k, v, offsets, visual, state, out, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms = max_over_ranks(e0.elapsed_time(e1), dev)
    clocks = stop_clock_sampler(proc, fh, clock_path)
    if ex.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during the timed region")
    ms_per_step = ms / args.steps
    vis_h = visual.cpu().pin_memory()
    st_h = state.cpu().pin_memory()
    out_h = torch.empty(B, 5, 2).pin_memory()
    e2e_steps = max(1, args.steps // 2)
    barrier()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        visual.copy_(vis_h, non_blocking=True)
        state.copy_(st_h, non_blocking=True)
        ex.paper_tick(k, v, offsets, visual, state, out, stream)
        out_h.copy_(out, non_blocking=True)
        stream.synchronize()
    e2e_s = max_over_ranks(time.perf_counter() - t0, dev)
    hbm, tensor_tfs, peak_kind = peaks()
    tick_bytes, _ = algorithmic_bytes(dims, [L] * B, "bf16", ex.weight_bytes())
    flops = tick_flops(dims, [L] * B)
    rl_us = max(tick_bytes / (hbm * 1e9), flops / (tensor_tfs * 1e12)) * 1e6
    achieved = tick_bytes / (ms_per_step / 1e3) / 1e9
    line = {
        "metric": PAPER_METRIC, "value": world * B / (ms_per_step / 1e3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step,
        "us_per_tick": ms_per_step * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f16 (fp32 accumulate)", "data": "synthetic (seeded N(0,1) cache/visual/state, N(0,1/fan_in) weights)",
        "config": {"workload": args.workload, "B": B, "cache_len": L, "layers": dims.n_layers, "tokens_per_vehicle": 10,
                   "l2": "inputs larger than L2 (the expert weights exceed 129 MB)",
                   "parallelism": f"replicas x{world}"},
        "gpu_launches": (1 + ex.launches(B)) * args.steps,
        "roofline": {"bound": "hbm", "kernel": "ten-token tick (state MLP, tick, head)", "achieved": achieved,
                     "peak": hbm, "unit": "GB/s", "frac": achieved / hbm, "traffic": None, "peak_source": peak_kind,
                     "bytes_per_launch": tick_bytes, "launch_us": ms_per_step * 1e3, "flops_per_tick": flops,
                     "roofline_us": rl_us, "frac_of_tick_roofline": rl_us / (ms_per_step * 1e3)},
        "e2e": {"value": world * B * e2e_steps / e2e_s, "unit": UNIT,
                "h2d_bytes_per_step": int(vis_h.numel() * vis_h.element_size() + st_h.numel() * 4),
                "d2h_bytes_per_step": int(out_h.numel() * 4)},
        "clocks": clocks,
    }
    ex.close()
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


FASTSLOW_METRIC = "vehicle-ticks/s (1e6 / mean tick latency) of the expert tick while the cache append runs every 4 ticks"


def run_fastslow_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    print(json.dumps({"impl": "reference", "unavailable": "the fast-slow schedule is a GPU stream schedule; its "
                      "arithmetic (the tick and the append) has reference arms of its own "
                      "(--workload bf16_b1_l224, --workload append_b1_l224)"}))


def run_fastslow(args):
    """Ticks of one vehicle paced at a fixed cadence with a 4-token cache append issued
    before every k-th tick, through an fsx session, in the serial and the concurrent
    schedule. A tick's latency runs from its issue (an event on an idle stream) to the end
    of its work on the tick stream, so it includes any wait for, or contention with, an
    append."""
    import torch
    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2607_15621_gb300 import fsx, synth
    spec = synth.FASTSLOW_WORKLOADS[args.workload]
    dims = synth.EXPERT if args.layers is None else dataclasses.replace(synth.EXPERT, n_layers=args.layers)
    bdims = dataclasses.replace(synth.BACKBONE, n_layers=dims.n_layers)
    L0, K, cadence = spec["length"], spec["k"], spec["cadence_ms"] / 1e3
    n_ticks = args.steps
    cap = L0 + (n_ticks // K + 8) * bdims.n_new + 64
    w = synth.make_weights(dims, 0, "bf16")
    bw = synth.make_backbone_weights(bdims, 0, "bf16")
    k0, v0, _ = synth.make_cache(dims, [L0], 0, "bf16", device=dev)
    frames = synth.make_frames(dims, 1, 0, "bf16", device=dev)
    x = synth.make_append_tokens(bdims, 1, 0, device=dev)
    hidden = torch.empty(1, bdims.n_new, bdims.d_model, device=dev)
    out = torch.empty(1, dims.n_waypoints, 2, device=dev)
    ex = fsx.Expert(dims, w, 1, cap, device=local)
    ap = fsx.Append(bdims, bw, 1, cap, device=local)
    del w, bw
    clock = torch.cuda.Stream(dev)
    modes = {}
    for name, concurrent in (("serial", False), ("concurrent", True)):
        kc = [torch.zeros(cap, dims.n_heads, dims.head_dim, dtype=torch.bfloat16, device=dev) for _ in k0]
        vc = [torch.zeros_like(t) for t in kc]
        for dst, src in zip(kc + vc, k0 + v0):
            dst[:L0] = src
        ses = fsx.Session(ex, ap, kc, vc, cap, L0, concurrent, device=local)
        tick_stream = torch.cuda.ExternalStream(ses.tick_stream(), device=dev)
        app_stream = torch.cuda.ExternalStream(ses.append_stream(), device=dev)
        for i in range(8):  # warm-up, appends included
            if i % K == 0:
                ses.append(x, hidden)
            ses.tick(frames, out)
        ses.sync()
        pairs, apairs, snaps = [], [], []
        t0 = time.perf_counter()
        for i in range(n_ticks):
            wait = t0 + i * cadence - time.perf_counter()
            if wait > 0:
                time.sleep(wait)
            if i % K == 0:
                a0 = torch.cuda.Event(enable_timing=True)
                a1 = torch.cuda.Event(enable_timing=True)
                a0.record(app_stream)
                ses.append(x, hidden)
                a1.record(app_stream)
                apairs.append((a0, a1))
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(clock)
            snaps.append(ses.tick(frames, out))
            e1.record(tick_stream)
            pairs.append((e0, e1))
        ses.sync()
        if ex.status() != fsx.FSX_OK or ap.status() != fsx.FSX_OK:
            raise RuntimeError("device status set during the fast-slow schedule")
        lat = np.array([a.elapsed_time(b) * 1e3 for a, b in pairs])
        app = np.array([a.elapsed_time(b) * 1e3 for a, b in apairs])
        modes[name] = {"ticks": n_ticks, "tick_latency_us": {
                           "p50": float(np.percentile(lat, 50)), "p90": float(np.percentile(lat, 90)),
                           "p99": float(np.percentile(lat, 99)), "max": float(lat.max()), "mean": float(lat.mean()),
                           "with_append_issued_p50": float(np.percentile(lat[::K], 50)),
                           "without_append_p50": float(np.percentile(np.delete(lat, np.s_[::K]), 50))},
                       "append_us": {"p50": float(np.percentile(app, 50)), "max": float(app.max())},
                       "snapshot_rows": {"first": int(snaps[0]), "last": int(snaps[-1]),
                                         "stale_ticks": int(sum(1 for i, s_ in enumerate(snaps)
                                                                if i % K == 0 and s_ < snaps[min(i + 1, n_ticks - 1)]))}}
        ses.close()
        del kc, vc
    ex.close()
    ap.close()
    conc = modes["concurrent"]["tick_latency_us"]
    line = {
        "metric": FASTSLOW_METRIC, "value": 1e6 / conc["mean"], "unit": UNIT, "n_gpus": 1, "steps": n_ticks,
        "warmup": 8, "ms_per_step": conc["mean"] / 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f16 (fp32 accumulate)",
        "data": "synthetic (seeded N(0,1) cache/frames/new tokens, N(0,1/fan_in) weights)",
        "config": {"workload": args.workload, "cache_len": L0, "append_every": K, "cadence_ms": spec["cadence_ms"],
                   "layers": dims.n_layers, "backbone_d_model": bdims.d_model, "new_tokens": bdims.n_new},
        "gpu_launches": None, "schedules": modes,
    }
    if rank == 0:
        print(json.dumps(line))


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    spec, lengths = workload_info(args.workload)
    B = int(len(lengths))
    cb = cpu_baseline(args.workload, max(1.0, min(args.cpu_seconds, 60.0)))
    line = {"impl": "reference", "metric": METRIC, "value": cb["value"], "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * B / cb["value"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded)",
            "config": {"workload": args.workload, "B": B, "cache_len": [int(x) for x in lengths[:4]],
                       "layers": 32, "parallelism": f"replicas x{world}",
                       "sample": cb["sample"] + "; vehicles are independent, so vehicle-ticks/s is per vehicle"},
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))


def spawn_ranks(n):
    """--gpus N without torchrun: run N copies of this command, one per GPU, with the
    rank environment torchrun would set; rank 0's output is this process's output."""
    import socket
    with socket.socket() as sock:
        sock.bind(("127.0.0.1", 0))
        port = sock.getsockname()[1]
    procs = []
    for r in range(n):
        env = dict(os.environ, RANK=str(r), LOCAL_RANK=str(r), WORLD_SIZE=str(n), MASTER_ADDR="127.0.0.1",
                   MASTER_PORT=str(port))
        out = None if r == 0 else subprocess.DEVNULL
        procs.append(subprocess.Popen([sys.executable, os.path.abspath(__file__)] + sys.argv[1:], env=env, stdout=out))
    codes = [p.wait() for p in procs]
    return max(codes, key=abs)


def time_ticks(ex, k, v, offsets, frames, out, stream, steps, warmup):
    """Device milliseconds of `steps` ticks between CUDA events on `stream`, after `warmup`."""
    import torch
    from paper_2607_15621_gb300 import fsx
    for _ in range(max(warmup, 3)):
        ex.tick(k, v, offsets, frames, out, stream)
    torch.cuda.synchronize()
    if ex.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during warm-up")
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        ex.tick(k, v, offsets, frames, out, stream)
    e1.record(stream)
    torch.cuda.synchronize()
    if ex.status(stream) != fsx.FSX_OK:
        raise RuntimeError("device status set during the timed region")
    return e0.elapsed_time(e1)


def tick_roofline_us(dims, lengths, dtype, weight_bytes, hbm, tensor_tfs):
    """max(bytes / HBM bandwidth, FLOPs / tensor peak) of one tick, in microseconds."""
    tick_bytes, _ = algorithmic_bytes(dims, lengths, dtype, weight_bytes)
    return max(tick_bytes / (hbm * 1e9), tick_flops(dims, lengths) / (tensor_tfs * 1e12)) * 1e6


def run_extras(ex, dims, dev, stream, weight_bytes, hbm, tensor_tfs):
    """The B = 1 tick, the history sweep and the 16-vehicle batch through the headline's
    handle: us/tick and fraction of the tick roofline of each (CUDA events)."""
    import torch
    from paper_2607_15621_gb300 import synth
    res = []
    for name in EXTRA_WORKLOADS:
        spec, lengths = workload_info(name)
        B = len(lengths)
        k, v, off = synth.make_cache(dims, lengths, 0, spec["dtype"], device=dev)
        frames = synth.make_frames(dims, B, 0, spec["dtype"], device=dev)
        offsets = torch.as_tensor(off, device=dev)
        out = torch.empty(B, dims.n_waypoints, 2, device=dev)
        steps = 200 if B == 1 else 50
        ms = time_ticks(ex, k, v, offsets, frames, out, stream, steps, 5)
        us = ms / steps * 1e3
        rl = tick_roofline_us(dims, lengths, spec["dtype"], weight_bytes, hbm, tensor_tfs)
        tick_bytes, _ = algorithmic_bytes(dims, lengths, spec["dtype"], weight_bytes)
        res.append({"workload": name, "B": B, "cache_tokens": int(np.sum(lengths)), "us_per_tick": us,
                    "vehicle_ticks_per_s": B * 1e6 / us, "steps": steps, "launches_per_tick": ex.launches(B),
                    "roofline_us": rl, "frac": rl / us, "achieved_gbs": tick_bytes / (us * 1e-6) / 1e9,
                    "bytes_per_tick": tick_bytes})
        del k, v, frames
    torch.cuda.empty_cache()
    return res


def main():
    args = parse()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        sys.exit(spawn_ranks(args.gpus))
    from paper_2607_15621_gb300 import synth
    if args.workload in synth.APPEND_WORKLOADS:
        (run_append_reference if args.impl == "reference" else run_append)(args)
        return
    if args.workload in synth.CLIP_WORKLOADS:
        (run_clip_reference if args.impl == "reference" else run_clip)(args)
        return
    if args.workload in synth.FASTSLOW_WORKLOADS:
        (run_fastslow_reference if args.impl == "reference" else run_fastslow)(args)
        return
    if args.workload in synth.PAPER_WORKLOADS:
        (run_paper_reference if args.impl == "reference" else run_paper)(args)
        return
    if args.impl == "reference":
        run_reference(args)
        return
    import torch
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from paper_2607_15621_gb300 import fsx, synth
    spec, lengths = workload_info(args.workload)
    dims = synth.EXPERT if args.layers is None else dataclasses.replace(synth.EXPERT, n_layers=args.layers)
    dtype = spec["dtype"]
    B = len(lengths)
    extras = (not args.no_extras and args.workload == DEFAULT_WORKLOAD and args.layers is None)
    w = synth.make_weights(dims, 0, dtype)
    k, v, off = synth.make_cache(dims, lengths, 0, dtype, device=dev)
    frames = synth.make_frames(dims, B, 0, dtype, device=dev)
    offsets = torch.as_tensor(off, device=dev)
    out = torch.empty(B, dims.n_waypoints, 2, device=dev)
    ex = fsx.Expert(dims, w, B, int(off[-1]), dtype, dtype, device=local)
    del w
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    clock_path = os.path.join(clock_dir(), f"clocks_rank{rank}.csv")
    os.makedirs(os.path.dirname(clock_path), exist_ok=True)
    for _ in range(max(args.warmup, 3)):
        ex.tick(k, v, offsets, frames, out, stream)
    torch.cuda.synchronize()
    proc, fh = start_clock_sampler(clock_path, local)
    time.sleep(0.5)
    barrier()
    torch.cuda.synchronize()
    ms = time_ticks(ex, k, v, offsets, frames, out, stream, args.steps, 0)
    barrier()
    clocks = stop_clock_sampler(proc, fh, clock_path)
    ms = max_over_ranks(ms, dev)
    ms_per_step = ms / args.steps
    value = world * B * args.steps / (ms / 1e3)

    # ---- end to end through the host-buffer entry point (copies inside the timed region)
    frames_h = frames.cpu().pin_memory()
    off_h = torch.as_tensor(off).pin_memory()
    out_h = torch.empty(B, dims.n_waypoints, 2).pin_memory()
    for _ in range(3):
        ex.tick_host(k, v, off_h.numpy(), frames_h, out_h.numpy(), stream)
    barrier()
    e2e_steps = max(1, args.steps // 2)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        ex.tick_host(k, v, off_h.numpy(), frames_h, out_h.numpy(), stream)
    e2e_s = time.perf_counter() - t0
    barrier()
    e2e_s = max_over_ranks(e2e_s, dev)
    h2d = frames_h.numel() * frames_h.element_size() + off_h.numel() * 8
    d2h = out_h.numel() * 4

    # ---- dominant kernel: CUDA events around its launches inside the replayed tick graph
    kclass = args.kernel_class
    if ex.launches(B) == 1:  # single-launch persistent tick: the tick kernel is the dominant kernel
        kclass = "persistent"
    elif kclass is None:  # batched ticks: Eq. 1 attention streams the cache and dominates
        kclass = "attention"
    ex.set_kernel_timing(True, kclass)
    kt_ms, kt_n = [], 0
    for i in range(max(args.steps // 4, 5) + 2):
        ex.tick(k, v, offsets, frames, out, stream)
        t, n = ex.kernel_time()
        if i >= 2:
            kt_ms.append(t)
            kt_n = n
    ex.set_kernel_timing(False, kclass)
    per_launch_s = statistics.mean(kt_ms) / kt_n / 1e3
    d, hd, f = dims.d_model, dims.hd, dims.d_ff
    # a batch may run as several chains (vehicle groups), each with its own launch of a
    # kernel class per layer: average algorithmic bytes of one launch = the class's bytes
    # per tick / its launches per tick
    chains = max(1, kt_n // dims.n_layers) if kclass != "persistent" else 1
    Mc = B * dims.n_tok / chains  # token rows of one chain
    unit_bytes = {  # algorithmic bytes of one launch (one layer of one chain): weights + activations in/out
        "qkv": 3 * hd * d * 2 + Mc * d * 4 + Mc * 3 * hd * 2,
        "out_proj": d * hd * 2 + Mc * hd * 2 + 2 * Mc * d * 4,
        "gate_up": 2 * f * d * 2 + Mc * d * 4 + Mc * f * 2,
        "down": d * f * 2 + Mc * f * 2 + 2 * Mc * d * 4,
        "attention": (int(np.sum(lengths)) * 2 * hd * (2 if dtype == "bf16" else 4)) / chains + Mc * 3 * hd * 2
                     + Mc * hd * 2,
        "persistent": None,
    }[kclass]
    if unit_bytes is None:  # one launch = the whole tick: weights + cache rows
        unit_bytes = algorithmic_bytes(dims, lengths, dtype, ex.weight_bytes())[0]
    unit_bytes = int(unit_bytes)
    hbm, tensor_tfs, peak_kind = peaks()
    achieved = unit_bytes / per_launch_s / 1e9
    tick_bytes, kv_bytes = algorithmic_bytes(dims, lengths, dtype, ex.weight_bytes())
    tick_gbs = tick_bytes / (ms_per_step / 1e3) / 1e9
    flops = tick_flops(dims, lengths)
    # roofline time of one tick = max(bytes / HBM bandwidth, FLOPs / tensor peak)
    rl_meas_us = max(tick_bytes / (hbm * 1e9), flops / (tensor_tfs * 1e12)) * 1e6
    rl_nom_us = max(tick_bytes / (NOMINAL_HBM_GBS * 1e9), flops / (NOMINAL_TENSOR_TFS * 1e12)) * 1e6
    traffic, traffic_stale = traffic_for(kclass, args.workload)
    launches = ex.launches(B)
    weight_bytes = ex.weight_bytes()
    extra_lines = None
    if extras:
        del k, v, frames
        torch.cuda.empty_cache()
        extra_lines = run_extras(ex, dims, dev, stream, weight_bytes, hbm, tensor_tfs)

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_per_step, "us_per_tick": ms_per_step * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f16 (fp32 accumulate)",
        "data": "synthetic (seeded N(0,1) cache/frames, N(0,1/fan_in) weights)",
        "config": {"workload": args.workload, "B": B, "cache_len": [int(x) for x in lengths[:4]],
                   "cache_tokens": int(np.sum(lengths)), "layers": dims.n_layers, "d_model": dims.d_model,
                   "tokens_per_vehicle": dims.n_tok,
                   "l2": "inputs larger than L2 (weights + cache per tick exceed 129 MB)",
                   "parallelism": f"replicas x{world}"},
        "gpu_launches": launches * args.steps,
        "roofline": {"bound": "hbm", "kernel": kclass, "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm, "traffic": traffic, "traffic_stale": traffic_stale,
                     "peak_source": peak_kind, "bytes_per_launch": unit_bytes, "launch_us": per_launch_s * 1e6,
                     "launches_per_tick": kt_n},
        "tick_roofline": {"bytes_per_tick": tick_bytes, "kv_bytes_per_tick": kv_bytes, "achieved_gbs": tick_gbs,
                          "frac_of_measured_hbm": tick_gbs / hbm, "frac_of_8tbs": tick_gbs / NOMINAL_HBM_GBS,
                          "flops_per_tick": flops,
                          "bound": "hbm" if tick_bytes / hbm >= flops / (tensor_tfs * 1e3) else "tensor",
                          "roofline_us_measured_peaks": rl_meas_us, "frac_measured_peaks": rl_meas_us / (ms_per_step * 1e3),
                          "roofline_us_8tbs_2250tf": rl_nom_us, "frac_8tbs_2250tf": rl_nom_us / (ms_per_step * 1e3),
                          "peaks": {"hbm_gbs": hbm, "tensor_tflops_sustained": tensor_tfs, "source": peak_kind}},
        "e2e": {"value": world * B * e2e_steps / e2e_s, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h)},
        "clocks": clocks,
    }
    if extra_lines is not None:
        line["workloads"] = extra_lines
    ex.close()
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.workload, args.cpu_seconds)
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()

if __name__ == "__main__":
    main()
