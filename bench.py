"""Benchmark: batch-1 dual-sparse spMspV over a LLaMA-2-7B-shaped decoder layer.

One step = one decoder layer's seven projections at 50% weight / 50%
activation sparsity, launched as a decode step must order them: the fused
sparsify + spMspV of q/k/v (one shared input), then o, then gate/up (one
shared input), then down (four launches of the CUDA kernel).  Eight distinct
seeded layers rotate so that every step streams weights that are not in L2.

Printed metric: effective HBM GB/s on the required bytes (the kept channels'
fp16 non-zeros, one mask bit per kept position, x, kept ids/values and y),
plus microseconds per layer.  Padding, offset tables and index bytes are not
required bytes; the DRAM counters of a profile show them.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import tempfile
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "µs/layer and effective HBM GB/s (% of GB300 peak) for batch-1 dual-sparse spMspV"
WORKLOAD = "llama2-7b-layer"
STAGES = (("q", "k", "v"), ("o",), ("gate", "up"), ("down",))
STAGE_SRC = ("q", "o", "gate", "down")
FALLBACK_HBM_GBS = 6800.0
# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) per launch of
# the fused kernel from one ncu capture, valid only for the kernel source it
# was taken on (sha256 of kernels.cu + duo_device.cuh, first 16 hex digits).
TRAFFIC = {"sha": "68c049807b7c2ca1",
           "per_launch_bytes": [29113088.0, 9761024.0, 51911168.0, 26117632.0]}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=16000)
    ap.add_argument("--warmup", type=int, default=400)
    ap.add_argument("--impl", default="ours", choices=("ours", "reference"))
    ap.add_argument("--layers", type=int, default=8, help="distinct layers rotated")
    ap.add_argument("--px", type=int, default=50)
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--profile", action="store_true",
                    help="small case for ncu: 2 layers, a few direct (ungraphed) layer steps")
    ap.add_argument("--profile-coded", action="store_true",
                    help="small case for ncu: one 7B layer's four stages once per format (fp16, 8-bit, 4-bit)")
    ap.add_argument("--profile-calib", action="store_true",
                    help="small case for ncu: `--steps` calibration precomputes of a 4096-channel layer")
    ap.add_argument("--profile-sweep", action="store_true",
                    help="small case for ncu: one precompute, then `--steps` column sweeps of a 4096 x 4096 weight")
    ap.add_argument("--stack", default=None,
                    choices=("llama2-7b-layer", "llama3-8b-stack", "llama2-13b-stack", "llama2-70b-stack"),
                    help="per-token time over every layer of a stack workload (one CUDA graph per token)")
    ap.add_argument("--stack-layers", type=int, default=None, help="layers of the stack (default: all)")
    ap.add_argument("--stack-pw", type=float, default=None, help="weight sparsity (default: the workload's)")
    ap.add_argument("--no-dense", action="store_true", help="--stack: skip the dense cuBLAS baseline")
    ap.add_argument("--no-stack", action="store_true", help="default line: skip the llama3-8b stack")
    return ap.parse_args()


# ----------------------------------------------------------------- helpers --

def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_sha() -> str:
    import hashlib
    h = hashlib.sha256()
    for f in ("kernels.cu", "duo_device.cuh"):
        with open(os.path.join(ROOT, "paper_2506_20194_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


class ClockSampler:
    """nvidia-smi sampling during the timed region (clocks, throttle reasons)."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        out = os.environ.get("DUO_CLOCKS_DIR") or tempfile.gettempdir()
        self.path = os.path.join(out, f"clocks_rank{index}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, smax, reasons = [], None, set()
        names = ("active", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names[1:], parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": smax,
                "samples": len(sm), "reasons": sorted(reasons)}


def make_layers(duo, synth, L, device, px):
    """Packs L distinct LLaMA-2-7B-shaped layers; returns per-layer dicts."""
    wl = synth.WORKLOADS[WORKLOAD]
    shape = wl["shape"]
    layers = []
    for l in range(L):
        Ws = {p: synth.layer_weight(wl, p, layer=l, device=device) for p in synth.PROJS}
        hs = {p: duo.duo_pack(Ws[p], "bitmask") for p in synth.PROJS}
        nnz = {p: (Ws[p] != 0).sum(dim=0).to(torch.int64) for p in synth.PROJS}
        xs = {s: synth.layer_input(wl, s, layer=l, device=device) for s in STAGE_SRC}
        ys = {p: torch.empty(shape.O(p), dtype=torch.float32, device=device) for p in synth.PROJS}
        layers.append(dict(W=Ws, h=hs, nnz=nnz, x=xs, y=ys))
    return shape, layers


def k_of(I, px):
    return (I * (100 - px)) // 100


def side_bytes_from_sets(shape, nnz, kept, px):
    """Companions of the required bytes of one layer step, from the kept
    channel sets: the kept non-zero values alone (2 sum nnz_j over kept j:
    the weights loaded, the quantity the paper counts), and the worst case of
    the required-bytes formula, with the k densest channels of each stage
    selected instead of the ones x picks; then the values of both as
    fractions of the dense weights (Fig. 3's loaded fraction and its worst
    case, App. B.3).  nnz[p]: int64 tensor of non-zeros per input channel of
    projection p; kept[si]: int64 tensor of stage si's kept channel ids."""
    vals = worst = wvals = dense = 0.0
    for si, st in enumerate(STAGES):
        I = shape.I(st[0])
        k = k_of(I, px)
        for p in st:
            dense += 2.0 * shape.O(p) * shape.I(p)
        if k == 0:
            worst += 2.0 * I
            continue
        K = kept[si]
        tot = sum(nnz[p] for p in st)                    # per channel, over the stage's products
        dense_k = torch.topk(tot, k).indices
        for p in st:
            O = shape.O(p)
            vals += float(nnz[p][K].sum().item()) * 2.0
            wv = float(nnz[p][dense_k].sum().item()) * 2.0
            wvals += wv
            worst += wv + k * O / 8.0 + 4.0 * O
        worst += 2.0 * I + 4.0 * k
    return vals, worst, vals / dense, wvals / dense


def side_bytes_layer(duo, shape, layer, px):
    """side_bytes_from_sets with the kept sets from the library's own
    (parity-tested) sparsifier."""
    kept = []
    for st, src in zip(STAGES, STAGE_SRC):
        k = k_of(shape.I(st[0]), px)
        if k == 0:
            kept.append(None)
            continue
        idx, _ = duo.duo_sparsify(layer["x"][src], k)
        kept.append(idx.to(torch.int64) & 0xFFFF)
    return side_bytes_from_sets(shape, layer["nnz"], kept, px)


def required_bytes_layer(duo, shape, layer, px):
    """Format-neutral required bytes of one layer step, with the kept sets
    taken from the library's own (parity-tested) sparsifier."""
    total = 0.0
    per_stage = []
    for st, src in zip(STAGES, STAGE_SRC):
        I = shape.I(st[0])
        k = k_of(I, px)
        b = 0.0
        if k > 0:
            idx, _ = duo.duo_sparsify(layer["x"][src], k)
            K = idx.to(torch.int64) & 0xFFFF
        for p in st:
            O = shape.O(p)
            vals = float(layer["nnz"][p][K].sum().item()) * 2.0 if k > 0 else 0.0
            b += vals + k * O / 8.0 + 4.0 * O
        b += 2.0 * I + 4.0 * k
        per_stage.append(b)
        total += b
    return total, per_stage


def stage_calls(duo, shape, layer, px):
    def run():
        for si in range(len(STAGES)):
            stage_call(duo, shape, layer, px, si)
    return run


def capture(fn):
    """Captures fn() into a CUDA graph after one eager warm-up run."""
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):           # warm the launch path (attributes, module load)
        fn()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


def stage_call(duo, shape, layer, px, si):
    st, src = STAGES[si], STAGE_SRC[si]
    k = k_of(shape.I(st[0]), px)
    if len(st) == 1:
        duo.duo_spmspv(layer["h"][st[0]], layer["x"][src], k, y=layer["y"][st[0]])
    else:
        duo.duo_spmspv_multi([layer["h"][p] for p in st], layer["x"][src], k,
                             ys=[layer["y"][p] for p in st])


def capture_rotation(duo, shape, layers, px):
    """One CUDA graph replaying every layer once (L steps, 4 launches each)."""
    def fn():
        for layer in layers:
            for si in range(len(STAGES)):
                stage_call(duo, shape, layer, px, si)
    return capture(fn)


def capture_stage(duo, shape, layers, px, si):
    """One CUDA graph launching stage si of every layer (L launches)."""
    def fn():
        for layer in layers:
            stage_call(duo, shape, layer, px, si)
    return capture(fn)


def time_graph(g, reps):
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record()
    for _ in range(reps):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) * 1e-3


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(v, world):
    if world == 1:
        return v
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_gbs(bytes_per_step, steps, world, seconds):
    """Whole-job throughput of N replicas: every rank moves bytes_per_step
    per step, the time is the slowest rank's."""
    return bytes_per_step * steps * world / seconds / 1e9


# --------------------------------------------------------- CPU oracle arm --

def oracle_layer_sample(shape, cpu_layer, px, row_frac):
    """Runs the oracle on a row sample of every projection of one layer;
    returns (seconds, required bytes covered by the sample)."""
    import oracle as orc
    t0 = time.perf_counter()
    covered = 0.0
    for st, src in zip(STAGES, STAGE_SRC):
        x16 = cpu_layer["x"][src]
        I = x16.size
        k = k_of(I, px)
        for p in st:
            W = cpu_layer["W"][p]
            O = W.shape[0]
            nr = max(1, int(round(O * row_frac)))
            y = orc.oracle_spmspv_rows(W[:nr], x16, k)
            assert y.shape[0] == nr
            covered += cpu_layer["breq"][p] * nr / O
    return time.perf_counter() - t0, covered


def cpu_layer_from(layer, shape, px):
    """Host copies of one layer (fp16 numpy) plus per-projection required bytes."""
    W = {p: layer["W"][p].cpu().numpy().view(np.float16) for p in layer["W"]}
    x = {s: layer["x"][s].cpu().numpy().view(np.float16) for s in STAGE_SRC}
    import oracle as orc
    breq = {}
    for st, src in zip(STAGES, STAGE_SRC):
        I = shape.I(st[0])
        k = k_of(I, px)
        K, _ = orc.oracle_sparsify(x[src], k)
        for p in st:
            nnz = (W[p] != 0).sum(axis=0)
            breq[p] = orc.required_bytes(nnz, K, shape.O(p), I)
    return dict(W=W, x=x, breq=breq)


def cpu_baseline(shape, layer, px, seconds):
    cl = cpu_layer_from(layer, shape, px)
    # calibrate a row fraction so that one sample step takes ~0.5 s
    t, cov = oracle_layer_sample(shape, cl, px, 1.0 / 64)
    frac = min(1.0, (1.0 / 64) * 0.5 / max(t, 1e-6))
    tot_t, tot_b, n = 0.0, 0.0, 0
    while tot_t < seconds:
        t, cov = oracle_layer_sample(shape, cl, px, frac)
        tot_t += t
        tot_b += cov
        n += 1
    gbs = tot_b / tot_t / 1e9
    full_layer_b = sum(cl["breq"].values())
    return {"value": gbs, "unit": "GB/s", "cores": os.cpu_count(), "kind": "oracle",
            "us_per_layer": full_layer_b / (gbs * 1e9) * 1e6,
            "sample": f"{n} steps of the fp64 numpy oracle on {frac:.4f} of every projection's rows "
                      f"of one {WORKLOAD} (px={px}), {tot_t:.1f} s; numpy BLAS threads default "
                      f"(all {os.cpu_count()} cores)"}


def run_reference(args):
    world, rank, _ = dist_setup(args)
    if rank != 0:
        return
    from paper_2506_20194_gb300 import synth
    wl = synth.WORKLOADS[WORKLOAD]
    shape = wl["shape"]
    layer = {"W": {p: synth.layer_weight(wl, p, layer=0) for p in synth.PROJS},
             "x": {s: synth.layer_input(wl, s, layer=0) for s in STAGE_SRC}}
    cl = cpu_layer_from(layer, shape, args.px)
    t, _ = oracle_layer_sample(shape, cl, args.px, 1.0 / 256)
    budget = 120.0 / max(1, args.steps + args.warmup)
    frac = min(1.0, max(1.0 / 4096, (1.0 / 256) * budget / max(t, 1e-6)))
    for _ in range(args.warmup):
        oracle_layer_sample(shape, cl, args.px, frac)
    tot_t, tot_b = 0.0, 0.0
    for _ in range(args.steps):
        t, cov = oracle_layer_sample(shape, cl, args.px, frac)
        tot_t += t
        tot_b += cov
    gbs = tot_b / tot_t / 1e9
    sample = (f"fp64 numpy oracle on {frac:.5f} of every projection's rows of one {WORKLOAD} "
              f"layer per step (px={args.px})")
    line = {"impl": "reference", "metric": METRIC, "value": gbs, "unit": "GB/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": tot_t / max(1, args.steps) * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "px": args.px, "pw": 0.5},
            "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------- our arm --

def run_ours(args):
    world, rank, local = dist_setup(args)
    assert torch.cuda.is_available(), "bench.py needs a CUDA device"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo, synth
    duo.load_library()
    L = args.layers
    shape, layers = make_layers(duo, synth, L, dev, args.px)
    breq_layers = [required_bytes_layer(duo, shape, lay, args.px) for lay in layers]
    breq_mean = float(np.mean([b for b, _ in breq_layers]))
    side = np.mean(np.array([side_bytes_layer(duo, shape, lay, args.px) for lay in layers]), axis=0)
    stage_b = np.mean(np.array([ps for _, ps in breq_layers]), axis=0)

    # Exactly W warm-up and K timed layer steps: replays of the rotation graph
    # (L steps each) and one graph of the first K mod L layers.
    g = capture_rotation(duo, shape, layers, args.px)
    rem_graphs = {}

    def run_steps(n):
        for _ in range(n // L):
            g.replay()
        r = n % L
        if r:
            if r not in rem_graphs:
                rem_graphs[r] = capture_rotation(duo, shape, layers[:r], args.px)
            rem_graphs[r].replay()

    steps_timed = max(1, args.steps)
    reps = max(1, steps_timed // L)   # replays for the secondary timings below
    for n in (steps_timed, max(3, args.warmup)):   # capture every graph before any timing
        if n % L and n % L not in rem_graphs:
            rem_graphs[n % L] = capture_rotation(duo, shape, layers[:n % L], args.px)
    run_steps(max(3, args.warmup))
    # Clocks: nvidia-smi every 20 ms over a window of sustained load (the same
    # graph replayed for about 0.3 s on each side) that contains the timed
    # region, which alone may be shorter than one sample.
    sampler = ClockSampler(local)
    sampler.start()
    load_reps = max(1, int(0.3 / (L * 70e-6)))
    for _ in range(load_reps):
        g.replay()
    barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    run_steps(steps_timed)
    e1.record()
    torch.cuda.synchronize()
    barrier(world)
    t = e0.elapsed_time(e1) * 1e-3
    for _ in range(load_reps):
        g.replay()
    torch.cuda.synchronize()
    clocks = sampler.stop()
    clocks["window"] = "sustained replays of the timed graph, about 0.3 s before and after the timed steps"
    clocks["interval_ms"] = 20
    t = max_over_ranks(t, world)
    assert duo.duo_device_status() == duo.DUO_OK
    us_layer = t / steps_timed * 1e6
    value = whole_job_gbs(breq_mean, steps_timed, world, t)

    # Average launch duration of the fused kernel per stage: a graph of that
    # stage's launch for every layer, timed with CUDA events on the stream.
    stage_us = []
    for si in range(len(STAGES)):
        gs = capture_stage(duo, shape, layers, args.px, si)
        time_graph(gs, 3)
        r = max(3, min(reps, 500))
        stage_us.append(time_graph(gs, r) / (r * L) * 1e6)
        del gs
    stage_us = np.array(stage_us)
    peak, peak_kind = peaks()
    achieved = float(stage_b.sum() / (stage_us.sum() * 1e-6) / 1e9)
    traffic = None
    if kernel_sha() == TRAFFIC["sha"]:
        traffic = float(np.mean(TRAFFIC["per_launch_bytes"]))
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "peak_kind": peak_kind, "traffic": traffic,
                "bytes_per_launch": float(stage_b.mean()),
                "kernel": "cmb_spmspv_kernel<fused>",
                "per_launch_bytes": [float(b) for b in stage_b],
                "per_launch_us": [float(u) for u in stage_us],
                "per_launch_GBps": [float(b / (u * 1e-6) / 1e9) for b, u in zip(stage_b, stage_us)]}

    # end to end through the public API with host buffers
    e2e = run_e2e(duo, shape, layers, args, breq_mean)

    # dense fp16 GEMV (cuBLAS via F.linear) over the same rotation
    dense = run_dense(shape, layers, reps=max(1, min(reps, 200)))

    sweep = {}
    if not args.no_sweep:
        for px in (0, 25, 50, 70):
            gs = capture_rotation(duo, shape, layers, px)
            time_graph(gs, 5)
            r = max(1, min(reps, 400))
            ts = time_graph(gs, r)
            b = float(np.mean([required_bytes_layer(duo, shape, lay, px)[0] for lay in layers]))
            us = ts / (r * L) * 1e6
            sweep[str(px)] = {"us_per_layer": us, "GB/s": b / (us * 1e-6) / 1e9,
                              "frac_of_peak": b / (us * 1e-6) / 1e9 / peak, "required_MB": b / 1e6}
            del gs

    thresh = run_threshold_path(duo, shape, layers, args.px, reps, peak)
    quant = {f"int{b}": run_quant_path(duo, shape, layers, args.px, reps, peak, b) for b in (8, 4)}
    calib = run_calib(duo, reps)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(shape, layers[0], args.px, args.cpu_seconds)

    # The 32-layer LLaMA-3-8B-shaped stack (per-token time, the paper's
    # figure of merit), with its dense cuBLAS baseline; the 7B layers are
    # freed first.
    stack = None
    if rank == 0 and world == 1 and not args.no_stack:
        del g, rem_graphs
        for lay in layers:
            for h in lay["h"].values():
                h.free()
        layers.clear()
        torch.cuda.empty_cache()
        stack = measure_stack(duo, synth, dev, "llama3-8b-stack", px=args.px, reps=20, warmup=3)

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "GB/s", "us_per_layer": us_layer,
            "n_gpus": world, "steps": steps_timed, "warmup": max(3, args.warmup),
            "ms_per_step": us_layer * 1e-3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f16", "data": "synthetic",
            "config": {"workload": WORKLOAD, "shapes": "q/k/v/o 4096x4096, gate/up 11008x4096, down 4096x11008",
                       "pw": 0.5, "prune": "magnitude, exact count per 128-channel block",
                       "px": args.px, "format": "bitmask (CMB)", "layers_rotated": L,
                       "l2": f"inputs larger than L2: {L} distinct packed layers rotated",
                       "required_MB_per_layer": breq_mean / 1e6,
                       "vals_only_MB_per_layer": float(side[0]) / 1e6,
                       "worst_case_required_MB_per_layer": float(side[1]) / 1e6,
                       "loaded_weight_fraction": float(side[2]),
                       "worst_case_loaded_weight_fraction": float(side[3]),
                       "parallelism": "replicas" if world > 1 else "1gpu"},
            "roofline": roofline,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": steps_timed * len(STAGES),
            "clocks": clocks,
            "stack": stack,
            "dense_gemv_cublas": dense,
            "sweep_px": sweep,
            "threshold_path": thresh,
            "quantised_values": quant,
            "calibration_precompute": calib,
        }
        print(json.dumps(line), flush=True)
    for lay in layers:
        for h in lay["h"].values():
            h.free()


def run_threshold_path(duo, shape, layers, px, reps, peak):
    """The threshold-mask path (§5, threshold-based activation sparsity) on
    the same layers: per stage a fixed threshold, here the magnitude of the
    (k+1)-th largest |x| of that layer's input, so that about k channels are
    kept (all of the top-k set when there is no tie there).  Required bytes
    use the kept set of the library's own (parity-tested) threshold
    sparsifier."""
    L = len(layers)
    taus, breq = [], 0.0
    for lay in layers:
        t = {}
        for st, src in zip(STAGES, STAGE_SRC):
            I = shape.I(st[0])
            k = k_of(I, px)
            a = lay["x"][src].float().abs()
            t[src] = float(torch.sort(a, descending=True).values[k].item()) if k < I else -1.0
            tau = max(t[src], 0.0)
            idx, _, cnt = duo.duo_sparsify_threshold(lay["x"][src], tau)
            n = int(cnt.item())
            K = idx[:n].to(torch.int64) & 0xFFFF
            for p in st:
                breq += float(lay["nnz"][p][K].sum().item()) * 2.0 + n * shape.O(p) / 8.0 + 4.0 * shape.O(p)
            breq += 2.0 * I + 4.0 * n
        taus.append(t)
    breq /= L

    def fn():
        for lay, t in zip(layers, taus):
            for st, src in zip(STAGES, STAGE_SRC):
                duo.duo_spmspv_threshold([lay["h"][p] for p in st], lay["x"][src], max(t[src], 0.0),
                                         ys=[lay["y"][p] for p in st])
    g = capture(fn)
    time_graph(g, 3)
    r = max(3, min(reps, 500))
    us = time_graph(g, r) / (r * L) * 1e6
    gbs = breq / (us * 1e-6) / 1e9
    return {"us_per_layer": us, "GB/s": gbs, "frac_of_peak": gbs / peak, "required_MB": breq / 1e6,
            "tau": "magnitude of the (k+1)-th largest |x| of each stage input, fixed before timing"}


def run_quant_path(duo, shape, layers, px, reps, peak, bits):
    """The same layer steps (fused top-k) over RTN-quantised stored values
    (§5, weight-only quantisation with group size 128, Table 4): b-bit codes
    in the records and one grid table per (segment, 128-channel group).
    Required bytes: b/8 bytes per kept stored weight, one mask bit per kept
    position, an fp16 scale and a b-bit zero point per (row, group holding a
    kept channel), plus x, the kept list and y."""
    L = len(layers)
    fmt = "bitmask_q8" if bits == 8 else "bitmask_q4"
    qh = [{p: duo.duo_pack(lay["W"][p], fmt) for p in lay["W"]} for lay in layers]
    packed = sum(h.query().data_bytes + h.query().aux_bytes for h in qh[0].values())
    breq = 0.0
    for lay in layers:
        for st, src in zip(STAGES, STAGE_SRC):
            I = shape.I(st[0])
            k = k_of(I, px)
            groups = 0
            if k > 0:
                idx, _ = duo.duo_sparsify(lay["x"][src], k)
                K = idx.to(torch.int64) & 0xFFFF
                groups = int(torch.unique(K // 128).numel())
            for p in st:
                O = shape.O(p)
                if k > 0:
                    breq += (float(lay["nnz"][p][K].sum().item()) * bits / 8.0 + k * O / 8.0
                             + (2.0 + bits / 8.0) * O * groups)
                breq += 4.0 * O
            breq += 2.0 * I + 4.0 * k
    breq /= L

    def fn():
        for lay, hq in zip(layers, qh):
            for st, src in zip(STAGES, STAGE_SRC):
                k = k_of(shape.I(st[0]), px)
                if len(st) == 1:
                    duo.duo_spmspv(hq[st[0]], lay["x"][src], k, y=lay["y"][st[0]])
                else:
                    duo.duo_spmspv_multi([hq[p] for p in st], lay["x"][src], k,
                                         ys=[lay["y"][p] for p in st])
    g = capture(fn)
    time_graph(g, 3)
    r = max(3, min(reps, 500))
    us = time_graph(g, r) / (r * L) * 1e6
    del g
    for hq in qh:
        for h in hq.values():
            h.free()
    gbs = breq / (us * 1e-6) / 1e9
    return {"us_per_layer": us, "GB/s": gbs, "frac_of_peak": gbs / peak, "required_MB": breq / 1e6,
            "packed_MB_per_layer": packed / 1e6, "bits": bits, "group": 128,
            "grid": "asymmetric min-max per (row, 128-channel group), fp16 scale, RTN"}


def run_calib(duo, reps):
    """DuoGPT's calibration precompute (§4.3, Algorithm 1) for one
    4096-channel layer from 2048 calibration tokens with half the channels
    kept per token (the setting of the paper's efficiency measurement):
    duo_calib_precompute (sparse input, H, act_order, dampening, inverse
    Cholesky, Q, U, a, b, c, D), the score S of a 4096 x 4096 weight, and
    the column sweep that prunes and compensates that weight.
    Synthetic inputs: Laplace(0, 1) activations, N(0, 0.02) weights."""
    k, m = 4096, 2048
    keep = k // 2
    g = torch.Generator(device="cuda").manual_seed(2506)
    u = torch.rand(m, k, generator=g, device="cuda", dtype=torch.float32) - 0.5
    X = (-torch.sign(u) * torch.log1p(-2 * u.abs())).to(torch.float16)
    W = (torch.randn(k, k, generator=g, device="cuda") * 0.02).to(torch.float16)
    c = duo.Calib(k, m)
    S = torch.empty(k, k, dtype=torch.float32, device="cuda")
    for _ in range(3):
        c.precompute(X, keep)
        c.score(W, S)
    status = c.status()
    r = max(3, min(reps // 20, 20))
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    ev[0].record()
    for _ in range(r):
        c.precompute(X, keep)
    ev[1].record()
    for _ in range(r):
        c.score(W, S)
    ev[2].record()
    torch.cuda.synchronize()
    pre_ms = ev[0].elapsed_time(ev[1]) / r
    score_ms = ev[1].elapsed_time(ev[2]) / r
    c.prune(W, 50, 128)                    # warm-up (grows the sweep scratch)
    rp = max(2, r // 4)
    ev[2].record()
    for _ in range(rp):
        c.prune(W, 50, 128)
    ev[3].record()
    torch.cuda.synchronize()
    prune_ms = ev[2].elapsed_time(ev[3]) / rp
    gemm_flop = 4.0 * k * k * m + 4.0 * k ** 3     # H, dX X_hat^T, Q, D as issued
    # the sweep's lazy products: per block of 128 columns, trailing columns
    # x 4096 rows x depth 256 (E and W_pre against -L and D^T)
    B = 128
    sweep_flop = sum(2.0 * (k - i - B) * k * 2 * B for i in range(0, k, B) if k - i - B > 0)
    c.free()
    return {"k": k, "m": m, "keep": keep, "status": status, "precompute_ms": pre_ms,
            "score_ms": score_ms, "sweep_ms": prune_ms,
            "sweep": "Algorithm 1 column sweep of a 4096 x 4096 weight, B = 128, 50% pruned per block",
            "gemm_GFLOP": gemm_flop / 1e9,
            "gemm_TFLOP/s_over_precompute": gemm_flop / (pre_ms * 1e-3) / 1e12,
            "sweep_gemm_GFLOP": sweep_flop / 1e9,
            "sweep_gemm_TFLOP/s_over_sweep": sweep_flop / (prune_ms * 1e-3) / 1e12,
            "paper_context": "about 1 ms for a, b, c and S of a 4096 x 4096 layer, m = 2048, A100 (App. C)"}


def run_e2e(duo, shape, layers, args, breq_mean):
    """End to end through the public API: every step copies that layer's
    inputs from pinned host memory to the device, runs the four stage calls
    and copies every output back.  Measured two ways: with duo.StepGraph
    (the step captured once, one replay call per step, one SM-kernel copy
    each way: the serving call) as the reported value, and with the
    individual calls and per-tensor copy-engine copies issued eagerly from
    Python each step."""
    L = len(layers)
    hx = [{s: layers[l]["x"][s].cpu().pin_memory() for s in STAGE_SRC} for l in range(L)]
    hy = [{p: torch.empty(shape.O(p), dtype=torch.float32).pin_memory() for p in layers[l]["y"]}
          for l in range(L)]
    h2d = sum(t.numel() * 2 for t in hx[0].values())
    d2h = sum(t.numel() * 4 for t in hy[0].values())
    n = min(args.steps, 2000)

    def timed(step):
        for i in range(min(args.warmup, 50)):
            step(i)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for i in range(n):
            step(i)
        torch.cuda.synchronize()
        return time.perf_counter() - t0

    plans = []
    for l in range(L):
        plan = duo.StepGraph([{"h": [layers[l]["h"][p] for p in st], "k": k_of(shape.I(st[0]), args.px)}
                              for st in STAGES])
        for si, src in enumerate(STAGE_SRC):
            plan.x_host(si).copy_(hx[l][src])   # the layer's inputs, written once on the host
        plans.append(plan)
    h2d_graph = sum(p._xh.numel() * 2 for p in plans[:1])
    d2h_graph = sum(p._yh.numel() * 4 for p in plans[:1])
    t_graph = timed(lambda i: plans[i % L].run())

    def eager(i):
        l = i % L
        lay = layers[l]
        for s in STAGE_SRC:
            lay["x"][s].copy_(hx[l][s], non_blocking=True)
        stage_calls(duo, shape, lay, args.px)()
        for p in lay["y"]:
            hy[l][p].copy_(lay["y"][p], non_blocking=True)
    t_eager = timed(eager)
    del plans
    return {"value": breq_mean * n / t_graph / 1e9, "unit": "GB/s", "us_per_layer": t_graph / n * 1e6,
            "h2d_bytes_per_step": h2d_graph, "d2h_bytes_per_step": d2h_graph, "steps": n,
            "api": "duo.StepGraph: the step's inputs copied in from pinned host memory and all "
                   "outputs copied back by the library's SM copy kernel (duo_copy), the 4 stage "
                   "calls between, replayed as one graph per step",
            "gpu_launches_per_step": 2 + len(STAGES),
            "eager_calls": {"value": breq_mean * n / t_eager / 1e9, "us_per_layer": t_eager / n * 1e6,
                            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}}


def run_dense(shape, layers, reps):
    L = len(layers)
    xs = [{p: layers[l]["x"][{"k": "q", "v": "q", "up": "gate"}.get(p, p)] for p in layers[l]["W"]}
          for l in range(L)]
    outs = [{p: torch.empty(shape.O(p), dtype=torch.float16, device=layers[0]["x"]["q"].device)
             for p in layers[l]["W"]} for l in range(L)]

    def run():
        for l in range(L):
            for p, W in layers[l]["W"].items():
                torch.matmul(W, xs[l][p], out=outs[l][p])
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        run()
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        run()
    time_graph(g, 3)
    t = time_graph(g, reps)
    us = t / (reps * L) * 1e6
    dense_bytes = sum(W.numel() * 2 + W.shape[1] * 2 + W.shape[0] * 2 for W in layers[0]["W"].values())
    return {"us_per_layer": us, "GB/s": dense_bytes / (us * 1e-6) / 1e9, "bytes_per_layer": dense_bytes}


def run_profile(args):
    """Small workload for profiler captures: packs 2 layers and runs
    `--steps` layer steps (4 fused spMspV launches each) without graphs."""
    torch.cuda.set_device(0)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo, synth
    duo.load_library()
    shape, layers = make_layers(duo, synth, 2, torch.device("cuda", 0), args.px)
    for i in range(args.steps):
        stage_calls(duo, shape, layers[i % 2], args.px)()
    torch.cuda.synchronize()
    assert duo.duo_device_status() == duo.DUO_OK
    print("profile workload done", flush=True)


def run_profile_coded(args):
    """One LLaMA-2-7B-shaped layer packed as fp16 records and as 8- and
    4-bit RTN codes; the four stages once per format, in that order (12
    fused launches), for profiler captures."""
    torch.cuda.set_device(0)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo, synth
    duo.load_library()
    wl = synth.WORKLOADS[WORKLOAD]
    shape = wl["shape"]
    W = {p: synth.layer_weight(wl, p, layer=0, device="cuda") for p in synth.PROJS}
    X = {s: synth.layer_input(wl, s, layer=0, device="cuda") for s in STAGE_SRC}
    for fmt in ("bitmask", "bitmask_q8", "bitmask_q4"):
        hs = {p: duo.duo_pack(W[p], fmt) for p in W}
        for st, src in zip(STAGES, STAGE_SRC):
            duo.duo_spmspv_multi([hs[p] for p in st], X[src], k_of(shape.I(st[0]), args.px))
        torch.cuda.synchronize()
        for h in hs.values():
            h.free()
    assert duo.duo_device_status() == duo.DUO_OK
    print("profile workload done", flush=True)


def run_profile_calib(args):
    """Calibration for profiler captures: one 4096-channel layer from 2048
    tokens, one warm-up and `--steps` precomputes, no graphs; with
    --profile-sweep one precompute and then `--steps` column sweeps of a
    4096 x 4096 weight (B = 128, 50% per block)."""
    torch.cuda.set_device(0)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo
    duo.load_library()
    k, m = 4096, 2048
    g = torch.Generator(device="cuda").manual_seed(2506)
    u = torch.rand(m, k, generator=g, device="cuda", dtype=torch.float32) - 0.5
    X = (-torch.sign(u) * torch.log1p(-2 * u.abs())).to(torch.float16)
    c = duo.Calib(k, m)
    for _ in range(1 if args.profile_sweep else 1 + args.steps):
        c.precompute(X, k // 2)
    assert c.status() == duo.DUO_OK
    if args.profile_sweep:   # Algorithm 1's column sweep, B = 128, 50% per block
        W = (torch.randn(k, k, generator=g, device="cuda") * 0.02).to(torch.float16)
        for _ in range(args.steps):
            c.prune(W, 50, 128)
        torch.cuda.synchronize()
        assert c.status() == duo.DUO_OK
    c.free()
    print("profile workload done", flush=True)


def measure_stack(duo, synth, dev, workload, L=None, pw=None, px=50, reps=20, warmup=3, dense=True):
    """Per-token time of a whole stack: every layer's four launches (q/k/v,
    o, gate/up, down) in one CUDA graph, each layer with its own packed
    weights and inputs (no rotation needed: a 32-80 layer stack is far above
    L2); with dense=True also cuBLAS fp16 GEMVs of the same dense weights
    (F.linear, the pruned weights with their zeros) through one graph per
    token, as the dense baseline the paper's speedups are quoted against."""
    wl = synth.WORKLOADS[workload]
    shape = wl["shape"]
    L = L or wl["layers"]
    pw = wl["pw"] if pw is None else pw
    ys = {p: torch.empty(shape.O(p), dtype=torch.float32, device=dev) for p in synth.PROJS}
    yd = {p: torch.empty(shape.O(p), dtype=torch.float16, device=dev) for p in synth.PROJS}
    layers, dense_w, breq, packed = [], [], 0.0, 0
    t0 = time.time()
    for l in range(L):
        hs, nnz, dw = {}, {}, {}
        for p in synth.PROJS:
            W = synth.layer_weight(wl, p, layer=l, device=dev, pw=pw)
            hs[p] = duo.duo_pack(W, "bitmask")
            nnz[p] = (W != 0).sum(dim=0).to(torch.int64)
            packed += hs[p].query().data_bytes + hs[p].query().index_bytes
            if dense:
                dw[p] = W
            else:
                del W
        xs = {s: synth.layer_input(wl, s, layer=l, device=dev) for s in STAGE_SRC}
        lay = dict(h=hs, nnz=nnz, x=xs, y=ys)
        breq += required_bytes_layer(duo, shape, lay, px)[0]
        del lay["nnz"]
        layers.append(lay)
        dense_w.append(dw)
    torch.cuda.synchronize()
    pack_s = time.time() - t0

    def fn():
        for lay in layers:
            for si in range(len(STAGES)):
                stage_call(duo, shape, lay, px, si)
    g = capture(fn)
    time_graph(g, max(3, warmup))
    sampler = ClockSampler(dev.index or 0)
    sampler.start()
    t = time_graph(g, reps)
    clocks = sampler.stop()
    assert duo.duo_device_status() == duo.DUO_OK
    us_token = t / reps * 1e6
    peak, peak_kind = peaks()
    gbs = breq / (us_token * 1e-6) / 1e9
    dense_bytes = 2.0 * L * sum(shape.O(p) * shape.I(p) for p in synth.PROJS)
    out = {"workload": workload, "layers": L, "pw": pw, "px": px, "us_per_token": us_token,
           "required_GB_per_token": breq / 1e9, "GB/s": gbs, "frac_of_peak": gbs / peak, "peak": peak,
           "peak_kind": peak_kind, "roofline_us_per_token": breq / (peak * 1e9) * 1e6,
           "dense_fp16_GB_per_token": dense_bytes / 1e9,
           "dense_roofline_us_per_token": dense_bytes / (peak * 1e9) * 1e6,
           "packed_GB": packed / 1e9, "pack_seconds": pack_s, "calls_per_token": 4 * L,
           "reps": reps, "clocks": clocks}
    if dense:
        def fd():
            for lay, dw in zip(layers, dense_w):
                for si, st in enumerate(STAGES):
                    xin = lay["x"][STAGE_SRC[si]]
                    for p in st:
                        torch.mv(dw[p], xin, out=yd[p])
        gd = capture(fd)
        time_graph(gd, 3)
        td = time_graph(gd, reps)
        out["dense_cublas_us_per_token"] = td / reps * 1e6
        out["speedup_vs_dense_cublas"] = out["dense_cublas_us_per_token"] / us_token
    del dense_w
    return out


def run_stack(args):
    """The stack alone (--stack WORKLOAD): one JSON line, not the default
    bench line."""
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo, synth
    duo.load_library()
    st = measure_stack(duo, synth, dev, args.stack, L=args.stack_layers, pw=args.stack_pw, px=args.px,
                       reps=max(5, min(args.steps, 200)), warmup=args.warmup if args.warmup < 50 else 5,
                       dense=not args.no_dense)
    line = {"metric": "per-token µs over the stack (batch-1 dual-sparse spMspV, every projection of every layer)",
            "value": st["us_per_token"], "unit": "us/token", "higher_is_better": False,
            "data": "synthetic", "dtype": "f16", **st}
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.profile:
        run_profile(args)
    elif args.profile_calib or args.profile_sweep:
        run_profile_calib(args)
    elif args.profile_coded:
        run_profile_coded(args)
    elif args.stack is not None:
        run_stack(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
