"""Benchmark: EmTrackMichelId hit identification on GB300.

One step = one pass of the whole hot path over one synthetic event: the
patch cut (time-interval image + gather), the fused conv + dense-1 tensor-core
kernel and the dense-2/heads kernel, for all 18 planes of a full 6-APA event
(15,360 wires x 6000 ticks, 60,000 hits) in one batched call
(emtk_infer_batch), bf16.  Inputs are device-resident when a timed step
starts; L2 is flushed (a 256 MiB write, then a 256 MiB read) between timed steps.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle on
the host cores instead, on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2009_04509_gb300 import synth  # noqa: E402

FLOP_CONV = 2 * 44 * 44 * 48 * 25          # 4,646,400 per hit (25 taps)
FLOP_FC1 = 2 * 92928 * 128                  # 23,789,568
FLOP_TAIL = 2 * (128 * 32 + 32 * 4)         # 8,448
FLOP_PER_HIT = FLOP_CONV + FLOP_FC1 + FLOP_TAIL  # 28,444,416
METRIC = "hit patches/sec on 1 GB300 (extract+CNN); % bf16 tensor peak; gather HBM GB/s"

# DRAM bytes (read + write) of one network-kernel launch on the full event, per
# precision, each from one ncu capture of this benchmark (profiles/launch_list_full_event_*.md),
# with the kernel source it was taken on: reported as null once that source changes.
TC_TRAFFIC = {
    "bf16": (51_517_440 + 9_344_512, "cnn_tc.cu", "d9c50f1f72130cf7"),
    "fp8": (38_985_728 + 3_194_880, "cnn_tc.cu", "d9c50f1f72130cf7"),
    "tf32": (979_775_744 + 435_545_600, "cnn_split.cu", "b3b11cc28934b03a"),
}


def tc_traffic(precision: str, workload: str):
    import hashlib
    if precision not in TC_TRAFFIC or workload != "full_event":
        return None
    nbytes, name, sha = TC_TRAFFIC[precision]
    src = os.path.join(ROOT, "paper_2009_04509_gb300", "csrc", name)
    if not os.path.exists(src):
        return None
    h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    return nbytes if h == sha else None


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


# The fp32 path runs on the CUDA cores: one FMA (2 FLOP) per lane per clock,
# 128 fp32 lanes per SM (4 sub-partitions x 32), 152 SMs, 2070 MHz maximum SM clock.
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2070e6 / 1e12
FP32_ALU_SOURCE = "derived: 152 SMs x 128 fp32 lanes x 2 FLOP (FMA) x 2070 MHz"


def network_peak(precision: str, peaks: dict, sustained: bool = False):
    """Peak of the network kernel (TFLOP/s).  The fp32 path is CUDA-core
    arithmetic, against the derived fp32 FMA rate.  Otherwise the tensor peak
    of the network kernel's own mix of operand types, the burst figure by
    default (the kernel is one launch of about a millisecond, timed alone by
    its own CUDA events) or the sustained one: the 16-bit paths run at the
    bf16 rate; the fp8 path runs the conv at the bf16 rate and dense-1 on
    e4m3 operands at twice it (the nominal fp8 : bf16 ratio), so its peak is
    the FLOP-weighted harmonic mix; the split-fp16 path (tf32) executes three
    16-bit products per fp32 product at the bf16 rate, so the algorithmic
    fp32 FLOPs it can reach are a third of that rate."""
    p = peaks["bf16_sus"] if sustained else peaks["bf16"]
    kind = "sustained" if sustained else "burst"
    if precision == "fp32":
        return FP32_ALU_TFLOPS, FP32_ALU_SOURCE
    if precision == "tf32":
        return p / 3.0, f"{peaks['source']} bf16 {kind} / 3 (three fp16 products per fp32 product)"
    if precision != "fp8":
        return p, f"{peaks['source']} bf16 {kind}"
    return ((FLOP_CONV + FLOP_FC1) / (FLOP_CONV / p + FLOP_FC1 / (2.0 * p)),
            f"{peaks['source']} bf16 {kind}; dense-1 e4m3 at 2x (nominal ratio), conv bf16")


def window_union_bytes(planes, patch=48, ds=6):
    """Bytes of ADC inside the union of all hits' patch windows (48 wires x
    48 intervals of 6 ticks), clipped to the plane, each sample counted once:
    the least the patch cut has to read."""
    total = 0
    half = patch // 2
    for p in planes:
        nint = p.nticks // ds
        cover = np.zeros((p.nwires + 1, nint + 1), np.int32)
        if p.nhits:
            w0 = np.clip(p.hits[:, 0].astype(np.int64) - half, 0, p.nwires)
            w1 = np.clip(p.hits[:, 0].astype(np.int64) + half, 0, p.nwires)
            b = np.floor_divide(p.hits[:, 1].astype(np.int64), ds)
            b0 = np.clip(b - half, 0, nint)
            b1 = np.clip(b + half, 0, nint)
            np.add.at(cover, (w0, b0), 1)
            np.add.at(cover, (w1, b0), -1)
            np.add.at(cover, (w0, b1), -1)
            np.add.at(cover, (w1, b1), 1)
        cov = np.cumsum(np.cumsum(cover, 0), 1)[: p.nwires, :nint] > 0
        total += int(cov.sum()) * ds * 4
    return total


def tiled_cut(planes):
    """Whether the tensor-core paths cut only the image tiles some window touches:
    the library does so once a launch's planes with hits hold 96 MiB of ADC."""
    return sum(p.nwires * p.nticks * 4 for p in planes if p.nhits) >= 96 << 20


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""
    Q = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.path = os.path.join("/tmp", f"emtk_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 10:
                continue
            if self.uuid and self.uuid not in parts[1]:
                continue
            rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in rows if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[6 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def gpu_uuid():
    import torch
    try:
        u = str(torch.cuda.get_device_properties(torch.cuda.current_device()).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return None


# ------------------------------------------------------------- CPU oracle
def cpu_oracle_rate(planes, weights, budget_s: float = 15.0):
    """Oracle hits/s on the host cores: the patch cut of every hit of the
    event, then the network on as many hits as fit the time budget."""
    import oracle
    oracle.build()
    lib = oracle.load()
    threads = oracle.max_threads(lib)
    t0 = time.perf_counter()
    nh = 0
    patches = []
    for p in planes:
        patches.append(oracle.extract_patches(p.adc, p.nticks, p.hits, lib=lib))
        nh += p.nhits
    t_cut = time.perf_counter() - t0
    allp = np.concatenate(patches)
    rng = np.random.default_rng(0)
    idx = rng.permutation(allp.shape[0])
    done, t_net, chunk = 0, 0.0, 4 * threads
    while t_net < budget_s and done < allp.shape[0]:
        sel = idx[done: done + chunk]
        t1 = time.perf_counter()
        oracle.forward(allp[sel], weights, lib=lib)
        t_net += time.perf_counter() - t1
        done += sel.size
    per_hit = t_cut / nh + t_net / done
    # the same network on one thread, on a few hits
    oracle.set_threads(1, lib=lib)
    n1 = min(8, allp.shape[0])
    t1 = time.perf_counter()
    oracle.forward(allp[idx[:n1]], weights, lib=lib)
    t_one = (time.perf_counter() - t1) / n1
    oracle.set_threads(threads, lib=lib)
    single = 1.0 / (t_cut / nh + t_one)
    return 1.0 / per_hit, threads, (f"patch cut of all {nh} hits ({t_cut:.2f} s) + network (fp64) on "
                                    f"{done} random hits ({t_net:.2f} s), {threads} OpenMP threads"), single


WORKLOADS = {
    "full_event": "full 6-APA event: 18 planes (800/800/960 wires) x 6000 ticks, 60,000 hits, one emtk_infer_batch",
    "apa": "one APA: planes 800/800/480 x 6000 ticks, 20,000 hits, one emtk_infer per plane",
    "single": "one collection plane: 480 wires x 6000 ticks, 256 hits on 5 tracks, one emtk_infer",
}


def workload_planes(workload: str, seed: int):
    if workload == "full_event":
        return synth.full_event(seed=seed)
    if workload == "apa":
        return synth.apa(seed=seed)
    return [synth.single_plane(seed=seed)]


def reduce_over_ranks(local_ms: float, local_units: int, dist, device):
    """Replicas (one independent event per rank, no exchange in the data
    path): the job's time is the slowest rank's, its work the sum of the
    ranks' units.  Returns (max ms, total units); single process: the inputs."""
    if not dist:
        return local_ms, local_units
    import torch
    t = torch.tensor([local_ms], dtype=torch.float64, device=device)
    u = torch.tensor([float(local_units)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), int(round(u.item()))


# -------------------------------------------------------------------- main
class L2Flush:
    """Between timed steps: a 256 MiB write (nothing the previous step
    touched stays in the 126 MB L2), then a 256 MiB read of another buffer,
    which writes the first one's dirty lines back to memory before the timed
    region starts instead of inside it."""
    WHAT = "flushed between steps (256 MiB write, then a 256 MiB read so that the write's dirty lines drain before the step)"

    def __init__(self, torch, dev):
        n = 256 * 1024 * 1024 // 4
        self.w = torch.empty(n, dtype=torch.float32, device=dev)
        self.r = torch.zeros(n, dtype=torch.float32, device=dev)
        self.acc = torch.zeros((), dtype=torch.float32, device=dev)
        self.torch = torch

    def __call__(self):
        self.w.zero_()
        self.torch.sum(self.r, dim=0, out=self.acc)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="emtk", choices=["emtk", "reference"])
    ap.add_argument("--workload", default="full_event", choices=["full_event", "apa", "single", "service", "sweep", "hitfind"])
    ap.add_argument("--clients", type=int, default=64, help="service workload: client threads (one event each)")
    ap.add_argument("--streams", type=int, default=8, help="service workload: batcher streams")
    ap.add_argument("--max-delay-us", type=int, default=500, help="service workload: batcher delay")
    ap.add_argument("--precision", default="bf16", choices=["bf16", "fp16", "fp8", "fp32", "tf32"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        return run_reference(args, rank, world)
    if args.workload == "service":
        return run_service(args, rank, world, local_rank)
    if args.workload == "sweep":
        return run_sweep(args, rank, world, local_rank)
    if args.workload == "hitfind":
        return run_hitfind(args, rank, world, local_rank)

    import torch
    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))

    from paper_2009_04509_gb300 import emtk
    planes = workload_planes(args.workload, rank)
    weights = synth.he_normal_weights(0)
    nhits = sum(p.nhits for p in planes)
    dev = torch.device("cuda", local_rank)
    adc = [torch.from_numpy(p.adc).to(dev) for p in planes]
    hits = [torch.from_numpy(p.hits).to(dev) for p in planes]
    scores = [torch.empty((p.nhits, 4), dtype=torch.float32, device=dev) for p in planes]
    items = [(a, p.nticks, h, s) for a, p, h, s in zip(adc, planes, hits, scores)]
    # the timed steps run on a context as a user creates it; the per-kernel
    # times (roofline, extraction) come from a second context that records
    # CUDA events around each launch, timed the same way (the events sit
    # between the kernels and keep them from overlapping, so that context's
    # steps are not the headline)
    ctx = emtk.emtk_create(weights, precision=args.precision, device=local_rank)
    ctx_prof = emtk.emtk_create(weights, precision=args.precision, device=local_rank, profile=True)
    flush = L2Flush(torch, dev)
    stream = torch.cuda.current_stream()

    def step(c=ctx):
        if args.workload == "full_event":
            emtk.emtk_infer_batch(c, items, stream)
        else:
            for it in items:
                emtk.emtk_infer(c, it[0], it[1], it[2], it[3], stream)

    for c in (ctx, ctx_prof):
        for _ in range(args.warmup):
            step(c)
        assert emtk.emtk_check(c, stream) == emtk.EMTK_OK

    # clocks are sampled every 200 ms from here to the end of the timed
    # region; untimed steps keep the GPU under the same load for at least a
    # second before it starts, so that the samples see the step's clocks
    clocks = ClockSampler(gpu_uuid())
    clocks.start()
    t_soak = time.perf_counter()
    while time.perf_counter() - t_soak < 1.0:
        for _ in range(10):
            step()
        torch.cuda.synchronize()
    assert emtk.emtk_check(ctx, stream) == emtk.EMTK_OK

    def timed(c):
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        for i in range(args.steps):
            flush()
            ev[i][0].record(stream)
            step(c)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        rc = emtk.emtk_check(c, stream)
        assert rc == emtk.EMTK_OK, emtk.status_string(rc)
        return [a.elapsed_time(b) for a, b in ev]

    base = emtk.emtk_get_stats(ctx)
    step_ms = timed(ctx)
    st = emtk.emtk_get_stats(ctx)
    base_prof = emtk.emtk_get_stats(ctx_prof)
    step_ms_prof = timed(ctx_prof)
    st_prof = emtk.emtk_get_stats(ctx_prof)
    clk = clocks.stop()
    total_ms, all_hits = reduce_over_ranks(float(sum(step_ms)), nhits * args.steps, dist, dev)
    ms_per_step = total_ms / args.steps
    value = all_hits / (total_ms / 1e3)

    kms = {k: st_prof["kernel_ms"][k] - base_prof["kernel_ms"][k] for k in emtk.KERNELS}
    kn = {k: st_prof["kernel_launches"][k] - base_prof["kernel_launches"][k] for k in emtk.KERNELS}
    launches = st["launches"] - base["launches"]
    peaks = load_peaks()
    net_ms = kms["network"] / max(1, kn["network"])
    hits_per_launch = nhits * args.steps / max(1, kn["network"])
    flop_net = (FLOP_CONV + FLOP_FC1) * hits_per_launch
    achieved = flop_net / (net_ms / 1e3) / 1e12
    net_peak, net_peak_src = network_peak(args.precision, peaks)
    net_peak_sus, _ = network_peak(args.precision, peaks, sustained=True)
    union = window_union_bytes(planes)
    if args.precision == "fp32":  # the fp32 path writes every patch
        patch_bytes = nhits * 48 * 48 * 4
    elif args.precision == "tf32":  # the split path writes 4-byte interval words
        patch_bytes = sum(p.nwires * (p.nticks // 6) for p in planes) * 4
    else:  # the 16-bit paths write the interval image; the network reads the windows from it
        patch_bytes = sum(p.nwires * (p.nticks // 6) for p in planes) * 2
    cut_ms = (kms["intervals"] + kms["gather"]) / args.steps
    cut_gbs = (union + patch_bytes) / (cut_ms / 1e3) / 1e9

    # end to end through the public call: host planes and hits in, scores out
    e2e = None
    if rank == 0 or world > 1:
        e2e = measure_e2e(emtk, ctx, planes, dev, stream, args, torch)

    out = {
        "metric": METRIC,
        "value": value,
        "unit": "hits/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms_per_step,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": args.precision,
        "data": "synthetic (seeded ProtoDUNE-SP-shaped planes and hits; He-normal seed-0 weights)",
        "config": {"workload": WORKLOADS[args.workload],
                   "hits_per_step": nhits, "planes": len(planes), "precision": args.precision,
                   "l2": L2Flush.WHAT + ("; planes (368.6 MB) exceed L2" if args.workload == "full_event" else ""),
                   "parallelism": f"replicas x{world} (independent events, no collective)"},
        "gpu_launches": launches,
        "roofline": {"bound": "alu" if args.precision == "fp32" else "tensor",
                     "kernel": {"fp32": "cnn_fp32_kernel",
                                "tf32": "cnn_split_kernel (conv 5x5x48 + dense-1, tcgen05, split fp16 operands)"}.get(
                         args.precision, "cnn_tc_kernel (conv 5x5x48 + dense-1, tcgen05)"),
                     "achieved": achieved, "peak": net_peak, "unit": "TFLOP/s",
                     "frac": achieved / net_peak,
                     "peak_source": net_peak_src, "frac_of_sustained": None if args.precision == "fp32"
                     else achieved / net_peak_sus,
                     "flop_per_hit": FLOP_CONV + FLOP_FC1, "hits_per_launch": hits_per_launch,
                     "launch_ms": net_ms, "traffic": tc_traffic(args.precision, args.workload),
                     "traffic_unit": "bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum)"},
        "extraction": {"bound": "hbm", "achieved": cut_gbs, "peak": peaks["hbm"], "unit": "GB/s",
                       "frac": cut_gbs / peaks["hbm"], "algorithmic_bytes": union + patch_bytes,
                       "bytes_read": union, "bytes_written": patch_bytes,
                       "kernels": "interval_image_kernel + gather_kernel" if args.precision == "fp32" else
                       ("mark_tiles_kernel + interval_tiles_kernel (the image tiles some window touches, and the "
                        "window descriptors)" if tiled_cut(planes) else
                        "interval_desc_kernel (images + window descriptors, one launch)"),
                       "ms_per_step": cut_ms},
        "step_ms_stats": {"median": statistics.median(step_ms), "min": min(step_ms), "max": max(step_ms),
                          "mean": total_ms / args.steps, "n": len(step_ms)},
        "kernel_ms_per_step": {k: v / args.steps for k, v in kms.items()},
        "kernel_times": "CUDA events around each launch, on a second context timed the same way "
                        f"(its steps: {statistics.median(step_ms_prof):.4f} ms median)",
        "whole_step_frac_of_bf16_peak": value * FLOP_PER_HIT / 1e12 / peaks["bf16"] / world,
        "clocks": clk,
    }
    if e2e:
        out["e2e"] = e2e
        # the paper's scale-out model (Sec. 3.3, Eqs. 2-5) with its CPU job and, as t_gpu, this
        # library's end-to-end throughput (the planes cross the host link inside it)
        from paper_2009_04509_gb300 import sonic
        job = sonic.gb300_job(e2e["value"])
        out["sonic_model"] = {"t_gpu_s_per_55k_inferences": job.t_gpu, "cpu_jobs_per_gpu": sonic.cpu_per_gpu(job),
                              "throughput": "e2e (emtk_infer_batch_host: host planes in, scores out)",
                              "paper_cpu_jobs_per_gpu_model": sonic.cpu_per_gpu(sonic.paper_job()),
                              "paper_measured": "about 68 CPU processes per T4 (270 on 4 GPUs)"}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rate, cores, sample, single = cpu_oracle_rate(planes, weights, args.cpu_budget)
        out["cpu_baseline"] = {"value": rate, "unit": "hits/s", "cores": cores, "kind": "oracle", "sample": sample,
                               "value_single_thread": single}
    emtk.emtk_destroy(ctx)
    emtk.emtk_destroy(ctx_prof)
    if rank == 0:
        print(json.dumps(out))
    if dist:
        dist.destroy_process_group()


def measure_e2e(emtk, ctx, planes, dev, stream, args, torch):
    """Same metric through the public call with host buffers
    (emtk_infer_batch_host): every step copies the event's planes (one pinned
    buffer, planes back to back) and hits from pinned host memory to the
    device, runs the batch and copies the scores back.  Calls are issued back to back, so the copy-in of one event
    overlaps the kernels of the one before (the library's two staging areas);
    wall clock over the steps, device synchronised on both sides.  The serial
    time (each call waited for before the next) is reported beside it."""
    # the event's planes back to back in one pinned buffer, as an event read from one
    # file would be: the call copies host-contiguous planes in one piece
    big = torch.empty(sum(p.adc.size for p in planes), dtype=torch.float32).pin_memory()
    h_adc, off = [], 0
    for p in planes:
        v = big[off:off + p.adc.size].view(p.adc.shape)
        v.copy_(torch.from_numpy(p.adc))
        h_adc.append(v)
        off += p.adc.size
    h_hits = [torch.from_numpy(p.hits).pin_memory() for p in planes]
    h_sc = [torch.empty((p.nhits, 4), dtype=torch.float32).pin_memory() for p in planes]
    items = [(a, p.nticks, h, s) for a, p, h, s in zip(h_adc, planes, h_hits, h_sc)]
    nhits = sum(p.nhits for p in planes)
    steps = max(3, min(args.steps, 30))
    for _ in range(3):
        emtk.emtk_infer_batch_host(ctx, items, stream)
    torch.cuda.synchronize()
    # three repetitions of `steps` calls, the median reported (on this machine about one run of
    # thirty calls in eight takes ~40% longer, whatever the build; every repetition is listed)
    reps = []
    for _ in range(3):
        t0 = time.perf_counter()
        for _ in range(steps):
            emtk.emtk_infer_batch_host(ctx, items, stream)
        torch.cuda.synchronize()
        reps.append((time.perf_counter() - t0) * 1e3 / steps)
    ms = statistics.median(reps)
    t0 = time.perf_counter()
    for _ in range(steps):
        emtk.emtk_infer_batch_host(ctx, items, stream)
        torch.cuda.synchronize()
    ms_serial = (time.perf_counter() - t0) * 1e3 / steps
    assert emtk.emtk_check(ctx, stream) == emtk.EMTK_OK
    h2d = sum(x.numel() * x.element_size() for x in h_adc + h_hits)
    d2h = sum(x.numel() * x.element_size() for x in h_sc)
    return {"value": nhits / (ms / 1e3), "unit": "hits/s", "ms_per_step": ms, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps, "call": "emtk_infer_batch_host",
            "timing": "wall clock over back-to-back calls (copy-in of one overlapping the kernels of the one before)",
            "host_layout": "the event's planes back to back in one pinned buffer; hit lists and scores per plane",
            "repetitions_ms_per_step": reps,
            "ms_per_step_serial": ms_serial, "value_serial": nhits / (ms_serial / 1e3)}


def _apa_event(seed):
    return synth.apa(seed=seed)


def run_service(args, rank, world, local_rank):
    """Service load: `clients` threads, each owning one synthetic one-APA event
    (3 planes, 20,000 hits, seeds 1..clients), submit their planes as separate
    requests to one request batcher and wait for the scores, round after round.
    Reports the sustained hits/s (wall clock over the timed rounds) and the
    per-request latency from submit to scores complete."""
    import concurrent.futures
    import multiprocessing
    import threading
    seeds = [1 + rank * args.clients + i for i in range(args.clients)]
    # events are drawn in spawned processes, before this process touches CUDA
    with concurrent.futures.ProcessPoolExecutor(max_workers=min(16, os.cpu_count() or 1),
                                                mp_context=multiprocessing.get_context("spawn")) as ex:
        events = list(ex.map(_apa_event, seeds))
    import torch
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    from paper_2009_04509_gb300 import emtk
    weights = synth.he_normal_weights(0)
    ctx = emtk.emtk_create(weights, precision=args.precision, device=local_rank)
    bat = emtk.emtk_batcher_create(ctx, nstreams=args.streams, max_hits=65536, max_delay_us=args.max_delay_us)
    bufs = [[(torch.from_numpy(p.adc).to(dev), p.nticks, torch.from_numpy(p.hits).to(dev),
              torch.empty((p.nhits, 4), dtype=torch.float32, device=dev)) for p in ev] for ev in events]
    torch.cuda.synchronize()
    hits_per_round = sum(p.nhits for ev in events for p in ev)
    lat, lock = [], threading.Lock()
    errors = []

    def client(c, rounds, record):
        mine = []
        try:
            for _ in range(rounds):
                sent = []
                for (a, nt, h, sc) in bufs[c]:
                    sent.append((emtk.emtk_batcher_submit(bat, a, nt, h, sc), time.perf_counter()))
                for t, t0 in sent:
                    rc = emtk.emtk_batcher_wait(bat, t)
                    if rc != emtk.EMTK_OK:
                        raise emtk.EmtkError(rc, "emtk_batcher_wait")
                    mine.append(time.perf_counter() - t0)
        except Exception as e:
            errors.append(e)
        if record:
            with lock:
                lat.extend(mine)

    def run(rounds, record):
        ths = [threading.Thread(target=client, args=(c, rounds, record)) for c in range(args.clients)]
        t0 = time.perf_counter()
        for t in ths:
            t.start()
        for t in ths:
            t.join()
        return time.perf_counter() - t0

    run(max(1, args.warmup), False)
    s0 = emtk.emtk_batcher_stats(bat)
    wall = run(args.steps, True)
    s1 = emtk.emtk_batcher_stats(bat)
    emtk.emtk_batcher_destroy(bat)
    emtk.emtk_destroy(ctx)
    if errors:
        raise errors[0]
    lat_ms = np.array(lat) * 1e3
    batches = s1["batches"] - s0["batches"]
    out = {"metric": "service load: hits/s sustained through the request batcher; p50/p99 request latency",
           "value": hits_per_round * args.steps / wall, "unit": "hits/s", "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": wall / args.steps * 1e3, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": args.precision,
           "data": "synthetic (seeded one-APA events, seeds 1..clients; He-normal seed-0 weights)",
           "config": {"workload": f"{args.clients} client threads x one APA event (3 planes 800/800/480 x 6000 "
                                  f"ticks, 20,000 hits), each plane a request; a step = every client's 3 requests",
                      "requests_per_step": 3 * args.clients, "hits_per_step": hits_per_round,
                      "streams": args.streams, "max_hits_per_batch": 65536, "max_delay_us": args.max_delay_us,
                      "precision": args.precision},
           "latency_ms": {"p50": float(np.percentile(lat_ms, 50)), "p99": float(np.percentile(lat_ms, 99)),
                          "max": float(lat_ms.max()), "requests": int(lat_ms.size)},
           "batches": {"count": batches, "mean_hits": (s1["hits"] - s0["hits"]) / max(1, batches),
                       "mean_requests": (s1["requests"] - s0["requests"]) / max(1, batches)},
           "timing": "host wall clock over the timed steps (a service metric); inputs resident on the device"}
    if rank == 0:
        print(json.dumps(out))


def run_sweep(args, rank, world, local_rank):
    """Inference-only batch sweep: pre-cut fp32 patches (70% zeros, else
    lognormal(2, 1)) through emtk_infer_patches at batch sizes 256 ... 65,536
    and the paper's 235, 1,693 and 5,358, bf16, fp8, tf32 and fp32 paths.  Per point:
    CUDA events around `steps` calls on the stream, inputs resident, after
    `warmup` calls."""
    import torch
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    from paper_2009_04509_gb300 import emtk
    weights = synth.he_normal_weights(0)
    sizes = [235, 256, 1024, 1693, 4096, 5358, 16384, 65536]
    x_all = torch.from_numpy(synth.inference_patches(max(sizes), seed=rank)).to(dev)
    sc = torch.empty((max(sizes), 4), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    table = []
    for prec in ("bf16", "fp8", "tf32", "fp32"):
        ctx = emtk.emtk_create(weights, precision=prec, device=local_rank)
        for n in sizes:
            x = x_all[:n]
            for _ in range(max(3, args.warmup)):
                emtk.emtk_infer_patches(ctx, x, sc[:n], stream)
            steps = max(3, min(args.steps, 200 if n <= 4096 else 5 if prec == "fp32" else 30))
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(steps):
                emtk.emtk_infer_patches(ctx, x, sc[:n], stream)
            b.record(stream)
            torch.cuda.synchronize()
            assert emtk.emtk_check(ctx, stream) == emtk.EMTK_OK
            ms = a.elapsed_time(b) / steps
            table.append({"precision": prec, "batch": n, "ms_per_batch": ms, "hits_per_s": n / (ms / 1e3),
                          "tflops": n * FLOP_PER_HIT / (ms / 1e3) / 1e12})
        emtk.emtk_destroy(ctx)
    best = max(r["hits_per_s"] for r in table if r["precision"] == "bf16")
    best_fp8 = max(r["hits_per_s"] for r in table if r["precision"] == "fp8")
    best_tf32 = max(r["hits_per_s"] for r in table if r["precision"] == "tf32")
    out = {"metric": "inference-only batch sweep: patches/s of emtk_infer_patches per batch size", "value": best,
           "unit": "hits/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": None, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "bf16, fp8, tf32 and fp32", "data": "synthetic (pre-cut patches, 70% zeros, lognormal(2,1))",
           "best_fp8": best_fp8, "best_tf32": best_tf32,
           "config": {"workload": "pre-cut 48x48 fp32 patches, batch sizes " + ", ".join(map(str, sizes)),
                      "includes": "network (the 16-bit and fp8 kernels read the fp32 patches and round them as they "
                                  "load them; tf32: a conversion launch to split-fp16 words first), heads"},
           "points": table}
    if rank == 0:
        print(json.dumps(out))


HITFIND_THRESHOLD = 15.0  # 5 sigma of the synthetic planes' noise
# DRAM bytes (read + write) of one hf_find_kernel launch on the full event, from one ncu
# capture of this workload (profiles/hitfind_full_event.md); null once hitfind.cu changes.
HF_TRAFFIC_BYTES = 369_188_864 + 4_362_496
HF_TRAFFIC_SOURCE_SHA256 = "2ba949573c38cacd"


def hf_traffic():
    import hashlib
    src = os.path.join(ROOT, "paper_2009_04509_gb300", "csrc", "hitfind.cu")
    if not os.path.exists(src):
        return None
    h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    return HF_TRAFFIC_BYTES if h == HF_TRAFFIC_SOURCE_SHA256 else None


def run_hitfind(args, rank, world, local_rank):
    """Hit finding on the full event: the 18 planes (15,360 wires x 6000
    ticks, 368.6 MB of fp32 samples) in one emtk_find_hits call per step,
    threshold 15 ADC.  Device time from CUDA events around each call on its
    stream (the call synchronises the stream to return the counts); L2
    flushed before every timed step.  Roofline: HBM, algorithmic bytes = each
    sample read once + the hits and runs written."""
    import torch
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    from paper_2009_04509_gb300 import emtk
    planes = synth.full_event(seed=rank)
    ctx = emtk.emtk_create(synth.he_normal_weights(0), precision="bf16", device=local_rank, profile=True)
    cap = 262_144
    items = [(torch.from_numpy(p.adc).to(dev), p.nticks, HITFIND_THRESHOLD,
              torch.empty((cap, 2), dtype=torch.int32, device=dev), torch.empty((cap, 4), dtype=torch.int32, device=dev))
             for p in planes]
    flush = L2Flush(torch, dev)
    stream = torch.cuda.current_stream()
    for _ in range(max(3, args.warmup)):
        found = emtk.emtk_find_hits(ctx, items, stream)
    clocks = ClockSampler(gpu_uuid())
    clocks.start()
    t_soak = time.perf_counter()
    while time.perf_counter() - t_soak < 1.0:
        emtk.emtk_find_hits(ctx, items, stream)
    base = emtk.emtk_get_stats(ctx)
    ms = []
    for _ in range(args.steps):
        flush()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        found = emtk.emtk_find_hits(ctx, items, stream)
        b.record(stream)
        b.synchronize()
        ms.append(a.elapsed_time(b))
    clk = clocks.stop()
    st = emtk.emtk_get_stats(ctx)
    emtk.emtk_destroy(ctx)
    nfound = sum(found)
    samples = sum(p.nwires * p.nticks for p in planes)
    kern_ms = (st["kernel_ms"]["hitfind"] - base["kernel_ms"]["hitfind"]) / args.steps
    step_ms = statistics.mean(ms)
    alg_bytes = samples * 4 + nfound * (8 + 16)
    peaks = load_peaks()
    out = {"metric": "hit finding: fp32 wire samples scanned/s (full event, threshold runs)", "impl": "emtk",
           "value": samples / (step_ms / 1e3), "unit": "samples/s", "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded ProtoDUNE-SP-shaped full event)",
           "config": {"workload": "full 6-APA event: 18 planes (800/800/960 wires) x 6000 ticks, threshold 15 ADC, "
                                  "one emtk_find_hits call",
                      "samples_per_step": samples, "hits_found": nfound,
                      "l2": L2Flush.WHAT + "; planes (368.6 MB) exceed L2"},
           "hits_per_s": nfound / (step_ms / 1e3),
           "roofline": {"bound": "hbm", "kernel": "hf_find_kernel + hf_place_kernel",
                        "achieved": alg_bytes / (kern_ms / 1e3) / 1e9, "peak": peaks["hbm"], "unit": "GB/s",
                        "frac": alg_bytes / (kern_ms / 1e3) / 1e9 / peaks["hbm"],
                        "peak_source": f"{peaks['source']} HBM copy", "algorithmic_bytes": alg_bytes,
                        "launch_ms": kern_ms, "traffic": hf_traffic(), "traffic_kernel": "hf_find_kernel",
                        "traffic_unit": "bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum)"},
           "clocks": clk}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        lib = oracle.load()
        t0 = time.perf_counter()
        reps = 0
        while time.perf_counter() - t0 < 2.0:  # whole steps, at least 2 s
            n_cpu = sum(oracle.find_hits(p.adc, p.nticks, HITFIND_THRESHOLD, lib=lib)["wire"].size for p in planes)
            reps += 1
        t_cpu = (time.perf_counter() - t0) / reps
        out["cpu_baseline"] = {"value": samples / t_cpu, "unit": "samples/s", "cores": 1, "kind": "oracle",
                               "sample": f"whole steps: or_find_hits on all 18 planes, {reps} times "
                                         f"({t_cpu:.3f} s each, {n_cpu} hits), one thread"}
    if rank == 0:
        print(json.dumps(out))


def run_reference(args, rank, world):
    """The oracle on the host cores, on the same workload.  Every step is a
    fixed-size sample of the workload's hits, different hits each step: the
    patch cut of those hits from their planes and the fp64 network on them.
    The sample size is set once, before the warm-up steps, so that a step
    takes about `budget` seconds; each step is timed with the host clock."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    lib = oracle.load()
    threads = oracle.max_threads(lib)
    planes = workload_planes(args.workload, 0)
    weights = synth.he_normal_weights(0)
    budget = max(1.0, min(args.cpu_budget, 120.0 / max(1, args.steps + args.warmup)))
    where = np.concatenate([np.stack([np.full(p.nhits, i), np.arange(p.nhits)], 1) for i, p in enumerate(planes)])
    order = where[np.random.default_rng(0).permutation(len(where))]
    nh = len(order)

    def step(k0, n):
        sel = order[np.arange(k0, k0 + n) % nh]
        t0 = time.perf_counter()
        patches = [oracle.extract_patches(planes[i].adc, planes[i].nticks, planes[i].hits[sel[sel[:, 0] == i, 1]],
                                          lib=lib) for i in np.unique(sel[:, 0])]
        oracle.forward(np.concatenate(patches), weights, lib=lib)
        return time.perf_counter() - t0

    # sample size: about `budget` seconds of work at the rate of a short first run
    probe = 4 * threads
    rate = probe / step(0, probe)
    n_s = int(min(nh, max(threads, round(rate * budget / threads) * threads)))
    k = probe
    secs = []
    for i in range(args.warmup + args.steps):
        t = step(k, n_s)
        k += n_s
        if i >= args.warmup:
            secs.append(t)
    # the network on one thread, on a few hits, for the single-core figure
    oracle.set_threads(1, lib=lib)
    t1 = step(k, 8)
    oracle.set_threads(threads, lib=lib)
    total = float(sum(secs))
    value = n_s * len(secs) / total
    sample = (f"each step: patch cut + fp64 network of {n_s} hits (different hits each step, "
              f"{n_s * len(secs)} over the timed steps) of the {nh}-hit workload, {threads} OpenMP threads")
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": "hits/s", "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": total / len(secs) * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": WORKLOADS.get(args.workload, args.workload) + " (CPU oracle, sampled)",
                      "hits_per_step": n_s, "workload_hits": nh},
           "step_ms_stats": {"median": statistics.median(secs) * 1e3, "min": min(secs) * 1e3,
                             "max": max(secs) * 1e3, "n": len(secs)},
           "cpu_baseline": {"value": value, "unit": "hits/s", "cores": threads, "kind": "oracle", "sample": sample,
                            "value_single_thread": 8 / t1},
           "e2e": {"value": value, "unit": "hits/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))


if __name__ == "__main__":
    main()
