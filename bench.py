#!/usr/bin/env python3
"""Benchmark of the certified cache lookup on GB300.

A step is one batch of the online lookup (Algorithm 2: certified screen,
recheck and nearest-hit selection) against a cache built beforehand with the
certified insertion of Algorithm 1. Default workload: the scale stress case,
a 4,000,000-entry cache of d = 128 FP32 GuardNet-like features (C = 200
classes, Lipschitz-constrained head) probed in batches of 4,096 queries, 25%
of them near-duplicates of cached rows. Inputs are seeded synthetic data
(synth.py); the key table (2.06 GB) is larger than L2, so no L2 flush is
needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # FP64 CPU oracle on host cores

Prints one JSON line (rank 0). The lookup runs on one GPU: its tensor-core
probe kernels load query tiles with TMA multicast inside a thread-block
cluster, which is meant for single-GPU runs only, so the GPU arm refuses to
start under torchrun with WORLD_SIZE > 1 (exit status 2, one JSON line that
says why). The reference arm (the CPU oracle) runs on rank 0 alone there.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "certified probe queries/s and query-key pairs/s at N=4M; % of HBM/TC roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
TF32_OVER_BF16 = 1.1 / 2.25  # nominal dense TF32 / BF16 tensor rates of GB300
# LIPCACHE_DEBUG_INSERT_WIDE_TILE / LIPCACHE_DEBUG_INSERT_TILE64 of the C ABI
INSERT_KERNEL_FLAGS = {"auto": 0, "wide": 4, "tile64": 2}
DEBUG_INSERT_FIX_STANDALONE = 16  # LIPCACHE_DEBUG_INSERT_FIX_STANDALONE


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="scale", choices=sorted(synth.WORKLOADS))
    p.add_argument("--path", default="auto", choices=["auto", "tensor", "tensor_single", "tensor_pair", "exact"])
    p.add_argument("--cpu-seconds", type=float, default=15.0, help="budget of the oracle CPU baseline")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-tf32-peak", action="store_true", help="skip the live cuBLAS TF32 peak measurement")
    p.add_argument("--sustain-s", type=float, default=3.0,
                   help="seconds of back-to-back probe steps after the timed region, reported as `sustained` "
                        "with their clocks (0: skip)")
    p.add_argument("--cache-rows", type=int, default=0, help="override the workload's cache size N (profiling)")
    p.add_argument("--noise", type=float, default=None,
                   help="override the near-duplicate queries' per-feature noise (e.g. 0.002: most of them hit)")
    p.add_argument("--dup", type=float, default=None, help="override the fraction of near-duplicate queries")
    p.add_argument("--insert-kernel", default="auto", choices=sorted(INSERT_KERNEL_FLAGS),
                   help="certify on an FP32 kernel instead of the default choice (profiling)")
    p.add_argument("--insert-fp64-pass", default="kernel", choices=["kernel", "standalone"],
                   help="where the tensor certify kernel's listed rows are re-certified in FP64: on its own "
                        "spare warp (default) or by the stand-alone pass launched after it (profiling)")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ---------------------------------------------------------------- distributed plumbing
class Dist:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local_rank = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist
            os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
            dist.init_process_group("gloo", rank=self.rank, world_size=self.world)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def sum(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.SUM)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


def aggregate(dist: Dist, units: float, seconds: float) -> tuple[float, float]:
    """Whole-job throughput: units of all ranks over the slowest rank's time."""
    total = dist.sum(units)
    tmax = dist.max(seconds)
    return total / tmax, tmax


# ---------------------------------------------------------------- clocks
class Clocks:
    FIELDS = ["index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu_index: int):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", "--query-gpu=" + ",".join(self.FIELDS),
                                       "--format=csv,noheader,nounits", "-i", str(gpu_index), "-lms", "100"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        self.t0 = self.t1 = None

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    def stop(self) -> dict:
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.15)
        self.p.terminate()
        self.p.wait()
        self.f.seek(0)
        rows = [r.split(",") for r in self.f.read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax.append(float(r[2]))
            except ValueError:
                continue
            for name, v in zip(names, r[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------- workload
def workload_of(args) -> synth.Workload:
    w = synth.WORKLOADS[args.workload]
    if args.cache_rows:
        w = w.scaled(N=args.cache_rows)
    if args.noise is not None:
        w = w.scaled(noise=args.noise)
    if args.dup is not None:
        w = w.scaled(dup_frac=args.dup)
    return w


def workload_data(w: synth.Workload):
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    Q, _ = synth.queries(w, rows)
    return W, b, rows, Q


def roofline(w: synth.Workload, N: int, B: int, kernel_ms: float, pk: dict, pk_kind: str,
             kernel: str = "k_probe_tc") -> dict:
    flops = 2.0 * B * N * w.d
    bytes_ = N * (4.0 * w.d + 4.0) + 4.0 * B * w.d + 16.0 * B
    tf32_peak = pk["bf16_tflops"] * TF32_OVER_BF16
    hbm_peak = pk["hbm_gbs"]
    t_tc = flops / (tf32_peak * 1e12)
    t_hbm = bytes_ / (hbm_peak * 1e9)
    s = kernel_ms * 1e-3
    if t_tc >= t_hbm:
        ach = flops / s / 1e12
        return {"bound": "tensor", "achieved": ach, "peak": tf32_peak, "unit": "TFLOP/s", "frac": ach / tf32_peak,
                "traffic": None, "algorithmic_flops": flops, "algorithmic_bytes": bytes_,
                "peak_source": f"{pk_kind} bf16 burst x nominal tf32/bf16 ratio {TF32_OVER_BF16:.4f}",
                "kernel": kernel, "kernel_ms": kernel_ms,
                "hbm_frac": bytes_ / s / 1e9 / hbm_peak}
    ach = bytes_ / s / 1e9
    return {"bound": "hbm", "achieved": ach, "peak": hbm_peak, "unit": "GB/s", "frac": ach / hbm_peak,
            "traffic": None, "algorithmic_flops": flops, "algorithmic_bytes": bytes_,
            "peak_source": f"{pk_kind} copy bandwidth", "kernel": kernel, "kernel_ms": kernel_ms}


def event_floor_ms(dev, reps: int = 50) -> float:
    """CUDA-event interval of a one-element kernel launched right after
    another small kernel, bracketed the way the library brackets each probe
    kernel (event, kernel, event): the fixed cost inside every per-kernel
    interval on this GPU (kernel launch and completion), median of `reps`."""
    import torch

    x = torch.zeros(1, device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    stream = torch.cuda.current_stream(dev)
    out = []
    for i in range(reps + 5):
        # the GPU sleeps while the rest is queued, so the interval holds no
        # host-side launch time (as in the probe's timed loop, where the host
        # runs ahead of the GPU)
        torch.cuda._sleep(1_000_000)
        x.add_(1.0)
        e0.record(stream)
        x.mul_(1.0)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        if i >= 5:
            out.append(e0.elapsed_time(e1))
    return statistics.median(out)


def measure_tf32_peak(dev, n: int = 8192, reps: int = 10, sustain_s: float = 2.0) -> dict:
    """Dense TF32 tensor throughput of this GPU, measured in this run the way
    the BF16 peak of MEASURED_PEAKS.json was: a cuBLAS (torch.matmul) FP32 GEMM
    with TF32 tensor cores allowed, n^3 with n = 8192 (2 n^3 flops), best of
    `reps` timed with CUDA events (burst), then back to back for `sustain_s`
    seconds (sustained), with nvidia-smi clocks sampled meanwhile. A
    measurement for the roofline only; the lookup never calls cuBLAS."""
    import torch
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = True
    try:
        g = torch.Generator(device=dev).manual_seed(1)
        a = torch.randn(n, n, device=dev, generator=g)
        b = torch.randn(n, n, device=dev, generator=g)
        c = torch.empty(n, n, device=dev)
        for _ in range(3):
            torch.matmul(a, b, out=c)
        torch.cuda.synchronize(dev)
        clk = Clocks(dev.index)
        clk.mark_start()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        best = float("inf")
        for _ in range(reps):
            e0.record()
            torch.matmul(a, b, out=c)
            e1.record()
            torch.cuda.synchronize(dev)
            best = min(best, e0.elapsed_time(e1) * 1e-3)
        k, t0 = 0, time.perf_counter()
        e0.record()
        while time.perf_counter() - t0 < sustain_s:
            for _ in range(10):
                torch.matmul(a, b, out=c)
            k += 10
            torch.cuda.synchronize(dev)
        e1.record()
        torch.cuda.synchronize(dev)
        sustained = 2.0 * n ** 3 * k / (e0.elapsed_time(e1) * 1e-3) / 1e12
        clk.mark_end()
        clocks = clk.stop()
        del a, b, c
        return {"burst_tflops": 2.0 * n ** 3 / best / 1e12, "sustained_tflops": sustained, "clocks": clocks,
                "how": f"torch.matmul FP32 {n}^3 with TF32 tensor cores (cuBLAS): best of {reps} (burst), "
                       f"back to back for {sustain_s:.0f} s (sustained)"}
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev


# main probe kernel per path: name, ncu summary, the sources its hash covers
INSERT_KERNELS = {1: "k_certify_wt", 2: "k_certify_wres", 3: "k_certify", 4: "k_certify_tc"}
PROBE_KERNELS = {
    4: ("k_probe_pair", "k_probe_pair_scale.md", ("probe_pair.cu", "tc_ptx.cuh", "probe_common.cuh")),
    3: ("k_probe_tc", "k_probe_tc_scale.md", ("probe_tc.cu", "tc_ptx.cuh", "probe_common.cuh")),
    2: ("k_probe_exact", None, ()),
}


def recorded_traffic(workload: str, path_id: int = 3):
    """DRAM bytes per probe launch recorded in the kernel's profiles/ summary
    from an ncu capture, or None when the kernel sources changed since."""
    import hashlib
    name, summary, sources = PROBE_KERNELS[path_id]
    if summary is None:
        return None
    path = os.path.join(ROOT, "profiles", summary)
    if not os.path.exists(path):
        return None
    rec = {}
    for line in open(path):
        line = line.strip()
        for key in ("traffic_bytes_per_launch", "traffic_workload", "sources_sha256_16"):
            if line.startswith(key + ":"):
                rec[key] = line.split(":", 1)[1].strip()
    h = hashlib.sha256()
    for f in sources:
        with open(os.path.join(ROOT, "paper_2608_13144_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    if rec.get("sources_sha256_16") != h.hexdigest()[:16] or rec.get("traffic_workload") != workload:
        return None
    return float(rec["traffic_bytes_per_launch"])


def cpu_baseline(w, W, b, rows, Q, budget_s: float, gpu=None):
    """The FP64 oracle as it stands, on the host cores, on a bounded sample:
    the first n queries against the whole cache (n sized to the budget).
    With gpu = (index, label, dist) of the GPU's first batch, also compares
    the sampled queries with the GPU's answers (untimed): returns
    (baseline, parity) where parity counts identical answers, the oracle's
    1e-5 band, disagreements inside and outside it, and unsafe accepts (GPU
    hits the oracle's FP64 distance and radius reject)."""
    import oracle
    t0 = time.perf_counter()
    sigma = oracle.sigma_max(W)
    cache = oracle.build_cache(W, b, sigma, rows)
    t_build = time.perf_counter() - t0
    n = max(1, oracle.threads())
    t0 = time.perf_counter()
    res = [oracle.probe(cache["keys"], cache["radius"], cache["label"], Q[:n])]
    t1 = time.perf_counter() - t0
    total_q, total_t = n, t1
    if t1 < budget_s:
        m = int(min(len(Q) - n, max(0, (budget_s - t1) / t1 * n)))
        if gpu is not None:
            m = min(m, len(gpu[0]) - n)
        if m > 0:
            t0 = time.perf_counter()
            res.append(oracle.probe(cache["keys"], cache["radius"], cache["label"], Q[n:n + m]))
            total_t += time.perf_counter() - t0
            total_q += m
    N = len(cache["keys"])
    base = {"value": total_q / total_t, "unit": "queries/s", "cores": oracle.threads(), "kind": "oracle",
            "pairs_per_s": total_q * N / total_t,
            "sample": f"{total_q} queries of the '{w.name}' workload against the full {N}-entry cache "
                      f"(FP64 brute force, {total_t:.1f} s; oracle cache build {t_build:.1f} s untimed)"}
    if gpu is None:
        return base, None
    orc = {k: np.concatenate([r[k] for r in res]) for k in ("index", "label", "decision_band", "selection_band")}
    gi, gl = gpu[0][:total_q], gpu[1][:total_q]
    band = (orc["decision_band"] | orc["selection_band"]).astype(bool)
    same = (gi == orc["index"]) & (gl == orc["label"])
    hit = np.nonzero(gi >= 0)[0]
    unsafe = 0
    if hit.size:
        D = oracle.pair_dist(Q[:total_q], cache["keys"], hit, gi[hit])
        unsafe = int((~(D < cache["radius"][gi[hit]])).sum())
    parity = {"queries": int(total_q), "identical": int(same.sum()), "band": int(band.sum()),
              "mismatch_in_band": int((~same & band).sum()), "mismatch_outside_band": int((~same & ~band).sum()),
              "unsafe_accepts": unsafe, "gpu_hits": int(hit.size), "oracle_hits": int((orc["index"] >= 0).sum()),
              "sample": "the cpu_baseline queries (the first batch's first ones) against the oracle's FP64 cache"}
    return base, parity


# ---------------------------------------------------------------- our arm
SINGLE_GPU_ONLY = ("the GPU arm runs on one GPU only: its tensor-core probe kernels use TMA cluster "
                   "multicast, which is kept to single-GPU runs")


def run_ours(args, dist: Dist):
    import torch

    from paper_2608_13144_gb300.lipcache import LipCache

    w = workload_of(args)
    dev = torch.device("cuda", dist.local_rank)
    torch.cuda.set_device(dev)
    pk, pk_kind = peaks()
    W, b, rows, Q = workload_data(w)
    stream = torch.cuda.current_stream(dev)

    rows_d = torch.from_numpy(rows).to(dev)

    def build(mode):
        """Certified insertion (Algorithm 1) of every row, timed separately:
        CUDA events around the insert calls (asynchronous: no host count per
        call; the accepted total comes from the size afterwards), and the
        library's events around each certify kernel."""
        c = LipCache(w.d, w.C, w.N, mode, device=dev)
        flags = INSERT_KERNEL_FLAGS[args.insert_kernel] | (
            DEBUG_INSERT_FIX_STANDALONE if args.insert_fp64_pass == "standalone" else 0)
        if flags:
            c.set_debug(flags)
        sig = c.set_head(torch.from_numpy(W).to(dev), torch.from_numpy(b).to(dev))
        torch.cuda.synchronize(dev)
        c.enable_timing(True)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s, e in synth.batches(w.N, w.insert_batch):
            c.insert(rows_d[s:e], wait=False)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        acc = c.size
        inf = c.info()
        c.enable_timing(False)
        kern = (INSERT_KERNELS.get(inf["last_insert_kernel"], "?"), inf["insert_kernel_ms_total"],
                inf["insert_kernel_launches"], inf["insert_refined_pairs"], inf["insert_full_rows"],
                inf["insert_fp64_rows"])
        return c, sig, acc, e0.elapsed_time(e1), kern

    # the tight radius (Eq. 29, Sec. 5.6) on the same rows, then the
    # conservative radius (Eq. 21) whose cache the probe uses
    tcache, _, n_acc_t, insert_ms_t, insert_kernel_t = build("tight")
    tcache.close()
    del tcache
    cache, sigma, n_acc, insert_ms, insert_kernel = build("conservative")
    del rows_d
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    cache.set_probe_path(args.path)
    cache.reserve(w.batch)
    N = cache.size

    # query batches resident in HBM
    nb = max(1, len(Q) // w.batch)
    Qd = torch.from_numpy(Q[: nb * w.batch]).to(dev).view(nb, w.batch, w.d)
    B = w.batch
    outs = [(torch.empty(B, dtype=torch.int64, device=dev), torch.empty(B, dtype=torch.int32, device=dev),
             torch.empty(B, dtype=torch.float32, device=dev)) for _ in range(nb)]
    for i in range(args.warmup):
        cache.probe(Qd[i % nb], out=outs[i % nb])
    torch.cuda.synchronize(dev)
    cache.reset_stats()
    cache.enable_timing(True)

    clk = Clocks(dist.local_rank)
    dist.barrier()
    torch.cuda.synchronize(dev)
    clk.mark_start()
    e0.record(stream)
    for i in range(args.steps):
        cache.probe(Qd[i % nb], out=outs[i % nb])
    e1.record(stream)
    torch.cuda.synchronize(dev)
    clk.mark_end()
    dist.barrier()
    step_s = e0.elapsed_time(e1) * 1e-3
    clocks = clk.stop()
    info = cache.info()
    cache.enable_timing(False)
    kernel_ms = info["kernel_ms_total"] / max(1, info["kernel_launches"])
    hits = sum(int((o[0] >= 0).sum()) for o in outs[: min(nb, args.steps)])
    hit_rate = hits / (min(nb, args.steps) * B)

    value, tmax = aggregate(dist, args.steps * B, step_s)

    # the same step back to back for a few seconds, with its clocks: the
    # figure under the power cap beside the short timed region's
    sustained = None
    if args.sustain_s > 0:
        cache.reset_stats()
        cache.enable_timing(True)
        clk2 = Clocks(dist.local_rank)
        torch.cuda.synchronize(dev)
        clk2.mark_start()
        s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s0.record(stream)
        n_sus, t_wall = 0, time.perf_counter()
        while time.perf_counter() - t_wall < args.sustain_s:
            for _ in range(16):
                cache.probe(Qd[n_sus % nb], out=outs[n_sus % nb])
                n_sus += 1
            torch.cuda.synchronize(dev)
        s1.record(stream)
        torch.cuda.synchronize(dev)
        clk2.mark_end()
        sus_s = s0.elapsed_time(s1) * 1e-3
        inf2 = cache.info()
        cache.enable_timing(False)
        k2_ms = inf2["kernel_ms_total"] / max(1, inf2["kernel_launches"])
        sustained = {"value": n_sus * B / sus_s, "unit": "queries/s", "steps": n_sus, "seconds": sus_s,
                     "kernel_ms": k2_ms, "kernel_tflops": 2.0 * B * N * w.d / (k2_ms * 1e-3) / 1e12,
                     "clocks": clk2.stop()}

    # end to end through the host-buffer entry point: H2D of the queries,
    # probe, D2H of index/label/distance, every step
    hq = [torch.from_numpy(np.ascontiguousarray(Q[i * B:(i + 1) * B])).pin_memory() for i in range(nb)]
    ho = [(torch.empty(B, dtype=torch.int64).pin_memory(), torch.empty(B, dtype=torch.int32).pin_memory(),
           torch.empty(B, dtype=torch.float32).pin_memory()) for _ in range(nb)]
    for i in range(min(3, args.warmup + 1)):
        cache.probe_host(hq[i % nb], out=ho[i % nb])
    e2e_steps = max(1, min(args.steps, 50))
    dist.barrier()
    t0 = time.perf_counter()
    for i in range(e2e_steps):
        cache.probe_host(hq[i % nb], out=ho[i % nb])
    e2e_s = time.perf_counter() - t0
    e2e_value, _ = aggregate(dist, e2e_steps * B, e2e_s)

    cpu = parity = None
    if dist.rank == 0 and not args.no_cpu_baseline:
        g0 = [t.cpu().numpy() for t in outs[0]]  # the first batch, Q[:B]
        cpu, parity = cpu_baseline(w, W, b, rows, Q, args.cpu_seconds, gpu=g0)
    cache.close()

    path_id = info["last_probe_path"]
    rf = roofline(w, N, B, kernel_ms, pk, pk_kind, PROBE_KERNELS[path_id][0])
    tf32_derived = pk["bf16_tflops"] * TF32_OVER_BF16
    if rf["bound"] == "tensor" and not args.no_tf32_peak:
        # the TF32 peak measured live beside the derived one (MEASURED_PEAKS.json holds BF16 only)
        tf = measure_tf32_peak(dev)
        tf["frac_of_burst"] = rf["achieved"] / tf["burst_tflops"]
        tf["frac_of_sustained"] = rf["achieved"] / tf["sustained_tflops"]
        rf["tf32_measured"] = tf
    if path_id in (3, 4) and w.N == synth.WORKLOADS[w.name].N:
        rf["traffic"] = recorded_traffic(w.name, path_id)
    # context for short kernels: the part of each per-kernel event interval
    # that any kernel pays (launch, completion); the fraction above is not
    # corrected for it
    rf["event_floor_ms"] = event_floor_ms(dev)
    line = {
        "metric": METRIC, "value": value, "unit": "queries/s", "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": tmax / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "tf32" if info["last_probe_path"] in (3, 4) else "fp32",
        "data": "synthetic (seeded Gaussian-mixture GuardNet features; no datasets or trained weights)",
        "config": {"workload": w.name, "N": N, "d": w.d, "C": w.C, "batch": B, "radius": "conservative",
                   "near_duplicates": w.dup_frac, "near_duplicate_noise": w.noise,
                   "probe_path": {2: "exact", 3: "tensor_single", 4: "tensor_pair"}[info["last_probe_path"]],
                   "parallelism": "single",
                   "l2": f"inputs larger than L2 ({N * (4 * info['d_pad'] + 16) / 1e9:.2f} GB key table)"},
        "pairs_per_s": value * N,
        "roofline": rf,
        "cpu_baseline": cpu,
        "parity": parity,
        "e2e": {"value": e2e_value, "unit": "queries/s", "h2d_bytes_per_step": B * w.d * 4,
                "d2h_bytes_per_step": B * (8 + 4 + 4)},
        "gpu_launches": 3 * args.steps,
        "sustained": sustained,
        "clocks": clocks,
        "insert": insert_summary(w, n_acc, insert_ms, torch.cuda.get_device_properties(dev).multi_processor_count,
                                 clocks, kernel=insert_kernel, tf32_peak=tf32_derived, hbm_peak=pk["hbm_gbs"]),
        "insert_tight": insert_summary(w, n_acc_t, insert_ms_t,
                                       torch.cuda.get_device_properties(dev).multi_processor_count, clocks,
                                       kernel=insert_kernel_t, tf32_peak=tf32_derived, hbm_peak=pk["hbm_gbs"]),
        "stats": {"sigma": sigma, "hit_rate": hit_rate,
                  "candidates_per_query": info["candidates"] / max(1, args.steps * B),
                  "device_errors": info["device_errors"], "kernel_ms": kernel_ms,
                  "grid": info["last_grid"], "cluster": info["last_cluster"]},
    }
    for k in ("insert", "insert_tight"):
        line[k]["fp64_pass"] = "stand-alone kernel" if args.insert_fp64_pass == "standalone" else "in the kernel"
    return line


def insert_summary(w, n_acc, insert_ms, sms, clocks, kernel=None, tf32_peak=None, hbm_peak=None):
    """Certified insertion of the whole cache (Algorithm 1). Algorithmic work
    per row: 2 C d flops (the head contraction) and 8 d + 16 bytes (the row
    read, its key written to the table, the per-entry fields). The tensor
    kernel (k_certify_tc) runs the contraction as TF32 MMAs, so the larger of
    the byte time at the HBM peak and the flop time at the TF32 peak bounds
    it, and that is the byte time: `roofline` reports it against the measured
    HBM copy bandwidth, with the flops against the TF32 and FP32-ALU peaks
    beside it. The FP32 certify kernels run the contraction on the CUDA cores:
    roofline the FP32 ALU (SM count x 128 FP32 lanes x 2 flops x the maximum
    SM clock seen by nvidia-smi). `roofline` divides by the certify kernel's
    own time (CUDA events around each launch and its FP64 pass, summed over
    the launches); `e2e` by the time of the whole insert calls (certify, scan,
    scatter, the count read back to the host)."""
    mhz = (clocks or {}).get("sm_max_mhz") or 2070
    alu_peak = sms * 128 * 2 * mhz * 1e6 / 1e12
    alu_kind = f"derived: {sms} SMs x 128 FP32 lanes x 2 x {mhz} MHz"
    flops = 2.0 * w.N * w.C * w.d
    nbytes = float(w.N) * (8 * w.d + 16)
    e2e = flops / (insert_ms * 1e-3) / 1e12
    out = {"rows": w.N, "accepted": n_acc, "ms": insert_ms, "rows_per_s": w.N / (insert_ms * 1e-3),
           "batch": w.insert_batch,
           "e2e": {"achieved": e2e, "unit": "TFLOP/s", "frac_alu": e2e / alu_peak}}
    if kernel and kernel[2] > 0:
        name, k_ms_total, launches, pairs, full_rows, fp64_rows = kernel
        out["rows_fp64_pass"] = fp64_rows
        secs = k_ms_total * 1e-3
        achieved = flops / secs / 1e12
        out["kernel"] = name
        out["kernel_ms"] = k_ms_total / launches
        out["kernel_launches"] = launches
        if name == "k_certify_tc" and tf32_peak and hbm_peak:
            gbs = nbytes / secs / 1e9
            out["roofline"] = {"bound": "hbm", "achieved": gbs, "peak": hbm_peak, "unit": "GB/s",
                               "frac": gbs / hbm_peak, "algorithmic_bytes_per_row": 8 * w.d + 16,
                               "peak_kind": "measured copy bandwidth",
                               "tensor_equiv": {"achieved": achieved, "peak": tf32_peak, "unit": "TFLOP/s",
                                                "frac": achieved / tf32_peak,
                                                "peak_kind": "measured bf16 burst x nominal tf32/bf16 ratio"},
                               "alu_equiv": {"peak": alu_peak, "frac": achieved / alu_peak, "peak_kind": alu_kind},
                               "refined_pairs_per_row": pairs / w.N, "rows_refined_over_all_classes": full_rows}
        else:
            out["roofline"] = {"bound": "alu", "achieved": achieved, "peak": alu_peak, "unit": "TFLOP/s",
                               "frac": achieved / alu_peak, "peak_kind": alu_kind}
    else:
        out["roofline"] = {"bound": "alu", "achieved": e2e, "peak": alu_peak, "unit": "TFLOP/s",
                           "frac": e2e / alu_peak, "peak_kind": alu_kind}
    return out


# ---------------------------------------------------------------- reference arm (the oracle)
def run_reference(args, dist: Dist):
    """The FP64 CPU oracle, as it stands, timed on the host cores on the same
    workload: each step probes a bounded sample of queries (one per core)
    against the whole cache."""
    import oracle
    w = workload_of(args)
    W, b, rows, Q = workload_data(w)
    sigma = oracle.sigma_max(W)
    cache = oracle.build_cache(W, b, sigma, rows)
    N = len(cache["keys"])
    n = max(1, oracle.threads())
    for i in range(args.warmup):
        s = (i * n) % max(1, len(Q) - n)
        oracle.probe(cache["keys"], cache["radius"], cache["label"], Q[s:s + n])
    t0 = time.perf_counter()
    for i in range(args.steps):
        s = ((args.warmup + i) * n) % max(1, len(Q) - n)
        oracle.probe(cache["keys"], cache["radius"], cache["label"], Q[s:s + n])
    t = time.perf_counter() - t0
    value = args.steps * n / t
    sample = f"{n} queries per step of the '{w.name}' workload against the full {N}-entry cache (FP64 brute force)"
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "queries/s", "n_gpus": dist.world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": t / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "N": N, "d": w.d, "C": w.C, "batch": w.batch, "radius": "conservative"},
        "pairs_per_s": value * N,
        "cpu_baseline": {"value": value, "unit": "queries/s", "cores": oracle.threads(), "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    args = parse()
    dist = Dist()
    try:
        if args.impl == "reference":
            if dist.rank != 0:
                return
            line = run_reference(args, dist)
        elif dist.world > 1:
            if dist.rank == 0:
                print(json.dumps({"metric": METRIC, "n_gpus": dist.world, "error": SINGLE_GPU_ONLY}), flush=True)
            print(f"bench.py: {SINGLE_GPU_ONLY}; run it with --gpus 1 and no torchrun", file=sys.stderr)
            sys.exit(2)
        else:
            line = run_ours(args, dist)
        if dist.rank == 0:
            print(json.dumps(line), flush=True)
    finally:
        if args.impl != "reference":
            dist.close()


if __name__ == "__main__":
    main()
