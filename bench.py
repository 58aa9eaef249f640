"""Benchmark of the structure-aware banded LU dispatch on GB300.

One step = one dispatch_lu call (detect the bandwidths of the dense matrix,
decide, convert to band storage, factor the band) on the synthetic
n = 4096, kl = ku = 16 fp64 matrix (uniform[-1,1] band, no diagonal boost, so
partial pivoting swaps rows), inputs resident in HBM, L2 flushed between steps.

Prints ONE JSON line.  value = GFLOP/s of the whole job (banded-LU flops counted
from the pivots the kernels chose, summed over ranks, divided by the max-over-
ranks time).  N > 1 runs independent replicas (the single-matrix path has no
data-parallel split), one per GPU.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
  python bench.py --workload NAME [--steps K]     per-stage report of a named workload
  python bench.py --custom N KL KU [BATCH]        the same report for a synthetic shape
  python bench.py --sweep                         the paper's experiments A-C on this GPU
"""
from __future__ import annotations

import argparse
import atexit
import hashlib
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

METRIC = "dispatch_lu time & GFLOP/s per matrix; detection HBM GB/s vs peak; speedup over dense"
WORKLOAD = "n4096_kl16_ku16"
FP64_PEAK_GFLOPS = 1250.0  # nominal dense FP64 of one GB300 (152 SMs x 2 DFMA/clk x 2 flop x ~2.07 GHz)
FALLBACK_HBM_GBS = 6800.0


# Sources of each kernel: a DRAM-traffic figure taken by ncu is valid only while
# their hash is the one recorded beside it under profiles/.
KERNEL_SOURCES = {
    "k_gbtrf_window": ["gbtrf.cu", "common.cuh", "rcp.cuh", "sync.cuh", "regwin.cuh"],
    "k_detect_vec": ["detect.cu", "common.cuh"],
    "k_dense_to_band_tiled": ["convert.cu", "common.cuh"],
}


def kernel_source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2608_22099_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from the
    committed ncu summary of the kernel, or None when there is none or the kernel's
    sources changed since it was captured."""
    pdir = os.path.join(ROOT, "profiles")
    if not os.path.isdir(pdir):
        return None
    want = kernel_source_hash(kernel)
    for fn in sorted(os.listdir(pdir)):
        if not fn.startswith(kernel + "_") or not fn.endswith(".md"):
            continue
        fields = {}
        with open(os.path.join(pdir, fn)) as f:
            for line in f:
                if line.startswith("traffic_bytes_per_launch:") or line.startswith("source_sha256:"):
                    k, v = line.split(":", 1)
                    fields[k.strip()] = v.strip()
        if fields.get("source_sha256") == want and "traffic_bytes_per_launch" in fields:
            return float(fields["traffic_bytes_per_launch"])
    return None


class L2Flush:
    """Cold L2 before a timed call: a 512 MiB write (larger than the 126 MiB L2), then a
    256 MiB read of another buffer, which writes the flush's dirty lines back to HBM before the
    call instead of during it.  Both run on the stream outside the timed events."""

    def __init__(self, torch, dev):
        self.w = torch.empty(512 * 1024 * 1024 // 4, dtype=torch.int32, device=dev)
        self.r = torch.zeros(256 * 1024 * 1024 // 4, dtype=torch.int32, device=dev)

    def __call__(self, k: int = 0):
        self.w.fill_(k)
        self.r.max()


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured (MEASURED_PEAKS.json, copy bandwidth)"
    return FALLBACK_HBM_GBS, "fallback 6.8 TB/s (no MEASURED_PEAKS.json)"


def band_flops(ipiv: np.ndarray, diag: np.ndarray, n: int, kl: int, ku: int) -> int:
    """sum_j [1 + km + 2*km*(ju_j - j)] over columns with a nonzero pivot, where
    ju_j is the running reach of U: max over k <= j of min(k + ku + p_k, n-1)."""
    j = np.arange(n, dtype=np.int64)
    p = ipiv.astype(np.int64) - 1 - j
    nzp = diag != 0.0
    reach = np.where(nzp, np.minimum(j + ku + p, n - 1), 0)
    ju = np.maximum.accumulate(reach)
    km = np.minimum(kl, n - 1 - j)
    per = 1 + km + 2 * km * (ju - j)
    return int(np.sum(np.where(nzp, per, 0)))


class ClockSampler:
    """nvidia-smi clocks/throttle reasons sampled every 100 ms in the background."""

    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.tmp = tempfile.NamedTemporaryFile(prefix="clocks_", suffix=".csv", delete=False)
        self.tmp.close()

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "100", "-i", str(self.index)],
                                         stdout=open(self.tmp.name, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float):
        rows = []
        try:
            with open(self.tmp.name) as f:
                for line in f:
                    parts = [x.strip() for x in line.split(",")]
                    if len(parts) < 10:
                        continue
                    try:
                        ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                        rows.append((ts, float(parts[2]), float(parts[3]), parts[6:10]))
                    except ValueError:
                        continue
        finally:
            os.unlink(self.tmp.name)
        inside = [r for r in rows if t0 - 1.0 <= r[0] <= t1 + 1.0] or rows
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in inside for k in range(4) if r[3][k].lower() == "active"})
        return {"sm_mhz": statistics.median(r[1] for r in inside), "sm_max_mhz": max(r[2] for r in inside),
                "reasons": reasons, "samples": len(inside)}


def dense_lu_ms(torch, A, stream, reps: int = 3):
    """Median time of the generic dense LU (the comparison F(N) of Sec. III-A, cuSOLVER getrf via
    torch) on a copy of A, or None when torch's linear-algebra library is unavailable."""
    times = []
    try:
        # the first call of the library initialises it: keep that out of the timing
        torch.linalg.lu_factor(torch.eye(64, dtype=A.dtype, device=A.device))
        torch.cuda.synchronize()
        for _ in range(reps):
            Ac = A.clone()
            torch.cuda.synchronize()
            a0 = torch.cuda.Event(enable_timing=True)
            a1 = torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            torch.linalg.lu_factor(Ac)
            a1.record(stream)
            torch.cuda.synchronize()
            times.append(a0.elapsed_time(a1))
            del Ac
    except RuntimeError:
        return None
    return statistics.median(times)


def cpu_oracle_dispatch(A_np: np.ndarray, ldab: int, budget_s: float, max_steps: int):
    """Time the CPU oracle's dispatch (detect + decide + convert + banded LU) on the
    whole matrix, repeated while the time budget lasts."""
    import oracle
    oracle.build()
    times, res = [], None
    t_start = time.perf_counter()
    while len(times) < max_steps:
        t0 = time.perf_counter()
        res = oracle.dispatch_lu(A_np, ldab)
        times.append(time.perf_counter() - t0)
        if time.perf_counter() - t_start > budget_s:
            break
    return times, res


def run_reference(args):
    """The oracle, as it stands, on this host's cores: one step = one dispatch of the workload."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2608_22099_gb300.workloads import WORKLOADS, make_workload
    w = WORKLOADS[WORKLOAD]
    A = make_workload(w).numpy()
    ldab = w.ldab
    # warm-up steps, then timed steps, all capped so the run ends within a few minutes
    _, res0 = cpu_oracle_dispatch(A, ldab, budget_s=30.0, max_steps=max(1, args.warmup))
    times, res = cpu_oracle_dispatch(A, ldab, budget_s=120.0, max_steps=args.steps)
    flops = band_flops(res["ipiv"], res["AB"][:, w.kl + w.ku], w.n, w.kl, w.ku)
    t = statistics.mean(times)
    value = flops / t / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": args.gpus,
        "steps": len(times), "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "n": w.n, "kl": w.kl, "ku": w.ku, "ldab": ldab},
        "cpu_baseline": {"value": value, "unit": "GFLOP/s", "cores": 1, "kind": "oracle",
                         "sample": f"{len(times)} of {args.steps} requested full dispatches of the n={w.n} matrix "
                                   f"(single-threaded C oracle; time-capped)"},
        "e2e": {"value": value, "unit": "GFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2608_22099_gb300 import bandlu, multirank
    from paper_2608_22099_gb300.workloads import WORKLOADS, make_workload

    rank, world, local = multirank.rank_info()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    def barrier():
        if world > 1:
            dist.barrier()

    w = WORKLOADS[WORKLOAD]
    n, kl, ku, ldab = w.n, w.kl, w.ku, w.ldab
    bandlu.load()
    A = make_workload(w, device=dev)
    AB = torch.zeros((n, ldab), dtype=torch.float64, device=dev)
    ipiv = torch.zeros(n, dtype=torch.int32, device=dev)
    info = torch.zeros(1, dtype=torch.int32, device=dev)
    flush = L2Flush(torch, dev)
    stream = torch.cuda.current_stream()

    def step():
        rc, gkl, gku = bandlu.dispatch_lu(A, n, n, AB, ldab, ipiv, info, stream)
        if rc != 0 or (gkl, gku) != (kl, ku):
            raise RuntimeError(f"dispatch_lu returned {rc} ({gkl}, {gku})")

    for _ in range(max(args.warmup, 3)):
        flush(1)
        step()
    torch.cuda.synchronize()
    if int(info.item()) != 0:
        raise RuntimeError("unexpected zero pivot")
    flops = band_flops(ipiv.cpu().numpy(), AB[:, kl + ku].cpu().numpy(), n, kl, ku)

    sampler = ClockSampler(local)
    if rank == 0:
        sampler.start()
        atexit.register(sampler.stop)  # never leave the sampler running if the bench fails
        time.sleep(0.3)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    for k in range(args.steps):
        flush(k)                       # L2 flush between steps, outside the timed events
        starts[k].record(stream)
        step()
        ends[k].record(stream)
    torch.cuda.synchronize()
    barrier()
    t_wall1 = time.time()
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    # replicas: every rank factors its own matrix; the job's time is the slowest rank's
    ms_per_step = multirank.max_over_ranks(sum(step_ms), device=dev) / args.steps
    value = multirank.job_throughput(multirank.sum_over_ranks(flops, device=dev), ms_per_step * 1e-3) / 1e9

    # the same step with the dispatch decision on the device (dispatch_lu_async: no host round trip)
    sc = torch.zeros(4, dtype=torch.int32, device=dev)

    def step_async():
        bandlu.check(bandlu.dispatch_lu_async(A, n, n, AB, ldab, ipiv, sc[0:1], sc[1:2], sc[2:3], sc[3:4], stream),
                     "dispatch_lu_async")
    for _ in range(3):
        step_async()
    areps = min(args.steps, 50)
    aev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(areps)]
    for r in range(areps):
        flush(r)
        aev[r][0].record(stream)
        step_async()
        aev[r][1].record(stream)
    torch.cuda.synchronize()
    async_ms = statistics.mean(a.elapsed_time(b) for a, b in aev)
    if tuple(int(v) for v in sc[:3].cpu()) != (kl, ku, 0):
        raise RuntimeError("dispatch_lu_async disagrees with dispatch_lu")

    # stage breakdown through the same C ABI, CUDA events on the launching stream
    klku = torch.zeros(2, dtype=torch.int32, device=dev)
    AB2 = torch.zeros_like(AB)
    ipiv2 = torch.zeros_like(ipiv)
    info2 = torch.zeros_like(info)
    reps = min(args.steps, 50)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(reps)]
    for r in range(reps):
        flush(r)
        e = ev[r]
        e[0].record(stream)
        bandlu.check(bandlu.detect_bandwidth(A, n, n, klku, klku.data_ptr() + 4, stream), "detect_bandwidth")
        e[1].record(stream)
        bandlu.check(bandlu.dense_to_band(A, n, n, kl, ku, AB2, ldab, stream), "dense_to_band")
        e[2].record(stream)
        bandlu.check(bandlu.gbtrf(n, kl, ku, AB2, ldab, ipiv2, info2, stream), "gbtrf")
        e[3].record(stream)
    torch.cuda.synchronize()
    t_detect = statistics.mean(e[0].elapsed_time(e[1]) for e in ev) * 1e-3
    t_convert = statistics.mean(e[1].elapsed_time(e[2]) for e in ev) * 1e-3
    t_gbtrf = statistics.mean(e[2].elapsed_time(e[3]) for e in ev) * 1e-3
    if not (torch.equal(AB2, AB) and torch.equal(ipiv2, ipiv)):
        raise RuntimeError("stage-by-stage results differ from dispatch_lu")

    hbm_peak, hbm_src = load_peaks()
    detect_bytes = 8.0 * n * n
    nnz_band = n * (kl + ku + 1) - kl * (kl + 1) // 2 - ku * (ku + 1) // 2
    convert_bytes = 8.0 * nnz_band + 8.0 * ldab * n
    stages = {
        "detect_us": t_detect * 1e6, "detect_gbs": detect_bytes / t_detect / 1e9,
        "detect_frac_hbm": detect_bytes / t_detect / 1e9 / hbm_peak,
        "convert_us": t_convert * 1e6, "convert_gbs": convert_bytes / t_convert / 1e9,
        "gbtrf_us": t_gbtrf * 1e6, "gbtrf_gflops": flops / t_gbtrf / 1e9,
        "gbtrf_ns_per_column": t_gbtrf / n * 1e9,
    }
    kernels = {"detect": t_detect, "convert": t_convert, "gbtrf": t_gbtrf}
    dominant = max(kernels, key=kernels.get)
    if dominant == "gbtrf":
        achieved = flops / t_gbtrf / 1e9
        roofline = {"bound": "alu", "achieved": achieved / 1e3, "peak": FP64_PEAK_GFLOPS / 1e3, "unit": "TFLOP/s",
                    "frac": achieved / FP64_PEAK_GFLOPS, "traffic": profiled_traffic("k_gbtrf_window"),
                    "kernel": "k_gbtrf_window",
                    "peak_source": "nominal FP64 (152 SMs x 2 DFMA/clk x 2 flop x 2.07 GHz)",
                    "frac_of_one_sm": achieved / (FP64_PEAK_GFLOPS / 152),
                    "note": "one matrix is one serial pivot chain on one SM (one CTA): latency-bound, see "
                            "ns_per_column; frac_of_one_sm is against that SM's share of the peak"}
    elif dominant == "detect":
        roofline = {"bound": "hbm", "achieved": detect_bytes / t_detect / 1e9, "peak": hbm_peak, "unit": "GB/s",
                    "frac": detect_bytes / t_detect / 1e9 / hbm_peak, "traffic": profiled_traffic("k_detect_vec"),
                    "kernel": "k_detect_vec",
                    "peak_source": hbm_src}
    else:
        roofline = {"bound": "hbm", "achieved": convert_bytes / t_convert / 1e9, "peak": hbm_peak, "unit": "GB/s",
                    "frac": convert_bytes / t_convert / 1e9 / hbm_peak,
                    "traffic": profiled_traffic("k_dense_to_band_tiled"),
                    "kernel": "k_dense_to_band_tiled", "peak_source": hbm_src}

    # end to end: pinned host input -> device, dispatch_lu, factors back to pinned host memory
    A_host = A.cpu().pin_memory()
    AB_host = torch.empty(AB.shape, dtype=AB.dtype).pin_memory()
    ipiv_host = torch.empty(ipiv.shape, dtype=ipiv.dtype).pin_memory()
    info_host = torch.empty(info.shape, dtype=info.dtype).pin_memory()
    A_e2e = torch.empty_like(A)
    e2e_reps = min(args.steps, 50)
    e2e_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(e2e_reps)]
    for r in range(e2e_reps):
        flush(r)
        e0, e1 = e2e_ev[r]
        e0.record(stream)
        A_e2e.copy_(A_host, non_blocking=True)
        rc, _, _ = bandlu.dispatch_lu(A_e2e, n, n, AB, ldab, ipiv, info, stream)
        bandlu.check(rc, "dispatch_lu")
        AB_host.copy_(AB, non_blocking=True)
        ipiv_host.copy_(ipiv, non_blocking=True)
        info_host.copy_(info, non_blocking=True)
        e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = multirank.max_over_ranks(statistics.mean(a.elapsed_time(b) for a, b in e2e_ev), device=dev)
    e2e_value = multirank.job_throughput(multirank.sum_over_ranks(flops, device=dev), e2e_ms * 1e-3) / 1e9
    h2d = A_host.numel() * 8
    d2h = AB_host.numel() * 8 + ipiv_host.numel() * 4 + info_host.numel() * 4

    # the generic algorithm F(N) of Sec. III-A on the same matrix: dense LU (cuSOLVER via torch)
    dense_t = dense_lu_ms(torch, A, stream)

    clocks = None
    if rank == 0:
        sampler.stop()
        clocks = sampler.summary(t_wall0, t_wall1)

    cpu_baseline = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        times, res = cpu_oracle_dispatch(A.cpu().numpy(), ldab, budget_s=20.0, max_steps=1000)
        cflops = band_flops(res["ipiv"], res["AB"][:, kl + ku], n, kl, ku)
        cpu_baseline = {"value": cflops / statistics.mean(times) / 1e9, "unit": "GFLOP/s", "cores": 1,
                        "kind": "oracle",
                        "sample": f"{len(times)} full dispatches of the n={n} matrix, single-threaded C oracle"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "n": n, "kl": kl, "ku": ku, "ldab": ldab, "dist": "uniform[-1,1]",
                       "l2": "flushed between steps (512 MiB write, then a 256 MiB read that writes its dirty lines back)",
                       "parallelism": "replicas" if world > 1 else "single"},
            "dispatch_ms": ms_per_step, "dispatch_async_ms": async_ms, "dense_lu_ms": dense_t,
            "speedup_over_dense": (dense_t / ms_per_step) if dense_t else None,
            "flops_per_step": flops, "stages": stages, "roofline": roofline,
            "cpu_baseline": cpu_baseline,
            "e2e": {"value": e2e_value, "unit": "GFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": e2e_ms},
            "gpu_launches": 3 * args.steps,
            "clocks": clocks,
            "wall_s_timed": t_wall1 - t_wall0,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_workload_report(args):
    """One JSON line per call for any workload (per-stage CUDA-event timings), used for the
    per-workload table; the contract line is the default workload's."""
    import torch

    from paper_2608_22099_gb300 import bandlu
    from paper_2608_22099_gb300.workloads import WORKLOADS, Workload, make_workload

    if args.custom:
        cn, ckl, cku = args.custom[:3]
        cb = args.custom[3] if len(args.custom) > 3 else 0
        w = Workload(f"custom_n{cn}_kl{ckl}_ku{cku}" + (f"_batch{cb}" if cb else ""), cn, ckl, cku, "uniform",
                     4.0 if cb else 0.0, 7, batch=cb)
    else:
        w = WORKLOADS[args.workload]
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    bandlu.load()
    A = make_workload(w, device=dev)
    n, kl, ku, ldab = w.n, w.kl, w.ku, w.ldab
    flush = L2Flush(torch, dev)
    stream = torch.cuda.current_stream()
    hbm_peak, hbm_src = load_peaks()
    out = {"workload": w.name, "n": n, "kl": kl, "ku": ku, "batch": w.batch}
    reps = max(1, args.steps)

    def timed(fn, reps):
        ts = []
        for r in range(reps):
            flush(r)
            a = torch.cuda.Event(enable_timing=True); b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b) * 1e-3)
        return statistics.median(ts)

    if w.batch:
        B = w.batch
        AB = torch.zeros((B, n, ldab), dtype=torch.float64, device=dev)
        ipiv = torch.zeros((B, n), dtype=torch.int32, device=dev)
        kls, kus, infos, sts = (torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(4))

        def step():
            bandlu.check(bandlu.dispatch_lu_batched(A, n, n, n * n, B, AB, ldab, n * ldab, ipiv, n, kls, kus,
                                                    infos, sts, stream), "dispatch_lu_batched")
        for _ in range(max(args.warmup, 3)):
            step()
        t = timed(step, reps)
        diag = AB[:, :, kl + ku].cpu().numpy()
        ip = ipiv.cpu().numpy()
        flops = sum(band_flops(ip[b], diag[b], n, kl, ku) for b in range(B))
        bytes_ = 8.0 * B * n * n
        out.update({"dispatch_batched_ms": t * 1e3, "gflops": flops / t / 1e9, "hbm_gbs": bytes_ / t / 1e9,
                    "hbm_frac": bytes_ / t / 1e9 / hbm_peak, "matrices_per_s": B / t, "flops": flops})
    else:
        AB = torch.zeros((n, ldab), dtype=torch.float64, device=dev)
        ipiv = torch.zeros(n, dtype=torch.int32, device=dev)
        info = torch.zeros(1, dtype=torch.int32, device=dev)
        klku = torch.zeros(2, dtype=torch.int32, device=dev)
        res = {}

        def disp():
            res["rc"] = bandlu.dispatch_lu(A, n, n, AB, ldab, ipiv, info, stream)

        def det():
            bandlu.check(bandlu.detect_bandwidth(A, n, n, klku, klku.data_ptr() + 4, stream), "detect")

        for _ in range(max(args.warmup, 3)):
            disp()
        t_disp = timed(disp, reps)
        t_det = timed(det, reps)
        # the same dispatch with the decision on the device (no host round trip), and that call
        # captured once in a CUDA graph and replayed; for the bands its one-CTA kernels cover
        # (wider bands take its block-wide fallback, seconds at n = 32768)
        if kl <= 27 and 2 * kl + ku + 1 <= 256:
            sc = torch.zeros(4, dtype=torch.int32, device=dev)

            def dasync(st):
                bandlu.check(bandlu.dispatch_lu_async(A, n, n, AB, ldab, ipiv, sc[0:1], sc[1:2], sc[2:3], sc[3:4],
                                                      st), "dispatch_lu_async")
            for _ in range(3):
                dasync(stream)
            t_async = timed(lambda: dasync(stream), reps)
            gs = torch.cuda.Stream()
            torch.cuda.synchronize()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=gs):
                dasync(gs)
            graph.replay()
            t_graph = timed(graph.replay, reps)
            out.update({"dispatch_async_ms": t_async * 1e3, "dispatch_graph_ms": t_graph * 1e3})
        rc, dkl, dku = res["rc"]
        out.update({"status": rc, "detected_kl": dkl, "detected_ku": dku, "dispatch_ms": t_disp * 1e3,
                    "detect_us": t_det * 1e6, "detect_gbs": 8.0 * n * n / t_det / 1e9,
                    "detect_frac_hbm": 8.0 * n * n / t_det / 1e9 / hbm_peak})
        if rc == 0:
            def conv():
                bandlu.check(bandlu.dense_to_band(A, n, n, kl, ku, AB, ldab, stream), "convert")

            AB2 = torch.zeros_like(AB)

            def fac():
                AB2.copy_(AB)
                bandlu.check(bandlu.gbtrf(n, kl, ku, AB2, ldab, ipiv, info, stream), "gbtrf")
            conv()
            t_conv = timed(conv, reps)
            t_fac = timed(fac, max(1, min(reps, 5))) if n > 20000 else timed(fac, reps)
            flops = band_flops(ipiv.cpu().numpy(), AB2[:, kl + ku].cpu().numpy(), n, kl, ku)
            # the solve with the factors, one right-hand side (forward and back substitution)
            xb = torch.empty(n, dtype=torch.float64, device=dev)
            b0 = torch.linspace(-1.0, 1.0, n, dtype=torch.float64, device=dev)

            def sol():
                xb.copy_(b0)
                bandlu.check(bandlu.gbtrs(n, kl, ku, 1, AB2, ldab, ipiv, xb, n, stream), "gbtrs")
            t_sol = timed(sol, max(1, min(reps, 5)))
            if n <= 20000:
                # the lower-triangular branch of the backslash dispatch on the matrix's own lower
                # triangle (bandwidth kl, read in place from the dense matrix)
                Lm = torch.tril(A)
                info2 = torch.zeros(1, dtype=torch.int32, device=dev)

                def trs():
                    xb.copy_(b0)
                    bandlu.check(bandlu.trsv_band(1, n, kl, Lm, n, xb, n, 1, info2, stream), "trsv_band")
                trs()
                out["trsv_lower_1rhs_ms"] = timed(trs, max(1, min(reps, 5))) * 1e3
                del Lm
            out.update({"convert_us": t_conv * 1e6, "gbtrf_ms": t_fac * 1e3, "gbtrf_gflops": flops / t_fac / 1e9,
                        "gbtrf_ns_per_column": t_fac / n * 1e9, "flops": flops,
                        "gflops_dispatch": flops / t_disp / 1e9, "gbtrs_1rhs_ms": t_sol * 1e3,
                        "gbtrs_ns_per_row": t_sol / n * 1e9})
        if n <= 20000:
            d_ms = dense_lu_ms(torch, A, stream)
            out["dense_lu_ms"] = d_ms
            if d_ms:
                t_dense = d_ms * 1e-3
                out["speedup_over_dense" if rc == 0 else "slowdown_vs_dense"] = (
                    t_dense / t_disp if rc == 0 else (t_det + t_dense) / t_dense)
        else:
            # dense LU of the full matrix would take tens of seconds: time it at n/2 on the
            # same GPU and scale by the 2n^3/3 operation count (labelled an estimate)
            h = n // 2
            Ah = A[:h, :h].contiguous()
            d_half = dense_lu_ms(torch, Ah, stream, reps=1)
            del Ah
            if d_half:
                est = d_half * (n / h) ** 3
                out["dense_lu_ms_estimate"] = est
                out["dense_lu_estimate_from"] = f"measured {d_half:.1f} ms at n={h}, scaled by (n/{h})^3"
                if rc == 0:
                    out["speedup_over_dense_estimate"] = est * 1e-3 / t_disp
    out["hbm_peak_source"] = hbm_src
    print(json.dumps(out), flush=True)


def run_sweep(args):
    """The paper's experiments on this GPU (Sec. IV): A, the speedup of dispatch_lu over the
    dense LU for N = 2000..8000 with P + Q = 1% and 10% of N (Eq. su-con; Sec. III-C predicts
    linear growth in N); B, the slowdown (I + F) / F on the same shapes with one stray entry
    that makes them non-banded (Eq. sd-con; predicted constant); C, the N = 10^4, 100 + 100
    diagonals case of Figs. 5-6, with the memory ratio.  One JSON line per point."""
    import torch

    from paper_2608_22099_gb300 import bandlu
    from paper_2608_22099_gb300.workloads import make_dense

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    bandlu.load()
    flush = L2Flush(torch, dev)
    stream = torch.cuda.current_stream()
    reps = max(1, min(args.steps, 5))

    def timed(fn):
        ts = []
        for r in range(reps):
            flush(r)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b) * 1e-3)
        return statistics.median(ts)

    points = [("A", n, f) for f in (0.01, 0.10) for n in range(2000, 8001, 1000)] + [("C", 10000, 0.02)]
    for exp, n, f in points:
        kl = ku = max(1, int(round(f * n / 2)))
        ldab = 2 * kl + ku + 1
        A = make_dense(n, kl, ku, dist="uniform", seed=n + kl, device=dev)
        AB = torch.zeros((n, ldab), dtype=torch.float64, device=dev)
        ipiv = torch.zeros(n, dtype=torch.int32, device=dev)
        info = torch.zeros(1, dtype=torch.int32, device=dev)
        res = {}

        def disp():
            res["rc"] = bandlu.dispatch_lu(A, n, n, AB, ldab, ipiv, info, stream)

        disp()
        torch.cuda.synchronize()
        t_disp = timed(disp)
        t_dense = dense_lu_ms(torch, A, stream)
        line = {"sweep": exp, "n": n, "kl": kl, "ku": ku, "p_plus_q_frac": (kl + ku) / n,
                "status": res["rc"][0], "dispatch_ms": t_disp * 1e3, "dense_lu_ms": t_dense,
                "speedup_over_dense": (t_dense * 1e-3 / t_disp) if t_dense else None,
                "memory_ratio_dense_over_band": (8.0 * n * n + 8 * n) / (3 * 8.0 * ldab * n + 8 * n)}
        # experiment B: the same shape with one stray entry -> not banded, detection + dense LU
        A[n - 1, 0] = 1e-3
        klku = torch.zeros(2, dtype=torch.int32, device=dev)

        def det():
            bandlu.check(bandlu.detect_bandwidth(A, n, n, klku, klku.data_ptr() + 4, stream), "detect")

        rc_c, _, _ = bandlu.dispatch_lu(A, n, n, AB, ldab, ipiv, info, stream)
        t_det = timed(det)
        if t_dense:
            line.update({"control_status": rc_c, "detect_us": t_det * 1e6,
                         "slowdown_control": (t_det + t_dense * 1e-3) / (t_dense * 1e-3)})
        print(json.dumps(line), flush=True)
        del A, AB


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="workload name (default: the n=4096, kl=ku=16 matrix); others for per-workload reports")
    ap.add_argument("--sweep", action="store_true", help="the paper's experiments A-C (speedup / slowdown in N)")
    ap.add_argument("--custom", type=int, nargs="+", metavar="N KL KU [BATCH]",
                    help="per-stage report of a synthetic uniform[-1,1] band of this shape (batched if BATCH > 0)")
    args = ap.parse_args()
    if args.custom is not None and len(args.custom) not in (3, 4):
        ap.error("--custom takes N KL KU [BATCH]")
    if args.impl == "reference":
        run_reference(args)
    elif args.sweep:
        run_sweep(args)
    elif args.custom or args.workload != WORKLOAD:
        run_workload_report(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
