"""Benchmark of the structure-aware banded LU dispatch on GB300.

One step = one dispatch_lu call (detect the bandwidths of the dense matrix,
decide, convert to band storage, factor the band) on the synthetic
n = 32768, kl = ku = 256 fp64 matrix stored dense (8 GiB; uniform[-1,1] band,
no diagonal boost, so partial pivoting swaps rows), inputs resident in HBM, L2
flushed between steps.  The wide band runs the multi-CTA blocked factorisation.

Prints ONE JSON line.  value = GFLOP/s of the whole job (banded-LU flops counted
from the pivots the kernels chose, summed over ranks, divided by the max-over-
ranks time).  N > 1 runs independent replicas (the single-matrix path has no
data-parallel split), one per GPU.  Beside the contract numbers the line carries
one key per other workload shape (stage times, GFLOP/s, detection's fraction of
HBM, the factorisation's fractions of the measured FP64 and HBM rooflines,
speedup over the dense LU), the FP64 peak measured in the same run, and the CPU
oracle's times on this host (single-threaded and with OpenMP).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
  python bench.py --peaks                         FP64 (FMA, DMMA) and read-bandwidth microbenchmarks
  python bench.py --workload NAME [--steps K]     per-stage report of a named workload
  python bench.py --custom N KL KU [BATCH]        the same report for a synthetic shape
  python bench.py --sweep                         the paper's experiments A-C on this GPU
  python bench.py --trace [--custom N KL KU]      timeline of the wide-band chain kernel (traced build)
"""
from __future__ import annotations

import argparse
import atexit
import hashlib
import json
import os
import platform
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "dispatch_lu time & GFLOP/s per matrix; detection HBM GB/s vs peak; speedup over dense"
WORKLOAD = "n32768_kl256_ku256"
# the other workload shapes, reported beside the contract line (in the order they are listed)
OTHER_WORKLOADS = ["n512_kl3_ku3", "n4096_kl16_ku16", "n16384_kl8_ku64", "n16384_kl8_ku64_stray",
                   "batch4096_n256_kl2_ku2"]
# the CPU oracle's bounded sample: the leading principal block of the matrix (same band)
REF_SAMPLE_N = 8192
CPU_SAMPLE_N = 8192
FP64_NOMINAL_GFLOPS = 1250.0  # 152 SMs x 2 DFMA/clk x 2 flop x ~2.07 GHz (context only)
FALLBACK_HBM_GBS = 6800.0


# Sources of each kernel: a DRAM-traffic figure taken by ncu is valid only while
# their hash is the one recorded beside it under profiles/.
KERNEL_SOURCES = {
    "k_gbtrf_wide": ["gbtrf_wide.cu", "gbtrf_wide_stream.cuh", "common.cuh", "rcp.cuh", "sync.cuh"],
    "k_gbtrf_wide_chain": ["gbtrf_wide.cu", "gbtrf_wide_stream.cuh", "common.cuh", "rcp.cuh", "sync.cuh"],
    "k_gbtrf_window": ["gbtrf.cu", "common.cuh", "rcp.cuh", "sync.cuh", "regwin.cuh"],
    "k_gbtrf_regwin": ["gbtrf.cu", "common.cuh", "rcp.cuh", "sync.cuh", "regwin.cuh"],
    "k_detect_vec": ["detect.cu", "common.cuh"],
    "k_detect_flat": ["detect.cu", "common.cuh"],
    "k_dense_to_band_tiled": ["convert.cu", "common.cuh"],
    "k_batch_scan_convert": ["batched.cu", "common.cuh", "regwin.cuh", "rcp.cuh"],
}


def kernel_source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    for name in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2608_22099_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, workload: str | None = None):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from the
    committed ncu summary of the kernel (for `workload` when given), or None when there is
    none or the kernel's sources changed since it was captured."""
    pdir = os.path.join(ROOT, "profiles")
    if not os.path.isdir(pdir) or kernel not in KERNEL_SOURCES:
        return None
    want = kernel_source_hash(kernel)
    for fn in sorted(os.listdir(pdir)):
        if not fn.startswith(kernel + "_") or not fn.endswith(".md"):
            continue
        if workload is not None and workload not in fn:
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


def gbtrf_kernel(n: int, kl: int, ku: int) -> str:
    """The factorisation kernel the library's launcher picks for a band (its size rules)."""
    if (kl + 1) * (kl + ku + 1) <= 32:
        return "k_gbtrf_regwin"
    if kl <= 27:
        return "k_gbtrf_window"
    if (kl + 4 <= 288 and kl + ku >= 8 and n >= 16 and os.environ.get("BANDLU_WIDE_SINGLE") != "1"
            and os.environ.get("BANDLU_WIDE_PAIR") != "1"):
        return "k_gbtrf_wide_chain"  # where its clusters of five fit (else the pair or single-CTA kernel)
    return "k_gbtrf_wide"


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
            self.proc = None

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


def cpu_model() -> str:
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu part")):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.processor() or platform.machine()


def host_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def workload_config(w) -> dict:
    """The `config` object of both arms' lines (identical keys, so the driver can compare them)."""
    return {"workload": w.name, "n": w.n, "kl": w.kl, "ku": w.ku, "ldab": w.ldab}


def oracle_sample_dispatch(w, m: int, steps: int, budget_s: float | None = None):
    """The CPU oracle's dispatch (detect + decide + convert + banded LU), single-threaded, on
    the leading m x m principal block of workload w (same band, same values): per-call times
    and the flops of the factorisation it performed."""
    import oracle
    from paper_2608_22099_gb300.workloads import principal_block
    oracle.build()
    A = principal_block(w, m).numpy()
    times, res = [], None
    t_start = time.perf_counter()
    for _ in range(max(1, steps)):
        t0 = time.perf_counter()
        res = oracle.dispatch_lu(A, w.ldab)
        times.append(time.perf_counter() - t0)
        if budget_s is not None and time.perf_counter() - t_start > budget_s:
            break
    if res["status"] != 0:
        raise RuntimeError("the oracle declined the sample")
    flops = band_flops(res["ipiv"], res["AB"][:, w.kl + w.ku], A.shape[0], w.kl, w.ku)
    return times, flops


def run_reference(args):
    """The oracle, as it stands, on this host's cores: each step is one single-threaded
    dispatch of a bounded sample of the workload (its leading principal block)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2608_22099_gb300.workloads import WORKLOADS
    w = WORKLOADS[WORKLOAD]
    oracle_sample_dispatch(w, REF_SAMPLE_N, args.warmup)
    times, flops = oracle_sample_dispatch(w, REF_SAMPLE_N, args.steps)
    t = statistics.mean(times)
    value = flops / t / 1e9
    sample = (f"each step: one dispatch (detect, decide, convert, banded LU) of the leading "
              f"{REF_SAMPLE_N} x {REF_SAMPLE_N} principal block of the n={w.n} matrix (same kl={w.kl}, "
              f"ku={w.ku}, same values), single-threaded C oracle on {cpu_model()}")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": args.gpus,
        "steps": len(times), "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(w),
        "cpu_baseline": {"value": value, "unit": "GFLOP/s", "cores": 1, "kind": "oracle", "sample": sample,
                         "host_threads": host_threads(), "cpu_model": cpu_model()},
        "e2e": {"value": value, "unit": "GFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------------------
# measured ceilings

def event_ms(torch, stream, fn, reps: int, flush=None):
    """Per-call CUDA-event times (ms) of fn() on `stream`, after one untimed call."""
    fn()
    out = []
    for r in range(reps):
        if flush is not None:
            flush(r)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        torch.cuda.synchronize()
        out.append(a.elapsed_time(b))
    return out


def measure_fp64_fma(torch, dev, stream, sms: int, warps_per_sm: int = 16, chains: int = 8, iters: int = 2048):
    """GFLOP/s of the FP64 FMA microbenchmark: sms x (warps_per_sm/8) blocks of 256 threads,
    `chains` independent FMA chains per thread (best of 5 launches)."""
    from paper_2608_22099_gb300 import bandlu
    blocks = sms * max(1, warps_per_sm // 8)
    threads = 32 * min(8, warps_per_sm)
    sink = torch.empty(blocks, dtype=torch.float64, device=dev)
    flops = 2.0 * blocks * threads * chains * iters
    ts = event_ms(torch, stream, lambda: bandlu.check(
        bandlu.bandlu_peak_dfma(sink, blocks, threads, chains, iters, stream), "bandlu_peak_dfma"), 5)
    return flops / (min(ts) * 1e-3) / 1e9


def run_peaks(args):
    """One JSON line: the FP64 FMA rate by warps per SM and chains per thread, the FP64 MMA
    (mma.sync) rate of both shapes, and a read-only HBM stream."""
    import torch

    from paper_2608_22099_gb300 import bandlu
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    bandlu.load()
    stream = torch.cuda.current_stream()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    out = {"peaks": True, "gpu": torch.cuda.get_device_name(dev), "sms": sms}
    fma = {}
    for wps in (1, 2, 4, 8, 16, 32):
        for ch in (1, 4, 8):
            threads = 32 * min(wps, 8)
            blocks = sms * max(1, wps // 8)
            sink = torch.empty(blocks, dtype=torch.float64, device=dev)
            iters = 1024
            ts = event_ms(torch, stream, lambda: bandlu.check(
                bandlu.bandlu_peak_dfma(sink, blocks, threads, ch, iters, stream), "dfma"), 5)
            g = 2.0 * blocks * threads * ch * iters / (min(ts) * 1e-3) / 1e9
            fma[f"warps{wps}_chains{ch}"] = {"gflops": g, "fma_per_clk_per_sm": None}
    out["dfma"] = fma
    mma = {}
    for shape, mnk in ((0, 256), (1, 2048)):
        for warps in (4, 8, 16):
            for ch in (1, 2, 4):
                blocks = sms
                sink = torch.empty(blocks, dtype=torch.float64, device=dev)
                iters = 512 if shape == 0 else 128
                ts = event_ms(torch, stream, lambda: bandlu.check(
                    bandlu.bandlu_peak_dmma(shape, sink, blocks, warps, ch, iters, stream), "dmma"), 5)
                g = 2.0 * mnk * blocks * warps * ch * iters / (min(ts) * 1e-3) / 1e9
                mma[f"{'m8n8k4' if shape == 0 else 'm16n8k16'}_warps{warps}_chains{ch}"] = {"gflops": g}
    out["dmma"] = mma
    nbytes = 4 << 30
    buf = torch.empty(nbytes // 8, dtype=torch.float64, device=dev).fill_(1.0)
    rd = {}
    for bps in (2, 4, 8):
        blocks = sms * bps
        sink = torch.empty(blocks, dtype=torch.int64, device=dev)
        ts = event_ms(torch, stream, lambda: bandlu.check(
            bandlu.bandlu_peak_hbm_read(buf, nbytes, sink, blocks, stream), "hbm_read"), 5)
        rd[f"blocks{blocks}"] = nbytes / (min(ts) * 1e-3) / 1e9
    out["hbm_read_gbs_4gib"] = rd
    # the same read-only stream over 128 MiB (the size of the n = 4096 dense matrix), L2 flushed
    # before each read: the ceiling a detection pass of that size can reach (ramp and tail included)
    flush = L2Flush(torch, dev)
    small = {}
    for nbytes_s in (128 << 20, 512 << 20):
        for bps in (2, 4):
            blocks = sms * bps
            sink = torch.empty(blocks, dtype=torch.int64, device=dev)
            ts = event_ms(torch, stream, lambda: bandlu.check(
                bandlu.bandlu_peak_hbm_read(buf, nbytes_s, sink, blocks, stream), "hbm_read"), 10, flush)
            small[f"{nbytes_s >> 20}MiB_blocks{blocks}"] = {"us": statistics.median(ts) * 1e3,
                                                            "gbs": nbytes_s / (statistics.median(ts) * 1e-3) / 1e9}
    out["hbm_read_cold"] = small
    # per-warp cost of the operations a column step is made of, in SM clocks, on one block of
    # 1, 3 and 4 warps (include/bandlu_peaks.h): what the latency-bound factorisations pay
    ops = ("dfma_dependent", "dfma_independent", "shfl_f64_dependent", "shfl_b32_independent",
           "smem_roundtrip", "imad_dependent", "redux_ballot_dependent", "rcp_rn_dependent")
    clk_buf = torch.zeros(1, dtype=torch.int64, device=dev)
    sink_w = torch.empty(32 * 32, dtype=torch.float64, device=dev)
    costs = {}
    for op, name in enumerate(ops):
        row = {}
        for warps in (1, 3, 4):
            iters = 256
            for _ in range(2):  # the second launch is the measured one
                bandlu.check(bandlu.bandlu_peak_warp_costs(op, clk_buf, sink_w, warps, iters, stream), "warp_costs")
            torch.cuda.synchronize()
            row[f"warps{warps}"] = round(int(clk_buf.item()) / (16 * iters), 1)
        costs[name] = row
    out["warp_costs_clk"] = costs
    # clock while the FMA kernel runs, for the per-clock rates
    sampler = ClockSampler(0)
    sampler.start()
    time.sleep(0.3)
    t0 = time.time()
    g_best = 0.0
    while time.time() - t0 < 1.5:
        g_best = max(g_best, measure_fp64_fma(torch, dev, stream, sms))
    t1 = time.time()
    sampler.stop()
    clk = sampler.summary(t0, t1)
    out["dfma_best_gflops"] = g_best
    out["clocks"] = clk
    if clk.get("sm_mhz"):
        hz = clk["sm_mhz"] * 1e6
        for v in fma.values():
            v["fma_per_clk_per_sm"] = v["gflops"] * 1e9 / 2 / hz / sms
        out["dfma_best_fma_per_clk_per_sm"] = g_best * 1e9 / 2 / hz / sms
        for v in mma.values():
            v["fma_per_clk_per_sm"] = v["gflops"] * 1e9 / 2 / hz / sms
    print(json.dumps(out), flush=True)


# ---------------------------------------------------------------------------------------
# the per-workload measurements beside the contract line

def plain_read_s(torch, bandlu, A, dev, stream, flush, reps: int):
    """Median time of one read-only pass (bandlu_peak_hbm_read) over the same dense matrix,
    L2 flushed before each: the ceiling a detection pass over those bytes can reach."""
    nbytes = A.numel() * 8
    if nbytes < 16 or nbytes % 16 or A.data_ptr() % 16:
        return None
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    sink = torch.empty(4 * sms, dtype=torch.int64, device=dev)
    ts = event_ms(torch, stream, lambda: bandlu.check(
        bandlu.bandlu_peak_hbm_read(A, nbytes, sink, 4 * sms, stream), "hbm_read"), reps, flush)
    return statistics.median(ts) * 1e-3


def measure_single(torch, bandlu, w, dev, stream, flush, reps: int, fp64_peak: float, hbm_peak: float,
                   dense_ms=None):
    """Stage times of one workload through the C ABI (median of reps, L2 flushed before each
    call), GFLOP/s, detection's HBM fraction and the factorisation's roofline fractions."""
    from paper_2608_22099_gb300.workloads import make_workload
    n, kl, ku, ldab = w.n, w.kl, w.ku, w.ldab
    A = make_workload(w, device=dev)
    AB = torch.zeros((n, ldab), dtype=torch.float64, device=dev)
    ipiv = torch.zeros(n, dtype=torch.int32, device=dev)
    info = torch.zeros(1, dtype=torch.int32, device=dev)
    klku = torch.zeros(2, dtype=torch.int32, device=dev)
    res = {}

    def disp():
        res["rc"] = bandlu.dispatch_lu(A, n, n, AB, ldab, ipiv, info, stream)

    def det():
        bandlu.check(bandlu.detect_bandwidth(A, n, n, klku, klku.data_ptr() + 4, stream), "detect")

    t_disp = statistics.median(event_ms(torch, stream, disp, reps, flush)) * 1e-3
    t_det = statistics.median(event_ms(torch, stream, det, reps, flush)) * 1e-3
    rc, dkl, dku = res["rc"]
    # the same dispatch with the decision on the device (no host round trip)
    sc = torch.zeros(4, dtype=torch.int32, device=dev)
    ABa = torch.zeros_like(AB)
    ipa = torch.zeros_like(ipiv)

    def dasync():
        bandlu.check(bandlu.dispatch_lu_async(A, n, n, ABa, ldab, ipa, sc[0:1], sc[1:2], sc[2:3], sc[3:4], stream),
                     "dispatch_lu_async")
    t_async = statistics.median(event_ms(torch, stream, dasync, reps, flush)) * 1e-3
    if tuple(int(v) for v in sc[:3].cpu()) != (dkl, dku, rc) or (rc == 0 and not torch.equal(ABa, AB)):
        raise RuntimeError(f"{w.name}: dispatch_lu_async disagrees with dispatch_lu")
    del ABa, ipa
    det_bytes = 8.0 * n * n
    t_read = plain_read_s(torch, bandlu, A, dev, stream, flush, reps)
    out = {"status": rc, "detected_kl": dkl, "detected_ku": dku, "dispatch_ms": t_disp * 1e3,
           "dispatch_async_ms": t_async * 1e3, "plain_read_us": t_read * 1e6 if t_read else None,
           "detect_frac_of_plain_read": (t_read / t_det) if t_read else None,
           "detect_us": t_det * 1e6, "detect_gbs": det_bytes / t_det / 1e9,
           "detect_frac_hbm": det_bytes / t_det / 1e9 / hbm_peak}
    if rc == 0:
        AB2 = torch.zeros_like(AB)

        def conv():
            bandlu.check(bandlu.dense_to_band(A, n, n, kl, ku, AB2, ldab, stream), "convert")

        def fac():
            bandlu.check(bandlu.gbtrf(n, kl, ku, AB2, ldab, ipiv, info, stream), "gbtrf")
        t_conv = statistics.median(event_ms(torch, stream, conv, reps, flush)) * 1e-3
        tf = []
        for r in range(reps):   # the factorisation works in place: convert afresh before each call
            conv()
            flush(r)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fac()
            b.record(stream)
            torch.cuda.synchronize()
            tf.append(a.elapsed_time(b) * 1e-3)
        t_fac = statistics.median(tf)
        if not (torch.equal(AB2, AB) and int(info.item()) == 0):
            raise RuntimeError(f"{w.name}: stage-by-stage results differ from dispatch_lu")
        flops = band_flops(ipiv.cpu().numpy(), AB[:, kl + ku].cpu().numpy(), n, kl, ku)
        nnz = n * (kl + ku + 1) - kl * (kl + 1) // 2 - ku * (ku + 1) // 2
        conv_bytes = 8.0 * nnz + 8.0 * ldab * n
        band_bytes = 2 * 8.0 * ldab * n
        g = flops / t_fac / 1e9
        out.update({"convert_us": t_conv * 1e6, "convert_gbs": conv_bytes / t_conv / 1e9,
                    "gbtrf_kernel": gbtrf_kernel(n, kl, ku), "gbtrf_ms": t_fac * 1e3, "gbtrf_gflops": g,
                    "gbtrf_ns_per_column": t_fac / n * 1e9, "gbtrf_frac_fp64": g / fp64_peak,
                    "gbtrf_frac_hbm": band_bytes / t_fac / 1e9 / hbm_peak, "flops": flops,
                    "gflops_dispatch": flops / t_disp / 1e9})
    if dense_ms is None and n <= 16384:
        dense_ms = dense_lu_ms(torch, A, stream, reps=1 if n >= 8192 else 3)
        out["dense_lu_ms"] = dense_ms
    if dense_ms:
        key = "speedup_over_dense" if rc == 0 else "slowdown_vs_dense"
        out[key] = (dense_ms * 1e-3 / t_disp) if rc == 0 else (t_det + dense_ms * 1e-3) / (dense_ms * 1e-3)
    del A, AB
    return out


def measure_batched(torch, bandlu, w, dev, stream, flush, reps: int, fp64_peak: float, hbm_peak: float):
    from paper_2608_22099_gb300.workloads import make_workload
    n, kl, ku, ldab, B = w.n, w.kl, w.ku, w.ldab, w.batch
    A = make_workload(w, device=dev)
    AB = torch.zeros((B, n, ldab), dtype=torch.float64, device=dev)
    ipiv = torch.zeros((B, n), dtype=torch.int32, device=dev)
    kls, kus, infos, sts = (torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(4))

    def step():
        bandlu.check(bandlu.dispatch_lu_batched(A, n, n, n * n, B, AB, ldab, n * ldab, ipiv, n, kls, kus, infos,
                                                sts, stream), "dispatch_lu_batched")
    t = statistics.median(event_ms(torch, stream, step, reps, flush)) * 1e-3
    diag = AB[:, :, kl + ku].cpu().numpy()
    ip = ipiv.cpu().numpy()
    flops = sum(band_flops(ip[b], diag[b], n, kl, ku) for b in range(B))
    algo = 8.0 * B * n * n + 8.0 * B * n * ldab + 4.0 * B * n
    del A, AB
    return {"dispatch_batched_ms": t * 1e3, "gflops": flops / t / 1e9, "matrices_per_s": B / t,
            "hbm_gbs": algo / t / 1e9, "frac_hbm": algo / t / 1e9 / hbm_peak,
            "frac_fp64": flops / t / 1e9 / fp64_peak, "flops": flops,
            "status_all_banded": bool(int(sts.max().item()) == 0)}


def cpu_baseline_block(w, A_host_np, batched_w) -> dict:
    """The CPU oracle on this host: its dispatch single-threaded on a bounded sample of the
    workload (the leading principal block, same band and values) -- the reported value --
    plus detection and conversion of the whole matrix single-threaded and with OpenMP on all
    cores, and the batched workload with OpenMP over its matrices (timing build)."""
    import oracle
    from paper_2608_22099_gb300.workloads import make_workload
    times, flops = oracle_sample_dispatch(w, CPU_SAMPLE_N, steps=3, budget_s=12.0)
    value = flops / statistics.mean(times) / 1e9
    out = {"value": value, "unit": "GFLOP/s", "cores": 1, "kind": "oracle",
           "sample": (f"{len(times)} single-threaded oracle dispatches of the leading {CPU_SAMPLE_N} x "
                      f"{CPU_SAMPLE_N} principal block of the n={w.n} matrix (same kl, ku and values)"),
           "host_threads": host_threads(), "cpu_model": cpu_model()}
    stages = {}
    try:
        oracle.build(omp=True)
        omp_ok = True
    except Exception as e:  # noqa: BLE001 - reported, the single-threaded numbers stand
        omp_ok = False
        stages["omp_unavailable"] = str(e)[:200]
    n = w.n
    for omp in ((False, True) if omp_ok else (False,)):
        tag = "omp" if omp else "1t"
        t0 = time.perf_counter()
        kl, ku = oracle.detect_bandwidth(A_host_np, omp=omp)
        td = time.perf_counter() - t0
        t0 = time.perf_counter()
        oracle.dense_to_band(A_host_np, kl, ku, w.ldab, omp=omp)
        tc = time.perf_counter() - t0
        stages[f"detect_{tag}_s"] = td
        stages[f"detect_{tag}_gbs"] = 8.0 * n * n / td / 1e9
        stages[f"convert_{tag}_s"] = tc
    Ab = make_workload(batched_w).numpy()
    for omp in ((False, True) if omp_ok else (False,)):
        t0 = time.perf_counter()
        r = oracle.dispatch_lu_batched(Ab, batched_w.ldab, omp=omp)
        tb = time.perf_counter() - t0
        stages[f"batched_{'omp' if omp else '1t'}_s"] = tb
        stages[f"batched_{'omp' if omp else '1t'}_matrices_per_s"] = batched_w.batch / tb
    if int(r["status"].max()) != 0:
        raise RuntimeError("the oracle declined a batched matrix")
    out["stages"] = stages
    out["omp_threads"] = host_threads() if omp_ok else 1
    return out


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
    stream = torch.cuda.current_stream()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    hbm_peak, hbm_src = load_peaks()
    # the FP64 ceiling of this GPU, measured now (independent FMA chains, 16 warps per SM)
    fp64_peak = max(measure_fp64_fma(torch, dev, stream, sms) for _ in range(3))

    A = make_workload(w, device=dev)
    AB = torch.zeros((n, ldab), dtype=torch.float64, device=dev)
    ipiv = torch.zeros(n, dtype=torch.int32, device=dev)
    info = torch.zeros(1, dtype=torch.int32, device=dev)
    flush = L2Flush(torch, dev)

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
    torch.cuda.nvtx.range_push("timed_steps")  # lets a profiler select exactly these launches
    for k in range(args.steps):
        flush(k)                       # L2 flush between steps, outside the timed events
        starts[k].record(stream)
        step()
        ends[k].record(stream)
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_pop()
    barrier()
    t_wall1 = time.time()
    if rank == 0:
        sampler.stop()
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    # replicas: every rank factors its own matrix; the job's time is the slowest rank's
    ms_per_step = multirank.max_over_ranks(sum(step_ms), device=dev) / args.steps
    value = multirank.job_throughput(multirank.sum_over_ranks(flops, device=dev), ms_per_step * 1e-3) / 1e9

    # the same step with the decision on the device (dispatch_lu_async: no host round trip;
    # its factorisation is the same multi-CTA kernel, enqueued before the bandwidths are known)
    sc = torch.zeros(4, dtype=torch.int32, device=dev)
    AB3 = torch.zeros_like(AB)
    ipiv3 = torch.zeros_like(ipiv)

    def step_async():
        bandlu.check(bandlu.dispatch_lu_async(A, n, n, AB3, ldab, ipiv3, sc[0:1], sc[1:2], sc[2:3], sc[3:4], stream),
                     "dispatch_lu_async")
    async_ms = statistics.mean(event_ms(torch, stream, step_async, max(3, min(args.steps, 10)), flush))
    if tuple(int(v) for v in sc.cpu()) != (kl, ku, 0, 0) or not torch.equal(AB3, AB):
        raise RuntimeError("dispatch_lu_async disagrees with dispatch_lu")
    del AB3, ipiv3

    # stage breakdown through the same C ABI, CUDA events on the launching stream
    reps = max(3, min(args.steps, 10))
    klku = torch.zeros(2, dtype=torch.int32, device=dev)
    AB2 = torch.zeros_like(AB)
    ipiv2 = torch.zeros_like(ipiv)
    info2 = torch.zeros_like(info)
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

    detect_bytes = 8.0 * n * n
    nnz_band = n * (kl + ku + 1) - kl * (kl + 1) // 2 - ku * (ku + 1) // 2
    convert_bytes = 8.0 * nnz_band + 8.0 * ldab * n
    band_bytes = 2 * 8.0 * ldab * n
    fac_kernel = gbtrf_kernel(n, kl, ku)
    t_read = plain_read_s(torch, bandlu, A, dev, stream, flush, reps)
    stages = {
        "detect_us": t_detect * 1e6, "detect_gbs": detect_bytes / t_detect / 1e9,
        "detect_frac_hbm": detect_bytes / t_detect / 1e9 / hbm_peak,
        "plain_read_us": t_read * 1e6 if t_read else None,
        "detect_frac_of_plain_read": (t_read / t_detect) if t_read else None,
        "convert_us": t_convert * 1e6, "convert_gbs": convert_bytes / t_convert / 1e9,
        "gbtrf_kernel": fac_kernel, "gbtrf_us": t_gbtrf * 1e6, "gbtrf_gflops": flops / t_gbtrf / 1e9,
        "gbtrf_ns_per_column": t_gbtrf / n * 1e9, "gbtrf_frac_fp64": flops / t_gbtrf / 1e9 / fp64_peak,
        "gbtrf_frac_hbm": band_bytes / t_gbtrf / 1e9 / hbm_peak,
    }
    kernels = {"detect": t_detect, "convert": t_convert, "gbtrf": t_gbtrf}
    dominant = max(kernels, key=kernels.get)
    if dominant == "gbtrf":
        achieved = flops / t_gbtrf / 1e9
        roofline = {"bound": "alu", "achieved": achieved / 1e3, "peak": fp64_peak / 1e3, "unit": "TFLOP/s",
                    "frac": achieved / fp64_peak, "traffic": profiled_traffic(fac_kernel, WORKLOAD),
                    "kernel": fac_kernel,
                    "peak_source": "measured in this run: FP64 FMA microbenchmark (bandlu_peak_dfma, 16 warps/SM, "
                                   "8 independent chains per thread)",
                    "frac_of_nominal": achieved / FP64_NOMINAL_GFLOPS,
                    "algorithmic_flops_per_launch": flops}
    elif dominant == "detect":
        roofline = {"bound": "hbm", "achieved": detect_bytes / t_detect / 1e9, "peak": hbm_peak, "unit": "GB/s",
                    "frac": detect_bytes / t_detect / 1e9 / hbm_peak,
                    "traffic": profiled_traffic("k_detect_flat"), "kernel": "k_detect_flat", "peak_source": hbm_src}
    else:
        roofline = {"bound": "hbm", "achieved": convert_bytes / t_convert / 1e9, "peak": hbm_peak, "unit": "GB/s",
                    "frac": convert_bytes / t_convert / 1e9 / hbm_peak,
                    "traffic": profiled_traffic("k_dense_to_band_tiled"),
                    "kernel": "k_dense_to_band_tiled", "peak_source": hbm_src}

    # end to end: pinned host input -> device, dispatch_lu, factors back to pinned host memory
    A_host = torch.empty(A.shape, dtype=A.dtype, pin_memory=True)
    A_host.copy_(A)
    AB_host = torch.empty(AB.shape, dtype=AB.dtype, pin_memory=True)
    ipiv_host = torch.empty(ipiv.shape, dtype=ipiv.dtype, pin_memory=True)
    info_host = torch.empty(info.shape, dtype=info.dtype, pin_memory=True)
    A_e2e = torch.empty_like(A)
    e2e_reps = max(3, min(args.steps, 10))
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
    if not torch.equal(AB_host, AB.cpu()):
        raise RuntimeError("end-to-end factors differ")
    e2e_ms = multirank.max_over_ranks(statistics.mean(a.elapsed_time(b) for a, b in e2e_ev), device=dev)
    e2e_value = multirank.job_throughput(multirank.sum_over_ranks(flops, device=dev), e2e_ms * 1e-3) / 1e9
    h2d = A_host.numel() * 8
    d2h = AB_host.numel() * 8 + ipiv_host.numel() * 4 + info_host.numel() * 4
    del A_e2e, AB2

    # the other workload shapes, each through the same C ABI
    others = {}
    dense_16384 = None
    for name in OTHER_WORKLOADS:
        ow = WORKLOADS[name]
        if ow.batch:
            others[name] = measure_batched(torch, bandlu, ow, dev, stream, flush, 10, fp64_peak, hbm_peak)
        else:
            reuse = dense_16384 if (ow.n == 16384 and dense_16384) else None
            d = measure_single(torch, bandlu, ow, dev, stream, flush, 10 if ow.n <= 4096 else 5, fp64_peak,
                               hbm_peak, dense_ms=reuse)
            if ow.n == 16384:
                if dense_16384 is None:
                    dense_16384 = d.get("dense_lu_ms")
                else:
                    d["dense_lu_ms"] = dense_16384
                    d["dense_lu_from"] = "the n=16384 dense LU timed for n16384_kl8_ku64 (same n)"
            others[name] = d
    # the generic algorithm F(N) of Sec. III-A for this matrix: the dense LU at n/2 on this GPU
    # (timed above for the n=16384 shape), scaled by (n / (n/2))^3 -- an estimate, not three
    # full-size cuSOLVER runs
    dense_est = dense_16384 * 8.0 if (dense_16384 and n == 32768) else None

    cpu_baseline = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu_baseline = cpu_baseline_block(w, A_host.numpy(), WORKLOADS["batch4096_n256_kl2_ku2"])

    clocks = sampler.summary(t_wall0, t_wall1) if rank == 0 else None
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "GFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w),
            "config_notes": {"dist": "uniform[-1,1] band, no diagonal boost, seed 1005",
                             "l2": "inputs (8 GiB) larger than L2, and L2 flushed between steps (512 MiB write, "
                                   "then a 256 MiB read)",
                             "parallelism": "replicas" if world > 1 else "single"},
            "dispatch_ms": ms_per_step, "dispatch_async_ms": async_ms, "flops_per_step": flops, "stages": stages,
            "dense_lu_ms_estimate": dense_est,
            "dense_lu_estimate_from": "cuSOLVER getrf (torch) timed at n=16384 on this GPU, x (32768/16384)^3",
            "speedup_over_dense_estimate": (dense_est / ms_per_step) if dense_est else None,
            "memory_ratio_dense_over_band": (8.0 * n * n) / (8.0 * ldab * n),
            "roofline": roofline, "fp64_peak_measured_gflops": fp64_peak,
            "cpu_baseline": cpu_baseline,
            "e2e": {"value": e2e_value, "unit": "GFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "ms_per_step": e2e_ms},
            "gpu_launches": 4 * args.steps,
            "gpu_launches_note": "per step: k_detect_reset, k_detect_flat, k_dense_to_band_tiled and the factorisation kernel",
            "clocks": clocks,
            "wall_s_timed": t_wall1 - t_wall0,
            "workloads": others,
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
        # captured once in a CUDA graph and replayed
        if True:
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


def trace_summary(T: np.ndarray, lo: int, hi: int) -> dict:
    """Summary of a chain-kernel timeline (roles x entries x slots, include/bandlu_trace.h)
    over entries [lo, hi): medians, means and 90th percentiles of the intervals between its
    stamps, in the timer's unit."""
    def st(x):
        x = np.asarray(x, dtype=np.float64)
        return {"median": float(np.median(x)), "mean": float(x.mean()), "p90": float(np.percentile(x, 90))}
    A0, S1, S2, L = T[0], T[1], T[2], T[3]
    q = np.arange(lo, hi)
    out = {}
    out["panel_cta"] = {
        "period": st(A0[q + 1, 0] - A0[q, 0]),
        "factor_to_step2_records_sent": st(A0[q, 1] - A0[q, 0]),
        "step2_records_sent_to_panel_done": st(A0[q, 2] - A0[q, 1]),
        "wait_for_next_block": st(A0[q, 3] - A0[q, 2]),
        "block_in_to_next_panel_start": st(A0[q + 1, 0] - A0[q, 3]),
    }
    for k in range(4):
        out["panel_cta"][f"step{k}_start_to_barrier"] = st(A0[q, 5 + 3 * k] - A0[q, 4 + 3 * k])
        out["panel_cta"][f"step{k}_barrier_to_records_sent"] = st(A0[q, 6 + 3 * k] - A0[q, 5 + 3 * k])
    out["panel_cta"]["panel_start_to_step0_start"] = st(A0[q, 4] - A0[q, 0])
    # streamer 1 applies panel q's steps 0..2 to block q+1; its last records are step 2's
    out["streamer1"] = {
        "block_in_to_first_records": st(S1[q, 1] - S1[q, 0]),
        "last_records_wait_starts_after_sent": st(S1[q, 2] - A0[q, 1]),
        "last_records_seen_after_sent": st(S1[q, 3] - A0[q, 1]),
        "last_step_and_band_send": st(S1[q, 4] - S1[q, 3]),
        "band_sent_to_panel_cta_has_block": st(A0[q, 3] - S1[q, 4]),
    }
    out["streamer2"] = {
        "block_in_to_first_records": st(S2[q, 1] - S2[q, 0]),
        "last_records_seen_after_panel_cta_done": st(S2[q, 3] - A0[q, 2]),
        "band_sent_to_streamer1_block_in": st(S1[q + 1, 0] - S2[q, 4]),
    }
    bq = q[L[q, 0] > 0]
    out["loader_wait_for_hand_over"] = st(L[bq, 1] - L[bq, 0]) if bq.size else None
    # the supply path: panel b-5 done on A -> its update CTA has applied it and handed block b
    # over (the loader sees the flag)
    bs = bq[bq >= lo + 5]
    out["panel_done_to_hand_over_seen"] = st(L[bs, 1] - A0[bs - 5, 2]) if bs.size else None
    return out


def run_trace(args):
    """Timeline of the wide-band chain kernel from the traced build (include/bandlu_trace.h):
    one factorisation of the workload's band (after two untimed ones), the global timer at
    every panel boundary and wait of the panel CTA, streamers 1 and 2 and the last streamer's
    loader, summarised over the panels away from both ends.  One JSON line."""
    os.environ["BANDLU_TRACE"] = "1"  # before the library is loaded
    import torch

    from paper_2608_22099_gb300 import bandlu
    from paper_2608_22099_gb300.workloads import WORKLOADS, Workload, make_workload

    if args.custom:
        cn, ckl, cku = args.custom[:3]
        w = Workload(f"custom_n{cn}_kl{ckl}_ku{cku}", cn, ckl, cku, "uniform", 0.0, 7)
    else:
        w = WORKLOADS[args.workload]
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    bandlu.load()
    cap = bandlu.bandlu_trace_capacity()
    if cap <= 0:
        raise RuntimeError("the traced library was not loaded")
    n, kl, ku, ldab = w.n, w.kl, w.ku, w.ldab
    kern = gbtrf_kernel(n, kl, ku)
    A = make_workload(w, device=dev)
    AB0 = torch.zeros((n, ldab), dtype=torch.float64, device=dev)
    stream = torch.cuda.current_stream()
    bandlu.check(bandlu.dense_to_band(A, n, n, kl, ku, AB0, ldab, stream), "convert")
    del A
    AB = torch.empty_like(AB0)
    ipiv = torch.zeros(n, dtype=torch.int32, device=dev)
    info = torch.zeros(1, dtype=torch.int32, device=dev)
    times = []
    for rep in range(3):
        AB.copy_(AB0)
        if rep == 2:
            bandlu.check(bandlu.bandlu_trace_clear(), "trace_clear")
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        bandlu.check(bandlu.gbtrf(n, kl, ku, AB, ldab, ipiv, info, stream), "gbtrf")
        b.record(stream)
        torch.cuda.synchronize()
        times.append(a.elapsed_time(b))
    T = np.zeros(4 * cap * 16, dtype=np.uint64)
    bandlu.check(bandlu.bandlu_trace_read(T, T.size), "trace_read")
    T = T.reshape(4, cap, 16).astype(np.int64)
    npan = (n + 3) // 4
    lo, hi = min(64, npan // 4), min(cap, npan) - min(64, npan // 4)
    out = {"mode": "trace", "workload": w.name, "kernel": kern, "n": n, "kl": kl, "ku": ku,
           "gbtrf_ms_traced_run": times[2],
           "panels_summarised": [lo, hi], "unit": "ns"}
    if kern != "k_gbtrf_wide_chain" or hi - lo < 8 or not T[0, lo:hi, 0].all():
        out["note"] = "no chain-kernel timeline for this band"
        print(json.dumps(out))
        return

    out.update(trace_summary(T, lo, hi))
    print(json.dumps(out))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="workload name (default: the n=32768, kl=ku=256 matrix); others for per-workload reports")
    ap.add_argument("--sweep", action="store_true", help="the paper's experiments A-C (speedup / slowdown in N)")
    ap.add_argument("--peaks", action="store_true", help="FP64 FMA / DMMA and HBM read microbenchmarks")
    ap.add_argument("--trace", action="store_true",
                    help="timeline of the wide-band chain kernel from the traced build (bandlu_trace.h)")
    ap.add_argument("--custom", type=int, nargs="+", metavar="N KL KU [BATCH]",
                    help="per-stage report of a synthetic uniform[-1,1] band of this shape (batched if BATCH > 0)")
    args = ap.parse_args()
    if args.custom is not None and len(args.custom) not in (3, 4):
        ap.error("--custom takes N KL KU [BATCH]")
    if args.impl == "reference":
        run_reference(args)
    elif args.trace:
        run_trace(args)
    elif args.peaks:
        run_peaks(args)
    elif args.sweep:
        run_sweep(args)
    elif args.custom or args.workload != WORKLOAD:
        run_workload_report(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
