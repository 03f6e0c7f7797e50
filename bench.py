"""Benchmark of LAM's quantized-memory hot path on GB300.

Headline workload (mem_n8388608_l2): a memory of 8,388,608 unit-norm fp32
embeddings (D = 768, 25.8 GB) resident in HBM.  One step is one pass of the
whole path over it: Q_eps of the eight 1M-row slabs to int8 codes at
eps = 1e-2 (the forced width the workload names), then exact L2 top-100 search
of one query over the whole quantized memory (fused dequant + score + top-k,
then the merge of partial lists).  Everything runs through the C ABI;
`value` is memory vectors per second through the whole step, and `roofline`
is the step's dominant kernel against the measured HBM copy bandwidth.

The other workloads (the PR1 cosine case, the 27,986-chunk eps sweep, the
flat 2^26 quantize microbench, the 361,802-record memory at B = 1 / 64 /
4,096, and the 8.4M-row memory at B = 256) are measured call by call in the
same run and reported under "configs", each with the oracle timed beside it.

    python bench.py [--gpus N] [--steps K] [--warmup W]
    python bench.py --impl reference ...       # the CPU oracle on host cores
    python bench.py --kernels --workload NAME  # per-call timings of one workload

With --gpus N > 1 (launched by torchrun) every rank runs an independent
replica of the workload on its own GPU; there is no exchange between ranks.
"""
from __future__ import annotations

import argparse
import concurrent.futures as cf
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "Q_ε GB/s and fused score+top-k memory vectors/s at D=768; % of HBM roofline"
UNIT = "memory vectors/s"
L2_FLUSH_BYTES = 512 << 20
HEADLINE = "mem_n8388608_l2"
SLAB_SEED = 1000  # slab j of the 8.4M-row memory is drawn with seed 1000 + j
# rows of the headline memory the oracle processes per timed sample
ORACLE_ROWS = 1 << 18
ORACLE_ROWS_1CORE = 1 << 16


class L2Flush:
    """Evicts the 129 MB L2 between timed calls: writes one buffer larger
    than L2, then reads another, so that no dirty line of the flush is left
    for the timed kernels to write back."""

    def __init__(self, torch, dev):
        self.a = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
        self.b = torch.zeros(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)

    def __call__(self, i):
        self.a.fill_(float(i))
        self.b.sum()


# DRAM bytes (read + write) of one launch of a kernel, from one ncu capture
# (the profiles/ summary of that kernel).  Reported only while the kernel's
# source file is the one the counters were taken on.
KERNEL_TRAFFIC = {
    "quantize_forced_kernel": {"source": "quantize.cu", "source_sha256_16": "6a8dfe92d4b7bb82",
                               "bytes": 4 * (805358080 + 184268288),
                               "launch": "ncu, cold caches, one launch on 262,144 rows x 768 "
                                         "(805 MB of fp32) scaled x 4 to a 1M-row slab"},
    "score_bw_kernel": {"source": "score_bw.cu", "source_sha256_16": "", "bytes": 0,
                        "launch": ""},
}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=100)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="lam", choices=["lam", "reference"])
    p.add_argument("--workload", default=HEADLINE, help="(--kernels) workload to time")
    p.add_argument("--batch", type=int, default=0, help="(--kernels) one query batch")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-configs", action="store_true",
                   help="skip the per-call measurements of the other workloads")
    p.add_argument("--kernels", action="store_true",
                   help="time each C-ABI call of --workload separately (not the headline step)")
    p.add_argument("--reps", type=int, default=20)
    p.add_argument("--eps", type=float, default=0.0, help="(--kernels) one eps instead of the sweep")
    p.add_argument("--width", type=int, default=-1, help="(--kernels) forced code width")
    p.add_argument("--rows", type=int, default=0,
                   help="(--kernels) a smaller memory of the same workload (profiling captures)")
    p.add_argument("--only", default="",
                   help="(--kernels) comma list of parts: quantize,bands,codec,admit,score,rows")
    return p.parse_args()


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return pk["hbm_gbs"], pk["bf16_tflops"], "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the GPU is measured.
    The samples go to a temporary file that is removed afterwards."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index, interval_ms=20):
        self.index = index
        self.interval_ms = interval_ms
        self.proc = None
        self.rows = []

    def __enter__(self):
        try:
            self.fh = tempfile.NamedTemporaryFile("w+", prefix="lam_clocks_", suffix=".csv")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", str(self.interval_ms)],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        try:
            self.fh.flush()
            self.fh.seek(0)
            for line in self.fh:
                f = [x.strip() for x in line.split(",")]
                if len(f) >= 9:
                    self.rows.append(f)
        finally:
            self.fh.close()

    def summary(self, window):
        if self.proc is None or not self.rows:
            return None

        def num(v):
            try:
                return float(v)
            except ValueError:
                return None
        sm = [num(r[1]) for r in self.rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in self.rows if num(r[2]) is not None]
        pw = [num(r[3]) for r in self.rows if num(r[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[j] for r in self.rows for j in range(4) if r[5 + j] == "Active"})
        # samples taken while the GPU drew well above its idle power
        loaded = [num(r[1]) for r in self.rows
                  if num(r[1]) is not None and (num(r[3]) or 0.0) > 300.0]
        return {"sm_mhz": statistics.median(loaded or sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(self.rows), "samples_under_load": len(loaded),
                "power_w_max": max(pw) if pw else None, "window": window}


def dist_setup(args, backend=None):
    """Rank geometry from the torchrun environment; joins the process group
    when there is more than one rank (NCCL for the GPU arm, gloo otherwise)."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if backend is None:
            backend = "nccl" if args.impl == "lam" else "gloo"
        dist.init_process_group(backend=backend)
    return world, rank, local


def max_over_ranks(value, world, device=None):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def aggregate_replicas(ms_step_local, units_per_step, world, device=None):
    """Replicas only: every rank runs the whole workload on its own GPU, so the
    job's step time is the slowest rank's and its throughput counts the units
    of all ranks.  Returns (ms_per_step, units per second)."""
    ms = max_over_ranks(ms_step_local, world, device)
    return ms, units_per_step * world / (ms / 1e3)


def headline_config(wl, B):
    """The workload description both arms print (identical keys and values)."""
    return {"workload": wl.name, "N": wl.n, "D": wl.d, "batch": B, "k": wl.k,
            "metric": ["ip", "cosine", "l2"][wl.metric], "eps": list(wl.eps),
            "code_width": "int8 (forced)", "slab_rows": wl.slab_rows,
            "parallelism": "replicas only",
            "l2": "inputs larger than L2: 25.8 GB of fp32 read per step, no flush"}


def traffic_for(kname):
    """ncu DRAM bytes per launch of a kernel, while its source is unchanged."""
    tr = KERNEL_TRAFFIC.get(kname)
    if not tr or not tr["bytes"]:
        return None, None
    try:
        import hashlib
        with open(os.path.join(ROOT, "paper_2609_32256_gb300", "csrc", tr["source"]), "rb") as f:
            if hashlib.sha256(f.read()).hexdigest()[:16] == tr["source_sha256_16"]:
                return tr["bytes"], tr["launch"]
    except OSError:
        pass
    return None, None


# ------------------------------------------------------------ oracle timing --

def oracle_quantize_rows(x, eps, threads):
    """oracle.quantize over row chunks of x on `threads` host threads (the
    oracle call itself is unchanged; ctypes releases the GIL).  Returns
    (codes int32 [N, D], rmin, rmax)."""
    import numpy as np
    import oracle
    N = x.shape[0]
    if threads <= 1:
        c, rmin, rmax, _ = oracle.quantize(x, eps)
        return c.reshape(x.shape), rmin, rmax
    step = max(1, -(-N // (4 * threads)))
    spans = [(r, min(N, r + step)) for r in range(0, N, step)]
    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        parts = list(ex.map(lambda s: oracle.quantize(x[s[0]:s[1]], eps), spans))
    return (np.concatenate([p[0] for p in parts]).reshape(x.shape),
            min(p[1] for p in parts), max(p[2] for p in parts))


def oracle_mem_step(x, q, eps, metric, k, threads):
    """One sample of the headline step on the host: the oracle quantizes the
    rows x and searches them with the queries q.  Returns seconds."""
    import oracle
    t0 = time.perf_counter()
    c, _, _ = oracle_quantize_rows(x, eps, threads)
    oracle.search(q, c, eps, metric, k, nthreads=threads)
    return time.perf_counter() - t0


def oracle_timing(x, q, eps_list, metric, k, threads, dequant=False, search=True):
    """Seconds for the oracle to quantize (and dequantize) the rows x at every
    eps and search them with q."""
    import oracle
    t0 = time.perf_counter()
    for e in eps_list:
        c, _, _ = oracle_quantize_rows(x, e, threads)
        if dequant:
            oracle.dequantize(c, oracle.step(e))
        if search and q is not None:
            oracle.search(q, c.reshape(x.shape[0], -1), e, metric, k, nthreads=threads)
    return time.perf_counter() - t0


def cpu_baseline_mem(x_rows, q, wl, cores, min_s=6.0):
    """The oracle on the headline workload, on a bounded sample of its rows:
    all host cores on ORACLE_ROWS rows (the reference arm's step), and one
    core on ORACLE_ROWS_1CORE rows, each repeated until it has run for at
    least `min_s` seconds (at least twice); rows per second over all runs."""
    eps = wl.eps[0]

    def rate(rows, threads):
        n = t = 0
        while n < 2 or t < min_s:
            t += oracle_mem_step(x_rows[:rows], q, eps, wl.metric, wl.k, threads)
            n += 1
        return rows * n / t, n

    v_all, n_all = rate(ORACLE_ROWS, cores)
    v_one, n_one = rate(ORACLE_ROWS_1CORE, 1)
    return {"value": v_all, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "the oracle quantizes %d of the memory's rows (slab 0) to int8 at eps=%g "
                      "and runs the exact L2 top-%d search of the %d query over them, on %d "
                      "threads (row chunks for Q_eps, rows split for the search), %d times"
                      % (ORACLE_ROWS, eps, wl.k, q.shape[0], cores, n_all),
            "single_core": {"value": v_one, "unit": UNIT, "cores": 1,
                            "sample": "the same on %d rows, one thread, %d times"
                                      % (ORACLE_ROWS_1CORE, n_one)}}


# ----------------------------------------------------------------- lam arm --

class MemStep:
    """The headline step: Q_eps of every 1M-row slab of the resident fp32
    memory to int8 codes, then L2 top-k search of the query batch over all
    codes, all through the C ABI on one stream."""

    def __init__(self, lam, torch, wl, B, dev):
        self.lam, self.torch, self.wl, self.dev = lam, torch, wl, dev
        N, D, S = wl.n, wl.d, wl.slab_rows
        self.N, self.D, self.S, self.B = N, D, S, B
        self.eps = wl.eps[0]
        self.n_slabs = N // S
        self.x = torch.empty((N, D), dtype=torch.float32, device=dev)
        from paper_2609_32256_gb300 import inputs
        for j in range(self.n_slabs):
            self.x[j * S:(j + 1) * S] = inputs.unit_rows_device(S, D, seed=SLAB_SEED + j,
                                                                device=dev)
        self.codes = torch.empty((N, D), dtype=torch.int8, device=dev)
        # one 32-byte quantize status block per slab (256-byte stride)
        self.qws = torch.zeros((self.n_slabs, 256), dtype=torch.uint8, device=dev)
        self.q = torch.from_numpy(inputs.queries(B, D, seed=1)).to(dev)
        self.scores = torch.empty((B, wl.k), dtype=torch.float32, device=dev)
        self.ids = torch.empty((B, wl.k), dtype=torch.int64, device=dev)
        self.code_bound = 128  # every int8 code
        self.path = lam.lam_score_topk_path(B, N, D, wl.k, 1, self.code_bound)
        self.sws = torch.empty(lam.lam_score_topk_workspace_size(B, N, D, wl.k, 1,
                                                                 self.code_bound),
                               dtype=torch.uint8, device=dev)

    def slab(self, t, j):
        return t[j * self.S:(j + 1) * self.S]

    def step(self, stream=None):
        """Device-resident: the quantize statuses stay on the device and are
        checked after the timed steps (check())."""
        lam = self.lam
        for j in range(self.n_slabs):
            lam.lam_quantize_async(self.slab(self.x, j), self.eps, lam.LAM_I8,
                                   self.slab(self.codes, j), self.qws[j], stream=stream)
        lam.lam_score_topk(self.q, self.codes, 1, self.N, self.D, self.eps, self.code_bound,
                           self.wl.k, self.wl.metric, self.scores, self.ids, self.sws,
                           stream=stream)

    def step_host_sync(self):
        """The synchronous calls: the host reads every slab's quantize status
        (width and range) before it queues the search."""
        lam = self.lam
        for j in range(self.n_slabs):
            st, w, *_ = lam.lam_quantize(self.slab(self.x, j), self.eps, lam.LAM_I8,
                                         self.slab(self.codes, j), self.qws[j])
            assert st == 0 and w == 1
        lam.lam_score_topk(self.q, self.codes, 1, self.N, self.D, self.eps, self.code_bound,
                           self.wl.k, self.wl.metric, self.scores, self.ids, self.sws)

    def check(self):
        lam = self.lam
        for j in range(self.n_slabs):
            st, w, *_ = lam.lam_quantize_result(self.qws[j], self.eps, lam.LAM_I8)
            assert st == 0 and w == 1
        assert lam.lam_score_topk_status(self.sws) == 0


def measure_calls(lam, torch, dev, wl, parts, reps, batches=None, eps_list=None, width=-1,
                  x=None, codes_in=None):
    """Per-call timing of one workload: Q_eps (AUTO and at the workload's
    width), dequantisation and lam_score_topk per query batch, each as the mean
    of `reps` CUDA-event spans with a 512 MB L2 flush before every rep, plus
    the device time of the call's own kernels from the library's events."""
    from paper_2609_32256_gb300 import inputs
    if x is None and codes_in is None:
        if wl.d == 1:
            x = torch.from_numpy(inputs.flat_values(wl.n, seed=0)).to(dev)
        elif wl.slab_rows:
            x = inputs.unit_rows_device(wl.n, wl.d, seed=0, device=dev)
        elif wl.planted:
            x = torch.from_numpy(inputs.planted_rows(wl.n, wl.d, seed=0)).to(dev)
        else:
            x = torch.from_numpy(inputs.unit_rows(wl.n, wl.d, seed=0)).to(dev)
    n = wl.n * wl.d
    flush = L2Flush(torch, dev)
    ws = torch.zeros(64, dtype=torch.uint8, device=dev)
    codes = codes_in if codes_in is not None else torch.empty(n * 4, dtype=torch.uint8,
                                                              device=dev)
    out = torch.empty(n, dtype=torch.float32, device=dev) if "dequantize" in parts else None

    def timed(fn, kind):
        """(mean call span ms, mean device ms of the call's `kind` kernel launches)."""
        for i in range(3):
            flush(i)
            fn()
        tot = 0.0
        lam.lam_timing_begin(kind, reps * 64)
        for i in range(reps):
            flush(i)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize(dev)
            tot += e0.elapsed_time(e1)
        k_ms, _, _ = lam.lam_timing_read(kind)
        lam.lam_timing_end()
        return tot / reps, k_ms / reps

    res = {"workload": wl.name, "n_values": n}
    hbm, tc_peak, kind = load_peaks()
    widths = {}
    eps_list = eps_list or wl.eps
    for e in eps_list:
        if codes_in is not None:
            widths[e] = (width, 2.0 * e, 128 if width == 1 else 0)
            continue
        _, w, sc, cmin, cmax = lam.lam_quantize(x, e, 0, None, ws)
        wq = width if width > 0 else (wl.width or w)
        widths[e] = (wq, sc, max(-cmin, cmax))
        if "quantize" in parts:
            ms_auto, k_auto = timed(lambda: lam.lam_quantize(x, e, 0, codes, ws),
                                    lam.LAM_TIME_QUANTIZE)
            ms_forced, k_forced = timed(lambda: lam.lam_quantize(x, e, wq, codes, ws),
                                        lam.LAM_TIME_QUANTIZE)
            qb, qa = (4 + wq) * n, (4 + w) * n  # AUTO writes the resolved width
            res.setdefault("quantize", []).append({
                "eps": e, "width": wq, "width_auto": w, "ms_auto_span": ms_auto,
                "ms_auto_kernel": k_auto, "ms_forced_span": ms_forced,
                "ms_forced_kernel": k_forced,
                "gbs_auto_kernel": qa / (k_auto / 1e3) / 1e9,
                "frac_of_hbm_auto_kernel": qa / (k_auto / 1e3) / 1e9 / hbm,
                "gbs_forced_kernel": qb / (k_forced / 1e3) / 1e9,
                "frac_of_hbm_forced_kernel": qb / (k_forced / 1e3) / 1e9 / hbm})
        if "dequantize" in parts:
            lam.lam_quantize(x, e, wq, codes, ws)
            ms_d, k_d = timed(lambda: lam.lam_dequantize(codes, wq, n, sc, out),
                              lam.LAM_TIME_DEQUANTIZE)
            gbd = (wq + 4) * n / (k_d / 1e3) / 1e9
            res.setdefault("dequantize", []).append({
                "eps": e, "width": wq, "ms_span": ms_d, "ms_kernel": k_d, "gbs_kernel": gbd,
                "frac_of_hbm_kernel": gbd / hbm})
    if wl.d > 1 and "bands" in parts:
        # Q_eps fused with the band digests (r = 4 and 8, the paper's shipped and
        # best band widths), codes written, AUTO width
        res["bands"] = []
        N = wl.n
        for r in (4, 8):
            dig = torch.empty((N, wl.d // r), dtype=torch.int64, device=dev)
            for e in eps_list:
                xr = x.view(N, wl.d)
                st, w, *_ = lam.lam_quantize_bands(xr, e, 0, r, codes, dig, ws)
                ms, k_ms = timed(lambda: lam.lam_quantize_bands(xr, e, 0, r, codes, dig, ws),
                                 lam.LAM_TIME_QUANTIZE)
                nbytes = (4 + w) * n + 8 * (n // r)
                res["bands"].append({"r": r, "eps": e, "width": w, "ms_span": ms,
                                     "ms_kernel": k_ms,
                                     "gbs_kernel": nbytes / (k_ms / 1e3) / 1e9,
                                     "frac_of_hbm_kernel": nbytes / (k_ms / 1e3) / 1e9 / hbm})
            del dig
    if wl.d == 1 and "codec" in parts:
        # the error-bounded byte codec at the paper's relative bounds (its
        # deployed bound is 1% of max|x|), on the first 2^24 values and all
        res["codec"] = []
        for n_c in sorted({min(n, 1 << 24), n}):
            xc = x[:n_c]
            cbuf = torch.empty(lam.lam_lamz_bound(n_c), dtype=torch.uint8, device=dev)
            cws = torch.empty(lam.lam_lamz_workspace_size(n_c), dtype=torch.uint8, device=dev)
            yc = torch.empty(n_c, dtype=torch.float32, device=dev)
            for rel in (1e-3, 1e-2, 3e-2):
                st, nbytes = lam.lam_lamz_compress(xc, rel, cbuf, cws)
                ms_c, _ = timed(lambda: lam.lam_lamz_compress(xc, rel, cbuf, cws),
                                lam.LAM_TIME_AUX)
                ms_d, _ = timed(lambda: lam.lam_lamz_decompress(cbuf, nbytes, yc, cws),
                                lam.LAM_TIME_AUX)
                res["codec"].append({"n": n_c, "rel": rel, "ratio": 4.0 * n_c / nbytes,
                                     "compress_ms_span": ms_c,
                                     "compress_gbs": 4.0 * n_c / (ms_c / 1e3) / 1e9,
                                     "decompress_ms_span": ms_d,
                                     "decompress_gbs": 4.0 * n_c / (ms_d / 1e3) / 1e9})
            del cbuf, cws, yc
    if wl.planted and "admit" in parts:
        # batch admission (Algorithm 2) at cos >= 0.95 over band candidates at
        # the paper's shipped (r = 4, eps = 0.2 sigma) and relaxed (r = 8, 0.3 sigma)
        # operating points: digests from the fused pass, then lam_admit_batch
        res["admit"] = []
        N, sigma = wl.n, 1.0 / (wl.d ** 0.5)
        delta = (2.0 - 2.0 * 0.95) ** 0.5
        xr = x.view(N, wl.d)
        for r, rel in ((4, 0.2), (8, 0.3)):
            dig = torch.empty((N, wl.d // r), dtype=torch.int64, device=dev)
            lam.lam_quantize_bands(xr, rel * sigma, 0, r, None, dig, ws)
            rep = torch.empty(N, dtype=torch.int32, device=dev)
            dist = torch.empty(N, dtype=torch.float64, device=dev)
            mp = 1 << 20
            while True:
                aws = torch.empty(lam.lam_admit_batch_workspace_size(N, wl.d // r, mp),
                                  dtype=torch.uint8, device=dev)
                st, dh, kept, npairs = lam.lam_admit_batch(xr, dig, delta, rep, dist, aws, mp,
                                                           raise_on_error=False)
                if st == 0:
                    break
                mp = npairs
                del aws
            ms, _ = timed(lambda: lam.lam_admit_batch(xr, dig, delta, rep, dist, aws, mp),
                          lam.LAM_TIME_AUX)
            res["admit"].append({"r": r, "eps": rel * sigma, "t": 0.95, "ms_span": ms,
                                 "records_per_s": N / (ms / 1e3), "candidate_pairs": npairs,
                                 "retained": kept, "delta_hat": dh})
            del aws, dig
    if wl.batches and wl.d > 1 and "score" in parts:
        e = eps_list[0]
        wq, sc, bound = widths[e]
        if codes_in is None:
            lam.lam_quantize(x, e, wq, codes, ws)
        N = wl.n
        res["score"] = []
        for B in (batches or list(wl.batches)):
            q = torch.from_numpy(inputs.queries(B, wl.d, seed=1)).to(dev)
            nb = lam.lam_score_topk_workspace_size(B, N, wl.d, wl.k, wq, bound)
            sws = torch.empty(nb, dtype=torch.uint8, device=dev)
            s_ = torch.empty((B, wl.k), dtype=torch.float32, device=dev)
            i_ = torch.empty((B, wl.k), dtype=torch.int64, device=dev)
            path = lam.lam_score_topk_path(B, N, wl.d, wl.k, wq, bound)

            def call():
                lam.lam_score_topk(q, codes, wq, N, wl.d, e, bound, wl.k, wl.metric, s_, i_,
                                   sws)
            ms, k_s = timed(call, lam.LAM_TIME_SCORE)
            _, k_m = timed(call, lam.LAM_TIME_MERGE)
            _, k_a = timed(call, lam.LAM_TIME_AUX)
            assert lam.lam_score_topk_status(sws) == 0
            code_bytes = N * wl.d * wq
            fl = 2.0 * N * wl.d * B
            res["score"].append({"B": B, "path": ["bandwidth", "tensor", "generic"][path],
                                 "ms_span": ms, "ms_kernel": k_s, "ms_merge": k_m,
                                 "ms_prep": k_a,
                                 "vectors_per_s_span": N / (ms / 1e3),
                                 "code_gbs_kernel": code_bytes / (k_s / 1e3) / 1e9,
                                 "frac_of_hbm_kernel": code_bytes / (k_s / 1e3) / 1e9 / hbm,
                                 "tflops_kernel": fl / (k_s / 1e3) / 1e12,
                                 "frac_of_tensor_kernel": fl / (k_s / 1e3) / 1e12 / tc_peak})
            del sws
    if wl.batches and wl.d > 1 and "rows" in parts:
        # the per-vector byte codecs of the composite experiment: encode, and
        # exact search over the coded rows (decoding folded into the score)
        res["rows"] = []
        N, D = wl.n, wl.d
        xr = x.view(N, D)
        names = {lam.LAM_ROWS_INT8: "int8/vector", lam.LAM_ROWS_FP16: "fp16",
                 lam.LAM_ROWS_SIGN: "sign"}
        row_bytes = {lam.LAM_ROWS_INT8: D + 8, lam.LAM_ROWS_FP16: 2 * D,
                     lam.LAM_ROWS_SIGN: D // 8 + 4}
        for fmt in (lam.LAM_ROWS_INT8, lam.LAM_ROWS_FP16, lam.LAM_ROWS_SIGN):
            rc, rs, ro = lam.encode_rows(xr, fmt)
            ms_e, k_e = timed(lambda: lam.lam_encode_rows(xr, fmt, rc, rs, ro),
                              lam.LAM_TIME_QUANTIZE)
            eb = N * (4 * D + row_bytes[fmt])
            for B in (batches or list(wl.batches)):
                q = torch.from_numpy(inputs.queries(B, D, seed=1)).to(dev)
                nb = lam.lam_score_topk_rows_workspace_size(B, N, D, wl.k, fmt)
                sws = torch.empty(nb, dtype=torch.uint8, device=dev)
                s_ = torch.empty((B, wl.k), dtype=torch.float32, device=dev)
                i_ = torch.empty((B, wl.k), dtype=torch.int64, device=dev)
                path = lam.lam_score_topk_rows_path(B, N, D, wl.k, fmt)

                def call():
                    lam.lam_score_topk_rows(q, rc, fmt, rs, ro, N, D, wl.k, wl.metric, s_, i_,
                                            sws)
                ms, k_s = timed(call, lam.LAM_TIME_SCORE)
                _, k_m = timed(call, lam.LAM_TIME_MERGE)
                _, k_a = timed(call, lam.LAM_TIME_AUX)
                fl = 2.0 * N * D * B
                res["rows"].append({"codec": names[fmt], "ratio_vs_fp32": 4.0 * D / row_bytes[fmt],
                                    "encode_ms_kernel": k_e,
                                    "encode_gbs_kernel": eb / (k_e / 1e3) / 1e9,
                                    "B": B, "path": ["bandwidth", "tensor", "generic"][path],
                                    "ms_span": ms, "ms_kernel": k_s, "ms_merge": k_m,
                                    "ms_prep": k_a,
                                    "vectors_per_s_span": N / (ms / 1e3),
                                    "code_gbs_kernel": N * row_bytes[fmt] / (k_s / 1e3) / 1e9,
                                    "frac_of_hbm_kernel": N * row_bytes[fmt] / (k_s / 1e3) / 1e9 / hbm,
                                    "tflops_kernel": fl / (k_s / 1e3) / 1e12,
                                    "frac_of_tensor_kernel": fl / (k_s / 1e3) / 1e12 / tc_peak})
                del sws
            del rc, rs, ro
    res["peaks"] = {"hbm_gbs": hbm, "bf16_tflops": tc_peak, "kind": kind}
    return res


def other_configs(lam, torch, dev, mem, cores, reps, with_oracle):
    """Per-call measurements of the other workloads (and of the headline
    memory at B = 256), each with the oracle timed on a bounded sample."""
    import numpy as np
    from paper_2609_32256_gb300 import inputs
    W = inputs.WORKLOADS
    out = {}

    def host_rows(wl):
        if wl.d == 1:
            return inputs.flat_values(wl.n, seed=0)
        if wl.planted:
            return inputs.planted_rows(wl.n, wl.d, seed=0)
        return inputs.unit_rows(wl.n, wl.d, seed=0)

    # PR1: 4,096 rows, forced int16, cosine top-10 of 16 queries
    wl = W["pr1_n4096_cos"]
    r = measure_calls(lam, torch, dev, wl, {"quantize", "dequantize", "score"}, reps)
    if with_oracle:
        xh = host_rows(wl)
        q = inputs.queries(16, wl.d, seed=1)
        t = oracle_timing(xh, q, wl.eps, wl.metric, wl.k, cores)
        r["oracle"] = {"vectors_per_s": wl.n / t, "cores": cores,
                       "sample": "all rows quantized and searched by all 16 queries"}
    out[wl.name] = r
    # chunks: 27,986 rows with planted near-duplicates, eps sweep, AUTO width,
    # dequantisation, 1,024 queries IP top-10
    wl = W["chunks_n27986_ip"]
    r = measure_calls(lam, torch, dev, wl, {"quantize", "dequantize", "score"}, reps)
    if with_oracle:
        xh = host_rows(wl)
        q = inputs.queries(1024, wl.d, seed=1)[:64]
        t = oracle_timing(xh, q, wl.eps, wl.metric, wl.k, cores, dequant=True)
        r["oracle"] = {"vectors_per_s_64_queries": wl.n * len(wl.eps) / t, "cores": cores,
                       "sample": "all rows quantized and dequantized at the three eps and "
                                 "searched by 64 of the 1,024 queries"}
    out[wl.name] = r
    # flat 2^26 values: Q_eps (AUTO and forced at the resolved width) and
    # the dequantisation round trip at three eps
    wl = W["flat_2p26"]
    r = measure_calls(lam, torch, dev, wl, {"quantize", "dequantize"}, reps)
    if with_oracle:
        xh = host_rows(wl)[: 1 << 24].reshape(-1, 1)
        t = oracle_timing(xh, None, wl.eps, 0, 0, cores, dequant=True, search=False)
        r["oracle"] = {"gbs_quantize_plus_dequantize": (1 << 24) * 4 * len(wl.eps) / t / 1e9,
                       "cores": cores, "sample": "2^24 of the 2^26 values at the three eps"}
    out[wl.name] = r
    # records: 361,802 rows, forced int16, B = 1 / 64 / 4,096, IP top-10
    wl = W["records_n361802_ip"]
    r = measure_calls(lam, torch, dev, wl, {"quantize", "dequantize", "score"}, reps)
    if with_oracle:
        xh = host_rows(wl)
        q = inputs.queries(64, wl.d, seed=1)
        t = oracle_timing(xh, q[:1], wl.eps, wl.metric, wl.k, cores)
        c, _, _ = oracle_quantize_rows(xh, wl.eps[0], cores)
        import oracle
        t0 = time.perf_counter()
        oracle.search(q, c, wl.eps[0], wl.metric, wl.k, nthreads=cores)
        t64 = time.perf_counter() - t0
        r["oracle"] = {"vectors_per_s_b1": wl.n / t, "search_vectors_per_s_b64": wl.n / t64,
                       "cores": cores,
                       "sample": "all rows quantized and searched by 1 query; the search of "
                                 "64 queries timed alone"}
    out[wl.name] = r
    # the headline memory at B = 256 (tensor cores), on its resident codes
    wl = mem.wl
    r = measure_calls(lam, torch, dev, wl, {"score"}, max(3, reps // 4), batches=[256],
                      width=1, codes_in=mem.codes)
    if with_oracle:
        q = inputs.queries(256, wl.d, seed=1)[:32]
        xs = mem.x[:ORACLE_ROWS].cpu().numpy()
        c, _, _ = oracle_quantize_rows(xs, wl.eps[0], cores)
        import oracle
        t0 = time.perf_counter()
        oracle.search(q, c, wl.eps[0], wl.metric, wl.k, nthreads=cores)
        t = time.perf_counter() - t0
        r["oracle"] = {"search_vectors_per_s_b32": ORACLE_ROWS / t, "cores": cores,
                       "sample": "search of 32 of the 256 queries over %d rows" % ORACLE_ROWS}
    out[wl.name + "_b256"] = r
    return out


def host_mem_bytes():
    """MemTotal of the host (bytes), 0 if it cannot be read."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemTotal:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def run_e2e(lam, torch, mem, wl, B, stream, dev, world, steps, ref_s, ref_i):
    """The headline step end to end from pinned host memory (see run_lam)."""
    x_h = torch.empty((wl.n, wl.d), dtype=torch.float32, pin_memory=True)
    x_h.copy_(mem.x)
    q_h = mem.q.cpu().pin_memory()
    s_h = torch.empty((B, wl.k), dtype=torch.float32, pin_memory=True)
    i_h = torch.empty((B, wl.k), dtype=torch.int64, pin_memory=True)
    cs = torch.cuda.Stream(dev)
    copied = [torch.cuda.Event() for _ in range(mem.n_slabs)]
    e2e_steps = max(3, min(steps, 10))

    def e2e_step():
        cs.wait_stream(stream)
        with torch.cuda.stream(cs):
            for j in range(mem.n_slabs):
                mem.slab(mem.x, j).copy_(mem.slab(x_h, j), non_blocking=True)
                copied[j].record(cs)
        mem.q.copy_(q_h, non_blocking=True)
        for j in range(mem.n_slabs):
            stream.wait_event(copied[j])
            lam.lam_quantize_async(mem.slab(mem.x, j), mem.eps, lam.LAM_I8,
                                   mem.slab(mem.codes, j), mem.qws[j])
        lam.lam_score_topk(mem.q, mem.codes, 1, mem.N, mem.D, mem.eps, mem.code_bound,
                           wl.k, wl.metric, mem.scores, mem.ids, mem.sws)
        s_h.copy_(mem.scores, non_blocking=True)
        i_h.copy_(mem.ids, non_blocking=True)

    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize(dev)
    barrier(world)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps + 1)]
    ev[0].record(stream)
    for i in range(e2e_steps):
        e2e_step()
        ev[i + 1].record(stream)
    torch.cuda.synchronize(dev)
    e2e_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(e2e_steps)]
    ms_e2e = max_over_ranks(ev[0].elapsed_time(ev[-1]) / e2e_steps, world, dev)
    mem.check()
    assert torch.equal(s_h, ref_s.cpu()) and torch.equal(i_h, ref_i.cpu())
    del x_h
    return {"value": wl.n * world / (ms_e2e / 1e3), "unit": UNIT,
            "ms_per_step": ms_e2e, "steps": e2e_steps,
            "ms_per_step_min_median_max": [min(e2e_ms), statistics.median(e2e_ms), max(e2e_ms)],
            "host_link_gbs_at_min": wl.n * wl.d * 4 / (min(e2e_ms) / 1e3) / 1e9,
            "h2d_bytes_per_step": wl.n * wl.d * 4 + B * wl.d * 4,
            "d2h_bytes_per_step": B * wl.k * (4 + 8),
            "note": "fp32 memory and query from pinned host memory, results back to pinned "
                    "host memory, inside the timed region; bound by the host link (~211 GB/s "
                    "for these copies alone on this box, with occasional slow copies from "
                    "the shared host)"}


def run_lam(args):
    import numpy as np
    import torch
    import paper_2609_32256_gb300 as lam
    from paper_2609_32256_gb300 import build as lam_build, inputs

    world, rank, local = dist_setup(args)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0 or world == 1:
        lam_build.build()
    barrier(world)
    lam.load()

    wl = inputs.WORKLOADS[HEADLINE]
    B = wl.batches[0]
    mem = MemStep(lam, torch, wl, B, dev)
    stream = torch.cuda.current_stream(dev)
    for _ in range(args.warmup):
        mem.step()
    torch.cuda.synchronize(dev)
    mem.check()
    # the device-resident step gives the synchronous calls' results
    ref_s, ref_i = mem.scores.clone(), mem.ids.clone()
    mem.step_host_sync()
    torch.cuda.synchronize(dev)
    assert torch.equal(ref_s, mem.scores) and torch.equal(ref_i, mem.ids)

    kinds = (lam.LAM_TIME_QUANTIZE | lam.LAM_TIME_DEQUANTIZE | lam.LAM_TIME_SCORE |
             lam.LAM_TIME_AUX | lam.LAM_TIME_MERGE)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    with sampler:
        barrier(world)
        torch.cuda.synchronize(dev)
        # timed region: K headline steps; the library brackets each launch of
        # its quantize and score kernels with CUDA events on the launching
        # stream and counts every launch
        lam.lam_timing_begin(lam.LAM_TIME_QUANTIZE | lam.LAM_TIME_SCORE,
                             args.steps * (mem.n_slabs + 2))
        e0.record(stream)
        for _ in range(args.steps):
            mem.step()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        barrier(world)
        kern = {}
        n_launch = 0
        for name, kind in (("quantize", lam.LAM_TIME_QUANTIZE), ("score", lam.LAM_TIME_SCORE),
                           ("merge", lam.LAM_TIME_MERGE), ("aux", lam.LAM_TIME_AUX),
                           ("dequantize", lam.LAM_TIME_DEQUANTIZE)):
            tot, timed, launches = lam.lam_timing_read(kind)
            n_launch += launches
            kern[name] = {"ms_total": tot, "timed": timed, "launches": launches,
                          "ms_per_launch": tot / timed if timed else None}
        lam.lam_timing_end()
        mem.check()
        ms_local = e0.elapsed_time(e1) / args.steps
        # the same step through the synchronous calls (one host read per slab)
        h0, h1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        h0.record(stream)
        for _ in range(args.steps):
            mem.step_host_sync()
        h1.record(stream)
        torch.cuda.synchronize(dev)
        ms_sync = h0.elapsed_time(h1) / args.steps

        # end to end: the fp32 memory and the query in pinned host memory; each
        # step copies every slab to the device (a copy stream, slab j + 1
        # overlapping the quantization of slab j), quantizes it, searches, and
        # reads the results back to pinned host memory.  Every rank pins its own
        # 25.8 GB copy: skipped when the ranks' copies would take more than half
        # of the host's memory (the same decision on every rank).
        e2e = None
        if world * wl.n * wl.d * 4 <= host_mem_bytes() // 2:
            e2e = run_e2e(lam, torch, mem, wl, B, stream, dev, world, args.steps, ref_s, ref_i)
        else:
            e2e = {"unavailable": "%d ranks' pinned copies of the 25.8 GB fp32 memory would "
                                  "exceed half of the host memory" % world}

        configs = None
        if rank == 0 and not args.no_configs:
            configs = other_configs(lam, torch, dev, mem, os.cpu_count() or 1,
                                    args.reps, with_oracle=not args.no_cpu_baseline)
    barrier(world)

    units_per_step = wl.n
    ms_step, value = aggregate_replicas(ms_local, units_per_step, world, dev)
    hbm_peak, tc_peak, peak_kind = load_peaks()
    nd_slab = mem.S * wl.d
    kq, ks = kern["quantize"], kern["score"]
    # algorithmic bytes per launch: Q_eps reads 4 B and writes 1 B per value of
    # its slab; the search reads 1 B per code (the 3 KB query is negligible)
    q_bytes = 5.0 * nd_slab
    s_bytes = 1.0 * wl.n * wl.d
    rl = {}
    for kname, k_, nbytes in (("quantize_forced_kernel", kq, q_bytes),
                              ("score_bw_kernel", ks, s_bytes)):
        ach = nbytes / (k_["ms_per_launch"] / 1e3) / 1e9
        tr, tr_note = traffic_for(kname)
        rl[kname] = {"bound": "hbm", "achieved": round(ach, 1), "peak": hbm_peak,
                     "unit": "GB/s", "frac": round(ach / hbm_peak, 4), "traffic": tr,
                     "kernel": kname, "ms_per_launch": k_["ms_per_launch"],
                     "launches": k_["timed"], "algorithmic_bytes_per_launch": nbytes,
                     "share_of_step": k_["ms_total"] / (ms_local * args.steps),
                     "peak_source": peak_kind + " copy (MEASURED_PEAKS.json hbm_gbs)"}
        if tr_note:
            rl[kname]["traffic_launch"] = tr_note
    dominant = max(rl, key=lambda n: rl[n]["share_of_step"])

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        xs = mem.x[:ORACLE_ROWS].cpu().numpy()
        cpu = cpu_baseline_mem(xs, mem.q.cpu().numpy(), wl, os.cpu_count() or 1)

    if rank == 0:
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "ms_per_step_host_sync": ms_sync,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32 -> int8 codes; int8 dot products (int32) + fp32 scores",
            "data": "synthetic (seeded unit-Gaussian rows shaped like bge-base D=768 "
                    "embeddings, drawn on the device per 1M-row slab)",
            "config": headline_config(wl, B),
            "step": "per slab lam_quantize_async (forced int8; the statuses are checked after "
                    "the timed steps) then one lam_score_topk (L2 top-100, bandwidth kernel) "
                    "over all 8,388,608 code rows, on one stream; ms_per_step_host_sync: the "
                    "same with the synchronous lam_quantize",
            "score_path": ["bandwidth", "tensor", "generic"][mem.path],
            "breakdown": {"kernels": kern,
                          "quantize_gbs_algorithmic": rl["quantize_forced_kernel"]["achieved"],
                          "score_gbs_algorithmic": rl["score_bw_kernel"]["achieved"],
                          "score_vectors_per_s_kernel": wl.n / (ks["ms_per_launch"] / 1e3)},
            "roofline": rl[dominant],
            "roofline_kernels": rl,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": n_launch,
            "gpu_launches_note": "library kernel launches inside the K timed steps, counted "
                                 "by the library (%d per step)" % (n_launch // args.steps),
            "clocks": sampler.summary("the timed steps, the host-synchronous pass, the e2e "
                                      "pass and the per-config measurements"),
            "configs": configs,
        }
        print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


# ----------------------------------------------------------- reference arm --

def run_reference(args):
    """The CPU oracle on the host cores, on the headline workload's metric and
    config: each step quantizes ORACLE_ROWS of the memory's rows to int8 and
    runs the L2 top-100 search over them; ms_per_step is the elapsed time of
    that work and `value` the rows it processed per second."""
    world, rank, _ = dist_setup(args)
    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    import oracle
    from paper_2609_32256_gb300 import inputs
    oracle.build()
    wl = inputs.WORKLOADS[HEADLINE]
    B = wl.batches[0]
    cores = os.cpu_count() or 1
    # the first rows of slab 0 (drawn on the host: the same distribution and
    # shape as the GPU arm's device-drawn rows)
    x = inputs.unit_rows(ORACLE_ROWS, wl.d, seed=SLAB_SEED)
    q = inputs.queries(B, wl.d, seed=1)
    eps = wl.eps[0]
    for _ in range(args.warmup):
        oracle_mem_step(x, q, eps, wl.metric, wl.k, cores)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_mem_step(x, q, eps, wl.metric, wl.k, cores)
    ms = (time.perf_counter() - t0) / args.steps * 1e3
    value = ORACLE_ROWS / (ms / 1e3)
    sample = ("per step the oracle quantizes %d of the memory's rows to int8 at eps=%g and runs "
              "the exact L2 top-%d search of the %d query over them, on %d threads (row chunks "
              "for Q_eps, rows split for the search); value = rows per second" %
              (ORACLE_ROWS, eps, wl.k, B, cores))
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "config": headline_config(wl, B),
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                            "sample": sample},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_kernels(args):
    """Per-call timing of one workload (json to stdout)."""
    import torch
    import paper_2609_32256_gb300 as lam
    from paper_2609_32256_gb300 import build as lam_build, inputs
    lam_build.build()
    lam.load()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = inputs.WORKLOADS[args.workload]
    if args.rows:
        import dataclasses
        wl = dataclasses.replace(wl, n=args.rows,
                                 slab_rows=min(wl.slab_rows, args.rows) if wl.slab_rows else 0)
    parts = set(args.only.split(",")) if args.only else {"quantize", "dequantize", "bands",
                                                         "codec", "admit", "score", "rows"}
    if "quantize" in parts:
        parts.add("dequantize")
    res = measure_calls(lam, torch, dev, wl, parts, args.reps,
                        batches=[args.batch] if args.batch else None,
                        eps_list=(args.eps,) if args.eps else None, width=args.width)
    print(json.dumps(res))


def main():
    args = parse()
    if args.kernels:
        run_kernels(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_lam(args)


if __name__ == "__main__":
    main()
