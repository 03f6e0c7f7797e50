"""Benchmark of LAM's quantized-memory hot path on GB300.

One step is one pass of the whole path over one batch: for each eps of the
sweep, Q_eps at the narrowest width, dequantisation of the codes (round
trip), and exact top-k search of the query batch on the codes (fused
dequant + score + top-k, then the merge of partial lists).  All of it runs
through the C ABI on device-resident inputs; the value is memory vectors per
second through the whole path.  The headline pass drives the calls the way a
user would: Q_eps (synchronous, the width comes back) on one stream and the
dequantisation and search of that eps on a second, so the search of one eps
overlaps the quantization of the next; a second pass runs every call in
order on one stream for per-stage spans and per-kernel times.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...   # the CPU oracle, timed on host cores

With --gpus N > 1 (launched by torchrun) every rank runs an independent
replica of the workload on its own GPU; there is no exchange between ranks.
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

METRIC = "Q_ε GB/s and fused score+top-k memory vectors/s at D=768; % of HBM roofline"
UNIT = "memory vectors/s"
L2_FLUSH_BYTES = 512 << 20


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

# DRAM bytes (read + write) of one launch of the dominant kernel, from one ncu
# capture (the profiles/ summary of that kernel).  Reported only while the
# kernel's source file is the one the counters were taken on.
KERNEL_TRAFFIC = {
    "score_tc2_kernel": {"source": "score_tc.cu", "source_sha256_16": "343e9d742c33392e",
                         "bytes": 46567168,
                         "launch": "ncu, cold caches: int16 codes at eps=1e-4 (the fp16 operand "
                                   "image is the same for every width), 27,986 x 768, "
                                   "1,024 queries"},
}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=1000)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="lam", choices=["lam", "reference"])
    p.add_argument("--workload", default="chunks_n27986_ip")
    p.add_argument("--batch", type=int, default=0, help="query batch (default: workload's first)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--kernels", action="store_true",
                   help="time each C-ABI call of --workload separately (not the headline step)")
    p.add_argument("--reps", type=int, default=20)
    p.add_argument("--eps", type=float, default=0.0, help="(--kernels) one eps instead of the sweep")
    p.add_argument("--width", type=int, default=-1, help="(--kernels) forced code width")
    p.add_argument("--rows", type=int, default=0,
                   help="(--kernels) a smaller memory of the same workload (profiling captures)")
    p.add_argument("--no-graph", action="store_true",
                   help="time the device-resident step eagerly instead of replaying its CUDA graph")
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
    """nvidia-smi clock / throttle-reason samples during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = os.path.join(ROOT, "gpurun_out", "clocks_bench_rank%d.csv" % index)

    def __enter__(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None:
            return None
        rows = []
        try:
            for line in open(self.path):
                f = [x.strip() for x in line.split(",")]
                if len(f) >= 9:
                    rows.append(f)
        except Exception:
            return None
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[j] for r in rows for j in range(4) if r[5 + j] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


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


# ----------------------------------------------------------------- lam arm --

class Pipeline:
    """Buffers and calls of one step, all through the C ABI."""

    def __init__(self, lam, torch, x, q, eps_list, k, metric, dev):
        self.lam, self.torch = lam, torch
        self.x, self.q = x, q
        self.eps_list, self.k, self.metric = eps_list, k, metric
        self.N, self.D = x.shape
        self.B = q.shape[0]
        self.dev = dev
        n = x.numel()
        # one code buffer per eps (fits any width), so that the quantization of
        # the next eps can run while the previous one is being searched
        self.codes_e = [torch.empty(n * 4, dtype=torch.uint8, device=dev) for _ in eps_list]
        self.codes = self.codes_e[0]
        self.deq = torch.empty_like(x)
        self.sq = torch.cuda.Stream(dev)  # quantize stream
        self.sd = torch.cuda.Stream(dev)  # dequantize stream
        self.ss = torch.cuda.Stream(dev)  # score stream
        self.qdone = [torch.cuda.Event() for _ in eps_list]
        self.qws = torch.zeros(64, dtype=torch.uint8, device=dev)
        self.scores = [torch.empty((self.B, k), dtype=torch.float32, device=dev) for _ in eps_list]
        self.ids = [torch.empty((self.B, k), dtype=torch.int64, device=dev) for _ in eps_list]
        # widths and code bounds from a first (untimed) quantization
        self.plan = []
        wsz = 0
        for e in eps_list:
            st, w, s, cmin, cmax = lam.lam_quantize(x, e, 0, None, self.qws)
            bound = max(-cmin, cmax)
            wsz = max(wsz, lam.lam_score_topk_workspace_size(self.B, self.N, self.D, k, w, bound))
            self.plan.append((w, bound, lam.lam_score_topk_path(self.B, self.N, self.D, k, w, bound)))
        self.sws = torch.empty(wsz, dtype=torch.uint8, device=dev)
        # a second search stream (and workspace): the short kernels of one
        # search overlap the scoring kernel of the next
        self.ss2 = torch.cuda.Stream(dev)
        self.sws2 = torch.empty(wsz, dtype=torch.uint8, device=dev)
        # device-resident pipeline: one quantize status per eps, read by the
        # dequantisation and the search on the device
        self.qws_e = [torch.zeros(256, dtype=torch.uint8, device=dev) for _ in eps_list]
        fsz = lam.lam_score_topk_from_workspace_size(self.B, self.N, self.D, k)
        self.swsf = [torch.empty(fsz, dtype=torch.uint8, device=dev) for _ in range(2)]

    def step_device(self):
        """The step with no host round trip: each eps is quantized on one
        stream (lam_quantize_async), its dequantisation and search take the
        width from the quantize status on the device (lam_dequantize_from,
        lam_score_topk_from) on streams of their own; the same work and
        results as step()."""
        lam = self.lam
        n = self.x.numel()
        for j, e in enumerate(self.eps_list):
            lam.lam_quantize_async(self.x, e, 0, self.codes_e[j], self.qws_e[j],
                                   stream=self.sq.cuda_stream)
            self.qdone[j].record(self.sq)
            ss, sws = (self.ss, self.swsf[0]) if j % 2 == 0 else (self.ss2, self.swsf[1])
            self.sd.wait_event(self.qdone[j])
            ss.wait_event(self.qdone[j])
            lam.lam_dequantize_from(self.codes_e[j], self.qws_e[j], n, e, self.deq,
                                    stream=self.sd.cuda_stream)
            lam.lam_score_topk_from(self.q, self.codes_e[j], self.qws_e[j], self.N, self.D, e,
                                    self.k, self.metric, self.scores[j], self.ids[j], sws,
                                    stream=ss.cuda_stream)
        self.ss.wait_stream(self.sd)  # the step ends when all have finished
        self.ss.wait_stream(self.ss2)

    def step_overlapped(self):
        """The step as a user would drive it: Q_eps of each eps on one stream
        (synchronous: the width comes back to the host); the dequantisation
        and the search of that eps, which only read its codes, each on a
        stream of their own, so they overlap one another and the quantization
        of the next eps.  The same calls and work as step()."""
        lam = self.lam
        n = self.x.numel()
        for j, e in enumerate(self.eps_list):
            st, w, s, cmin, cmax = lam.lam_quantize(self.x, e, 0, self.codes_e[j], self.qws,
                                                    stream=self.sq.cuda_stream)
            self.qdone[j].record(self.sq)
            ss, sws = (self.ss, self.sws) if j % 2 == 0 else (self.ss2, self.sws2)
            self.sd.wait_event(self.qdone[j])
            ss.wait_event(self.qdone[j])
            lam.lam_dequantize(self.codes_e[j], w, n, s, self.deq, stream=self.sd.cuda_stream)
            lam.lam_score_topk(self.q, self.codes_e[j], w, self.N, self.D, e, max(-cmin, cmax),
                               self.k, self.metric, self.scores[j], self.ids[j], sws,
                               stream=ss.cuda_stream)
        self.ss.wait_stream(self.sd)  # the step ends when all have finished
        self.ss.wait_stream(self.ss2)

    def step(self, ev=None):
        """The step with every call in order on the current stream (per-stage
        spans when `ev` is given)."""
        lam = self.lam
        for j, e in enumerate(self.eps_list):
            if ev is not None:
                ev[j][0].record()
            st, w, s, cmin, cmax = lam.lam_quantize(self.x, e, 0, self.codes, self.qws)
            if ev is not None:
                ev[j][1].record()
            lam.lam_dequantize(self.codes, w, self.x.numel(), s, self.deq)
            if ev is not None:
                ev[j][2].record()
            lam.lam_score_topk(self.q, self.codes, w, self.N, self.D, e, max(-cmin, cmax), self.k,
                               self.metric, self.scores[j], self.ids[j], self.sws)
            if ev is not None:
                ev[j][3].record()


def cpu_baseline_lam_units(x_np, q_np, eps_list, k, metric, cores, budget_q=64):
    """Times the oracle on host cores on a bounded sample; returns a dict."""
    import numpy as np
    import oracle
    N, D = x_np.shape
    B = q_np.shape[0]
    b = min(B, budget_q)
    t_total = 0.0
    for e in eps_list:
        t0 = time.perf_counter()
        oc, *_ = oracle.quantize(x_np, e)
        t1 = time.perf_counter()
        oracle.dequantize(oc, oracle.step(e))
        t2 = time.perf_counter()
        oracle.search(q_np[:b], oc.reshape(N, D), e, metric, k, nthreads=cores)
        t3 = time.perf_counter()
        t_total += (t1 - t0) + (t2 - t1) + (t3 - t2) * (B / b)
    units = N * len(eps_list)
    return {"value": units / t_total, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "quantize + dequantize of all %dx%d values per eps and exact search of "
                      "%d of the %d queries (search time scaled to %d), eps %s" %
                      (N, D, b, B, B, list(eps_list))}


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

    wl = inputs.WORKLOADS[args.workload]
    B = args.batch or wl.batches[0]
    if wl.planted:
        x_np = inputs.planted_rows(wl.n, wl.d, seed=0)
    else:
        x_np = inputs.unit_rows(wl.n, wl.d, seed=0)
    q_np = inputs.queries(B, wl.d, seed=1)
    x = torch.from_numpy(x_np).to(dev)
    q = torch.from_numpy(q_np).to(dev)
    pipe = Pipeline(lam, torch, x, q, wl.eps, wl.k, wl.metric, dev)
    flush = L2Flush(torch, dev)
    stream = torch.cuda.current_stream(dev)

    cur = torch.cuda.current_stream(dev)

    graph = None  # the device-resident step captured once, replayed per step

    def overlapped_step(i, e0, e1, device=True, use_graph=False):
        # the previous step is finished and L2 is flushed before the step starts
        pipe.sq.wait_stream(pipe.ss)
        pipe.sq.wait_stream(pipe.ss2)
        pipe.sq.wait_stream(pipe.sd)
        pipe.sq.wait_stream(cur)
        with torch.cuda.stream(pipe.sq):
            flush(i)
        e0.record(pipe.sq)
        if use_graph:
            with torch.cuda.stream(pipe.sq):
                graph.replay()
            e1.record(pipe.sq)
            return
        if device:
            pipe.step_device()
        else:
            pipe.step_overlapped()
        e1.record(pipe.ss)

    for i in range(args.warmup):
        flush(i)
        pipe.step()
        overlapped_step(i, torch.cuda.Event(enable_timing=True),
                        torch.cuda.Event(enable_timing=True))
        overlapped_step(i, torch.cuda.Event(enable_timing=True),
                        torch.cuda.Event(enable_timing=True), device=False)
    torch.cuda.synchronize(dev)
    if not args.no_graph:
        # capture the device-resident step (its four streams fork from and
        # join the capture stream); every replay runs all of its launches
        gs = torch.cuda.Stream(dev)
        gs.wait_stream(cur)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=gs):
            for st_ in (pipe.sq, pipe.sd, pipe.ss, pipe.ss2):
                st_.wait_stream(gs)
            pipe.step_device()
            for st_ in (pipe.sq, pipe.sd, pipe.ss, pipe.ss2):
                gs.wait_stream(st_)
        torch.cuda.synchronize(dev)
        for i in range(args.warmup):
            overlapped_step(i, torch.cuda.Event(enable_timing=True),
                            torch.cuda.Event(enable_timing=True), use_graph=True)
        torch.cuda.synchronize(dev)
    # launches of one device-resident step (the graph replays the same ones),
    # counted by the library over one eager step
    all_kinds = (lam.LAM_TIME_QUANTIZE | lam.LAM_TIME_DEQUANTIZE | lam.LAM_TIME_SCORE |
                 lam.LAM_TIME_AUX | lam.LAM_TIME_MERGE)
    lam.lam_timing_begin(all_kinds, 1024)
    pipe.step_device()
    torch.cuda.synchronize(dev)
    launches_per_step = sum(lam.lam_timing_read(kd)[2] for kd in
                            (lam.LAM_TIME_QUANTIZE, lam.LAM_TIME_DEQUANTIZE, lam.LAM_TIME_SCORE,
                             lam.LAM_TIME_AUX, lam.LAM_TIME_MERGE))
    lam.lam_timing_end()
    # the device-resident step gives the synchronous calls' results
    overlapped_step(0, torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
                    use_graph=graph is not None)
    torch.cuda.synchronize(dev)
    dev_res = [(s_.clone(), i_.clone()) for s_, i_ in zip(pipe.scores, pipe.ids)]
    pipe.step()
    torch.cuda.synchronize(dev)
    for (s_d, i_d), s_, i_ in zip(dev_res, pipe.scores, pipe.ids):
        assert torch.equal(s_d, s_) and torch.equal(i_d, i_)

    ne = len(wl.eps)
    step_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
    evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(ne)]
           for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize(dev)
    sync_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
    eager_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(args.steps)]
    sampler = ClockSampler(local)
    with sampler:
        # headline pass: the step as a throughput user drives it, queued with
        # no host round trip (the width stays on the device), replayed from
        # its CUDA graph
        for i in range(args.steps):
            overlapped_step(i, *step_ev[i], use_graph=graph is not None)
        torch.cuda.synchronize(dev)
        # the same calls launched one by one
        for i in range(args.steps):
            overlapped_step(i, *eager_ev[i])
        torch.cuda.synchronize(dev)
        # the same step through the synchronous lam_quantize (the host reads
        # each width back before it launches that eps's search)
        for i in range(args.steps):
            overlapped_step(i, *sync_ev[i], device=False)
        torch.cuda.synchronize(dev)
        # Second pass, every call in order on one stream: per-stage spans and,
        # from the library, CUDA events around each launch of its quantize,
        # dequantize and score kernels (kept out of the first pass: the
        # host-side records would widen it) and a count of every launch.
        timed_kinds = {"quantize": lam.LAM_TIME_QUANTIZE,
                       "dequantize": lam.LAM_TIME_DEQUANTIZE, "score": lam.LAM_TIME_SCORE}
        lam.lam_timing_begin(lam.LAM_TIME_QUANTIZE | lam.LAM_TIME_DEQUANTIZE |
                             lam.LAM_TIME_SCORE, min(args.steps * len(wl.eps) * 8, 1 << 20))
        for i in range(args.steps):
            flush(i)  # L2 flush between timed steps (outside the events)
            pipe.step(evs[i])
        torch.cuda.synchronize(dev)
    barrier(world)
    kern = {}
    n_launch = 0
    for name, kind in list(timed_kinds.items()) + [("aux", lam.LAM_TIME_AUX)]:
        tot, timed, launches = lam.lam_timing_read(kind)
        n_launch += launches
        if name != "aux":
            kern[name] = {"ms_total": tot, "timed": timed, "launches": launches,
                          "ms_per_launch": tot / timed if timed else None}
    lam.lam_timing_end()

    t_q = t_d = t_s = 0.0
    for i in range(args.steps):
        for j in range(ne):
            e = evs[i][j]
            t_q += e[0].elapsed_time(e[1])
            t_d += e[1].elapsed_time(e[2])
            t_s += e[2].elapsed_time(e[3])
    units_per_step = wl.n * ne
    ms_local = sum(a.elapsed_time(b) for a, b in step_ev) / args.steps
    ms_sync = sum(a.elapsed_time(b) for a, b in sync_ev) / args.steps
    ms_eager = sum(a.elapsed_time(b) for a, b in eager_ev) / args.steps
    ms_step, value = aggregate_replicas(ms_local, units_per_step, world, dev)
    ms_serial = (t_q + t_d + t_s) / args.steps

    # per-stage figures (rank-local)
    nd = wl.n * wl.d
    widths = [w for (w, _, _) in pipe.plan]
    q_bytes = sum((4 + w) * nd for w in widths)       # one quantize pass at the resolved width
    d_bytes = sum((w + 4) * nd for w in widths)
    flops = 2.0 * wl.n * wl.d * B * ne
    ms_q, ms_d, ms_s = t_q / args.steps, t_d / args.steps, t_s / args.steps
    hbm_peak, tc_peak, peak_kind = load_peaks()
    path_names = {0: "bandwidth", 1: "tensor", 2: "generic"}
    paths = [path_names[p] for (_, _, p) in pipe.plan]
    sk = kern["score"]
    if all(p == "tensor" for p in paths):
        kname = "score_tc2_kernel" if B > 128 else "score_tc_kernel"
        # algorithmic work of the score kernel: 2 N D B flops per eps (one
        # launch per row slab; the hi/lo query split doubles the MMA issue)
        achieved = flops * args.steps / (sk["ms_total"] / 1e3) / 1e12
        roofline = {"bound": "tensor", "achieved": round(achieved, 2), "peak": tc_peak,
                    "unit": "TFLOP/s", "frac": round(achieved / tc_peak, 4),
                    "kernel": kname, "ms_per_launch": sk["ms_per_launch"],
                    "launches": sk["timed"],
                    "peak_source": peak_kind + " bf16 dense burst (fp16 has the same nominal "
                                   "rate)"}
    else:
        kname = "score_bw_kernel" if all(p == "bandwidth" for p in paths) else "score"
        sb = sum(w * nd for w in widths)  # the codes, read once per eps
        achieved = sb * args.steps / (sk["ms_total"] / 1e3) / 1e9
        roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm_peak,
                    "unit": "GB/s", "frac": round(achieved / hbm_peak, 4), "kernel": kname,
                    "ms_per_launch": sk["ms_per_launch"], "launches": sk["timed"],
                    "peak_source": peak_kind + " copy"}
    roofline["traffic"] = None
    tr = KERNEL_TRAFFIC.get(kname)
    if tr and tr["bytes"]:
        try:
            import hashlib
            with open(os.path.join(ROOT, "paper_2609_32256_gb300", "csrc", tr["source"]),
                      "rb") as f:
                if hashlib.sha256(f.read()).hexdigest()[:16] == tr["source_sha256_16"]:
                    roofline["traffic"] = tr["bytes"]
                    roofline["traffic_launch"] = tr["launch"]
        except OSError:
            pass

    # end to end: host (pinned) inputs, copies inside the timed region
    x_h = x.cpu().pin_memory()
    q_h = q.cpu().pin_memory()
    res_h = [(torch.empty((B, wl.k), dtype=torch.float32).pin_memory(),
              torch.empty((B, wl.k), dtype=torch.int64).pin_memory()) for _ in wl.eps]
    e2e_steps = max(3, min(args.steps, 50))
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    tot = 0.0
    for i in range(e2e_steps + 2):
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(pipe.sq):
            flush(i)
            e0.record(pipe.sq)
            x.copy_(x_h, non_blocking=True)
        pipe.ss.wait_event(e0)
        with torch.cuda.stream(pipe.ss):
            q.copy_(q_h, non_blocking=True)  # ordered before the searches on this stream
        pipe.ss2.wait_stream(pipe.ss)         # and on the other search stream
        pipe.step_device()
        with torch.cuda.stream(pipe.ss):
            for j in range(ne):
                res_h[j][0].copy_(pipe.scores[j], non_blocking=True)
                res_h[j][1].copy_(pipe.ids[j], non_blocking=True)
            e1.record(pipe.ss)
        torch.cuda.synchronize(dev)
        if i >= 2:
            tot += e0.elapsed_time(e1)
    ms_e2e = max_over_ranks(tot / e2e_steps, world, dev)
    e2e = {"value": units_per_step * world / (ms_e2e / 1e3), "unit": UNIT,
           "h2d_bytes_per_step": x_h.numel() * 4 + q_h.numel() * 4,
           "d2h_bytes_per_step": ne * B * wl.k * (4 + 8)}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cores = os.cpu_count() or 1
        cpu = cpu_baseline_lam_units(x_np, q_np, wl.eps, wl.k, wl.metric, cores)

    if rank == 0:
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "ms_per_step_serial": ms_serial,
            "ms_per_step_eager": ms_eager,
            "ms_per_step_host_sync": ms_sync,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32 in, int%d codes, fp16x2-split tensor / fp32 accumulate" % (8 * max(widths)),
            "data": "synthetic (seeded unit-Gaussian rows shaped like bge-base D=768 embeddings)",
            "config": {"workload": wl.name, "N": wl.n, "D": wl.d, "batch": B, "k": wl.k,
                       "metric": ["ip", "cosine", "l2"][wl.metric], "eps": list(wl.eps),
                       "widths": widths, "paths": paths, "parallelism": "replicas only",
                       "l2": "flushed between timed steps (512 MB write then 512 MB read, outside "
                             "the events)",
                       "step": "per eps: lam_quantize_async (AUTO width) on one stream, "
                               "lam_dequantize_from on a second and lam_score_topk_from on a "
                               "third or fourth (alternating), the width read from the quantize "
                               "status on the device, so nothing waits for the host; the step "
                               "is captured once in a CUDA graph and replayed (ms_per_step_eager: "
                               "the same calls launched one by one; ms_per_step_host_sync: with "
                               "the synchronous lam_quantize / lam_dequantize / lam_score_topk; "
                               "ms_per_step_serial: those all on one stream)",
                       "graph": graph is not None},
            "breakdown": {
                "quantize_ms": ms_q, "quantize_gbs_algorithmic": q_bytes / (ms_q / 1e3) / 1e9,
                "quantize_note": "lam_quantize span: status clear + quantize + status read-back",
                "dequantize_ms": ms_d, "dequantize_gbs": d_bytes / (ms_d / 1e3) / 1e9,
                "score_ms": ms_s, "score_vectors_per_s": wl.n * ne / (ms_s / 1e3),
                "score_tflops": flops / (ms_s / 1e3) / 1e12,
                "kernels": {
                    "quantize": dict(kern["quantize"], gbs_algorithmic=(
                        q_bytes / (kern["quantize"]["ms_total"] / args.steps / 1e3) / 1e9
                        if kern["quantize"]["ms_total"] else None)),
                    "dequantize": dict(kern["dequantize"], gbs_algorithmic=(
                        d_bytes / (kern["dequantize"]["ms_total"] / args.steps / 1e3) / 1e9
                        if kern["dequantize"]["ms_total"] else None)),
                    "score": kern["score"]}},
            "roofline": roofline,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches_per_step * args.steps,
            "gpu_launches_note": "kernel launches of the library in the K headline steps: %d per "
                                 "step, counted by the library over one eagerly launched step "
                                 "(the graph replays the same launches); the per-kernel pass of "
                                 "the synchronous calls launched %d" % (launches_per_step,
                                                                         n_launch),
            "clocks": sampler.summary(),
        }
        print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


# ----------------------------------------------------------- reference arm --

def run_reference(args):
    """The CPU oracle on the host cores, same metric, bounded sample per step."""
    world, rank, _ = dist_setup(args)
    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    import numpy as np
    import oracle
    from paper_2609_32256_gb300 import inputs
    oracle.build()
    wl = inputs.WORKLOADS[args.workload]
    B = args.batch or wl.batches[0]
    x_np = inputs.planted_rows(wl.n, wl.d, seed=0) if wl.planted else inputs.unit_rows(wl.n, wl.d, seed=0)
    q_np = inputs.queries(B, wl.d, seed=1)
    cores = os.cpu_count() or 1
    S, b = 2048, 4  # rows and queries per step
    ne = len(wl.eps)

    def one(i):
        e = wl.eps[i % ne]
        r0 = (i * S) % max(1, wl.n - S)
        xs = x_np[r0:r0 + S]
        t0 = time.perf_counter()
        oc, *_ = oracle.quantize(xs, e)
        oracle.dequantize(oc, oracle.step(e))
        t1 = time.perf_counter()
        oracle.search(q_np[:b], oc.reshape(xs.shape), e, wl.metric, wl.k, nthreads=cores)
        t2 = time.perf_counter()
        return (t1 - t0) + (t2 - t1) * (B / b)

    for i in range(args.warmup):
        one(i)
    tot = sum(one(i) for i in range(args.steps))
    ms = tot / args.steps * 1e3
    value = S / (ms / 1e3)
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "config": {"workload": wl.name, "N": wl.n, "D": wl.d, "batch": B,
                                           "k": wl.k, "eps": list(wl.eps)},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                            "sample": "per step %d rows quantized, dequantized and searched by "
                                      "%d queries (search time scaled to %d queries), eps rotating"
                                      % (S, b, B)},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_kernels(args):
    """Per-call timing of one workload: Q_eps (AUTO and at the resolved width),
    dequantisation and lam_score_topk per query batch, each as the mean of
    --reps CUDA-event spans with a 512 MB L2 flush before every rep."""
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
    parts = set(args.only.split(",")) if args.only else {"quantize", "bands", "codec", "admit",
                                                         "score", "rows"}
    if wl.d == 1:
        x = torch.from_numpy(inputs.flat_values(wl.n, seed=0)).to(dev)
    elif wl.slab_rows:
        x = inputs.unit_rows_device(wl.n, wl.d, seed=0, device=dev)
    elif wl.planted:
        x = torch.from_numpy(inputs.planted_rows(wl.n, wl.d, seed=0)).to(dev)
    else:
        x = torch.from_numpy(inputs.unit_rows(wl.n, wl.d, seed=0)).to(dev)
    n = x.numel()
    flush = L2Flush(torch, dev)
    ws = torch.zeros(64, dtype=torch.uint8, device=dev)
    codes = torch.empty(n * 4, dtype=torch.uint8, device=dev)
    out = torch.empty(n, dtype=torch.float32, device=dev)

    def timed(fn, kind):
        """(mean call span ms, mean device ms of the call's `kind` kernel launches)."""
        for i in range(3):
            flush(i)
            fn()
        tot = 0.0
        lam.lam_timing_begin(kind, args.reps * 64)
        for i in range(args.reps):
            flush(i)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize(dev)
            tot += e0.elapsed_time(e1)
        k_ms, _, _ = lam.lam_timing_read(kind)
        lam.lam_timing_end()
        return tot / args.reps, k_ms / args.reps

    res = {"workload": wl.name, "n_values": n, "quantize": [], "dequantize": [], "score": []}
    hbm, tc_peak, kind = load_peaks()
    widths = {}
    eps_list = (args.eps,) if args.eps else wl.eps
    for e in eps_list:
        _, w, sc, cmin, cmax = lam.lam_quantize(x, e, 0, None, ws)
        wq = args.width if args.width > 0 else (wl.width or w)
        widths[e] = (wq, sc, max(-cmin, cmax))
        if "quantize" not in parts:
            continue
        ms_auto, k_auto = timed(lambda: lam.lam_quantize(x, e, 0, codes, ws),
                                lam.LAM_TIME_QUANTIZE)
        ms_forced, k_forced = timed(lambda: lam.lam_quantize(x, e, wq, codes, ws),
                                    lam.LAM_TIME_QUANTIZE)
        qb = (4 + wq) * n
        qa = (4 + w) * n  # AUTO writes the resolved width
        res["quantize"].append({"eps": e, "width": wq, "width_auto": w, "ms_auto_span": ms_auto,
                                "ms_auto_kernel": k_auto, "ms_forced_span": ms_forced,
                                "ms_forced_kernel": k_forced,
                                "gbs_auto_kernel": qa / (k_auto / 1e3) / 1e9,
                                "frac_of_hbm_auto_kernel": qa / (k_auto / 1e3) / 1e9 / hbm,
                                "gbs_forced_kernel": qb / (k_forced / 1e3) / 1e9,
                                "frac_of_hbm_forced_kernel": qb / (k_forced / 1e3) / 1e9 / hbm})
        lam.lam_quantize(x, e, wq, codes, ws)
        ms_d, k_d = timed(lambda: lam.lam_dequantize(codes, wq, n, sc, out),
                          lam.LAM_TIME_DEQUANTIZE)
        gbd = (wq + 4) * n / (k_d / 1e3) / 1e9
        res["dequantize"].append({"eps": e, "width": wq, "ms_span": ms_d, "ms_kernel": k_d,
                                  "gbs_kernel": gbd, "frac_of_hbm_kernel": gbd / hbm})
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
        lam.lam_quantize(x, e, wq, codes, ws)
        N = wl.n
        batches = [args.batch] if args.batch else list(wl.batches)
        for B in batches:
            q = torch.from_numpy(inputs.queries(B, wl.d, seed=1)).to(dev)
            nb = lam.lam_score_topk_workspace_size(B, N, wl.d, wl.k, wq, bound)
            sws = torch.empty(nb, dtype=torch.uint8, device=dev)
            s_ = torch.empty((B, wl.k), dtype=torch.float32, device=dev)
            i_ = torch.empty((B, wl.k), dtype=torch.int64, device=dev)
            path = lam.lam_score_topk_path(B, N, wl.d, wl.k, wq, bound)
            ms, k_s = timed(lambda: lam.lam_score_topk(q, codes, wq, N, wl.d, e, bound, wl.k,
                                                       wl.metric, s_, i_, sws),
                            lam.LAM_TIME_SCORE)
            _, k_m = timed(lambda: lam.lam_score_topk(q, codes, wq, N, wl.d, e, bound, wl.k,
                                                      wl.metric, s_, i_, sws),
                           lam.LAM_TIME_MERGE)
            _, k_a = timed(lambda: lam.lam_score_topk(q, codes, wq, N, wl.d, e, bound, wl.k,
                                                      wl.metric, s_, i_, sws),
                           lam.LAM_TIME_AUX)
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
    if wl.batches and wl.d > 1 and "rows" in parts:
        # the per-vector byte codecs of the composite experiment: encode, and
        # exact search over the coded rows (decoding folded into the score)
        res["rows"] = []
        N, D = wl.n, wl.d
        xr = x.view(N, D)
        batches = [args.batch] if args.batch else list(wl.batches)
        names = {lam.LAM_ROWS_INT8: "int8/vector", lam.LAM_ROWS_FP16: "fp16",
                 lam.LAM_ROWS_SIGN: "sign"}
        row_bytes = {lam.LAM_ROWS_INT8: D + 8, lam.LAM_ROWS_FP16: 2 * D,
                     lam.LAM_ROWS_SIGN: D // 8 + 4}
        for fmt in (lam.LAM_ROWS_INT8, lam.LAM_ROWS_FP16, lam.LAM_ROWS_SIGN):
            rc, rs, ro = lam.encode_rows(xr, fmt)
            ms_e, k_e = timed(lambda: lam.lam_encode_rows(xr, fmt, rc, rs, ro),
                              lam.LAM_TIME_QUANTIZE)
            eb = N * (4 * D + row_bytes[fmt])
            for B in batches:
                q = torch.from_numpy(inputs.queries(B, D, seed=1)).to(dev)
                nb = lam.lam_score_topk_rows_workspace_size(B, N, D, wl.k, fmt)
                sws = torch.empty(nb, dtype=torch.uint8, device=dev)
                s_ = torch.empty((B, wl.k), dtype=torch.float32, device=dev)
                i_ = torch.empty((B, wl.k), dtype=torch.int64, device=dev)
                path = lam.lam_score_topk_rows_path(B, N, D, wl.k, fmt)
                call = lambda: lam.lam_score_topk_rows(q, rc, fmt, rs, ro, N, D, wl.k, wl.metric,
                                                       s_, i_, sws)
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
                                    "tflops_kernel": fl / (k_s / 1e3) / 1e12,
                                    "frac_of_tensor_kernel": fl / (k_s / 1e3) / 1e12 / tc_peak})
                del sws
            del rc, rs, ro
    res["peaks"] = {"hbm_gbs": hbm, "bf16_tflops": tc_peak, "kind": kind}
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
