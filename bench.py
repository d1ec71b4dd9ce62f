#!/usr/bin/env python
"""Benchmark of the RSLM IVF-probe search path on GB300.

One step = the whole query path over one batch of synthetic queries with the
index resident in HBM: probe (<q, centroid> GEMM + top-nprobe), query
rotation, code scan with the norm-correction epilogue and per-query top-k,
and (for configurations with rescoring codes) rotation + rescoring.

Default workload: C4 -- N=1e7 d=128 log-normal-norm mixture, IVF8192,
4-bit codes (680 MB index, larger than the 129 MB L2, so no flush is
needed), 1e5 queries, nprobe=64, top-10.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config C4] [--nq n]
  python bench.py --impl reference ...   # the float64 CPU oracle arm

Under torchrun every rank builds its own replica of the index and searches
the full query batch (weak scaling, no data-path collective); rank 0 prints
one JSON line with the max-over-ranks time.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_30384_gb300 import workloads as W  # noqa: E402

METRIC = "candidates scored/s (IVF probe + RSLM code scan + top-k)"
UNIT = "candidates/s"
HBM_FALLBACK = 6800.0
TENSOR_FALLBACK = 1900.0  # burst dense bf16 TFLOP/s (fallback figure)
GEMV_QUERIES = 1024       # queries of the single-query-regime leg
BATCH_MIN_QUERIES = 16    # rslm_search's rule: batched scan when nq*nprobe >= 16*nlist
CLOCK_FIELDS = ["index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
                "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
                "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]
SCAN_SOURCES = {
    "scan_kernel": ["paper_2608_30384_gb300/csrc/search.cu", "paper_2608_30384_gb300/csrc/device_common.cuh"],
    "scan_bt_kernel": ["paper_2608_30384_gb300/csrc/search.cu", "paper_2608_30384_gb300/csrc/device_common.cuh",
                       "paper_2608_30384_gb300/csrc/tcgen05.cuh"],
    "batched_pipe_kernel": ["paper_2608_30384_gb300/csrc/batched.cu",
                            "paper_2608_30384_gb300/csrc/device_common.cuh",
                            "paper_2608_30384_gb300/csrc/tcgen05.cuh"],
    "batched_kpipe_kernel": ["paper_2608_30384_gb300/csrc/batched.cu",
                             "paper_2608_30384_gb300/csrc/device_common.cuh",
                             "paper_2608_30384_gb300/csrc/tcgen05.cuh"],
}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--config", default="C4", choices=sorted(W.WORKLOADS))
    ap.add_argument("--nq", type=int, default=None, help="override the query count")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="CPU time of the oracle leg")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-gemv", action="store_true",
                    help="skip the single-query-regime leg (first 1024 queries, HBM roofline of scan_kernel)")
    ap.add_argument("--scan", default="auto", choices=["auto", "gemv", "batched"],
                    help="scan form; auto = rslm_search's rule (batched when nq*nprobe >= 16*nlist)")
    ap.add_argument("--lite", action="store_true",
                    help="Rslm4Lite scoring codes (4-bit workloads, D >= 64): scales in the codes' top bits")
    ap.add_argument("--reading", default="B", choices=["A", "B"],
                    help="rescoring approximation: B the stage-1 reconstruction (default), A the centroid")
    ap.add_argument("--full-vector", action="store_true", help="codes of x itself (approximation 0)")
    ap.add_argument("--score-bits", type=int, default=None, choices=[1, 2, 3, 4],
                    help="override the workload's scoring bit rate (3: Rslm3)")
    ap.add_argument("--recall", type=int, default=0, metavar="N",
                    help="diagnostic: recall of the first N queries against exact float64 MIPS over "
                         "the whole database (computed while the index is built): Recall@k@k of the "
                         "final top-k, and Recall@20@20/30/40 from one untimed deeper search")
    args = ap.parse_args()
    if args.lite:
        w = W.WORKLOADS[args.config]
        if (args.score_bits or w.bits) != 4 or w.D < 64:
            ap.error("--lite needs a 4-bit workload with D >= 64")
    return args


def workload_label(w: W.Workload, lite: bool = False, reading: str = "B", full_vector: bool = False) -> str:
    base = W.WORKLOADS.get(w.name)
    mods = ([f"{w.bits}-bit scoring codes" + (" (Rslm3)" if w.bits == 3 else "")]
            if base is not None and w.bits != base.bits else []) \
        + (["Rslm4Lite scoring codes"] if lite else []) + (["full-vector codes"] if full_vector else []) \
        + (["rescoring reading A"] if reading == "A" and w.rescore_bits else [])
    desc = w.description
    if base is not None and w.bits != base.bits:
        # the workload's own text names its stock bit rate
        for tail in ("-bit codes", "-bit scoring"):
            desc = desc.replace(f"{base.bits}{tail}", f"{w.bits}{tail}")
    if mods:
        return f"{w.name} with {', '.join(mods)}: {desc}"
    return f"{w.name}: {desc}"


# ------------------------------------------------------------------ helpers
def load_peaks():
    """(HBM GB/s, burst dense bf16/fp16 TFLOP/s, 'measured' | 'fallback').

    The burst tensor figure applies: the dominant kernel runs a few
    milliseconds inside a step, not a seconds-long loop under the power cap.
    """
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    return HBM_FALLBACK, TENSOR_FALLBACK, "fallback"


def scan_source_hash(kernel: str) -> str:
    h = hashlib.sha256()
    for rel in SCAN_SOURCES[kernel]:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def traffic_record(config: str, kernel: str):
    """DRAM bytes per candidate of a scan kernel from a committed ncu summary.

    Returns None when no capture exists or the kernel changed since.
    """
    p = os.path.join(ROOT, "profiles", "scan_kernel_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    rec = d.get(f"{config}/{kernel}") or (d.get(config) if kernel == "scan_kernel" else None)
    if not rec or rec.get("kernel_hash") != scan_source_hash(kernel):
        return None
    return rec


def visible_gpu_index(local_rank: int) -> str:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        parts = [p.strip() for p in vis.split(",") if p.strip()]
        if local_rank < len(parts):
            return parts[local_rank]
    return str(local_rank)


class ClockSampler:
    """nvidia-smi clock / throttle samples every 200 ms during the timed region."""

    def __init__(self, gpu: str):
        self.gpu, self.proc, self.lines = gpu, None, []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + ",".join(CLOCK_FIELDS), "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", self.gpu], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < len(CLOCK_FIELDS):
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def max_over_ranks(x: float, ws: int, device=None) -> float:
    """The largest x over the ranks (the job's time is its slowest rank's)."""
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank_step: float, ws: int, steps: int, total_ms: float) -> float:
    """Whole-job units per second: every rank processes its units each step."""
    return units_per_rank_step * ws * steps / (total_ms / 1e3)


def dist_setup(args):
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws != args.gpus:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE={ws}")
    return ws, rank, local


# ------------------------------------------------------ recall diagnostic
class ExactTopK:
    """Exact maximum-inner-product top-k (float64, ties to the lower row id)
    of a few queries over database rows streamed in blocks."""

    def __init__(self, Q, k):
        self.Q = np.asarray(Q, dtype=np.float64)
        self.k = k
        self.sc = np.full((len(Q), 0), -np.inf)
        self.ids = np.zeros((len(Q), 0), dtype=np.int64)

    def add(self, X, lo):
        S = self.Q @ np.asarray(X, dtype=np.float64).T
        ids = np.broadcast_to(np.arange(lo, lo + X.shape[0]), S.shape)
        sc = np.concatenate([self.sc, S], axis=1)
        ii = np.concatenate([self.ids, ids], axis=1)
        keep = np.argpartition(-sc, min(self.k, sc.shape[1] - 1), axis=1)[:, :self.k + 1] \
            if sc.shape[1] > self.k + 1 else np.tile(np.arange(sc.shape[1]), (len(sc), 1))
        sc = np.take_along_axis(sc, keep, 1)
        ii = np.take_along_axis(ii, keep, 1)
        o = np.lexsort((ii, -sc), axis=1)[:, :self.k]
        self.sc = np.take_along_axis(sc, o, 1)
        self.ids = np.take_along_axis(ii, o, 1)

    def recall_at(self, found, x):
        """Recall@x@y (Sec. 4, quality metrics): the share of the exact top x
        among the y results returned per query (y = found's width)."""
        assert x <= self.k
        n = len(self.Q)
        return float(np.mean([len(set(found[i].tolist()) & set(self.ids[i, :x].tolist())) / x
                              for i in range(n)]))

    def recall(self, found, deep=None):
        """Recall@k@k and Recall@1@k of the final top k (found: [n, k]); with
        deep ([n, 40] results of a deeper search), Recall@20@20, @20@30 and
        @20@40 from its prefixes."""
        k = found.shape[1]
        out = {"queries": len(self.Q), "k": k, "recall_k_at_k": self.recall_at(found, k),
               "recall_1_at_k": self.recall_at(found, 1),
               "exact": "float64 maximum inner product over every database row"}
        if deep is not None:
            for y in (20, 30, 40):
                out[f"recall_20_at_{y}"] = self.recall_at(deep[:, :y], 20)
        return out


# --------------------------------------------------------- oracle (CPU) leg
def oracle_sample(w: W.Workload, A, C, Q, n_queries: int, lite: bool = False, reading: str = "B",
                  full_vector: bool = False):
    """Oracle index over the rows of the partitions the sample queries probe
    (those rows are regenerated from their seeds)."""
    from oracle import search as osearch
    probes, _, _ = osearch.probe(Q[:n_queries], C, w.nprobe)
    parts = np.unique(probes)
    rows = np.nonzero(np.isin(A, parts))[0]
    X, _ = W.rows(w, rows)
    index = osearch.build_index(X, rows, A[rows], C, w.bits, w.rescore_bits, lite=lite,
                                reading=reading if w.rescore_bits else "B", full_vector=full_vector)
    sizes = np.bincount(A, minlength=w.P)
    cand = int(sizes[probes].sum())
    return index, cand, len(rows)


def oracle_time(w, index, Q, n_queries, cand_per_pass, seconds, min_passes=1):
    from oracle import search as osearch
    t0 = time.perf_counter()
    passes = 0
    while passes < min_passes or time.perf_counter() - t0 < seconds:
        osearch.search(index, Q[:n_queries], w.nprobe, w.k, w.k_final)
        passes += 1
    dt = time.perf_counter() - t0
    return cand_per_pass * passes / dt, passes, dt


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


SAMPLE_QUERIES = {"C1": 100, "C2": 8, "C3": 4, "C4": 8, "C5": 1}


def run_reference(args):
    ws, rank, _ = dist_setup(args)
    if rank != 0:
        return 0
    w = W.WORKLOADS[args.config]
    if args.nq:
        w = w.scaled(nq=args.nq)
    if args.score_bits:
        w = w.scaled(bits=args.score_bits)
    A = W.assignment(w)
    C = W.ivf_centroids(w)
    nqs = min(SAMPLE_QUERIES[w.name], w.nq)
    Q = W.queries(w, nqs)
    index, cand, nrows = oracle_sample(w, A, C, Q, nqs, args.lite, args.reading, args.full_vector)
    for _ in range(args.warmup):
        oracle_time(w, index, Q, nqs, cand, 0.0)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_time(w, index, Q, nqs, cand, 0.0)
    dt = time.perf_counter() - t0
    value = cand * args.steps / dt
    sample = (f"{nqs} of the {w.nq} queries of {w.name} per step ({cand} candidates), float64 oracle "
              f"index over the {nrows} rows of their probed partitions")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": workload_label(w, args.lite, args.reading, args.full_vector), "nq_per_step": nqs},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------- GPU arm
def finalize_launches(desc: dict, lite: bool) -> int:
    """Finalize kernels of the batched regime: the hi-only mode (4-bit codes
    without the Rslm4Lite head; padded D <= 128 also needs one coordinate
    per code in 16-byte chunks) finalizes rows of at most 256 coordinates
    with one warp kernel and longer rows with a select kernel and a block
    kernel; the other formats take the warp kernel and its block fallback."""
    g, bits = desc["group"], desc["score_bits"]
    dp16 = (desc["padded_dim"] + 15) // 16 * 16
    stride = (desc["code_bytes"] + 3) // 4 * 4
    chunk = 16 if stride % 16 == 0 else 8 if stride % 8 == 0 else 4
    hi = bits != 3 and not lite and ((g == 1 and chunk == 16) if dp16 <= 128 else True)
    return 1 if hi and 2 * g * stride <= 256 else 2


def launches_per_step(w: W.Workload, nq: int, batched: bool, fin: int = 2) -> int:
    """Kernels of librslm launched by one step (fin: finalize kernels)."""
    if (w.D + 15) // 16 * 16 <= 128 and w.P >= 32 * w.nprobe and w.nprobe <= 256:
        n = 4                # fused probe: query operands, two-pass probe, list selection,
                             # exact fallback for overflowed lists
    else:
        ld = (w.P + 3) // 4 * 4
        qc = max(128, (64 << 20) // ld // 128 * 128)
        # probe GEMM, per query chunk: query operand blocks, the GEMM, the
        # warp-per-query selection and the block kernel for the rows it
        # hands over (nprobe <= 256)
        n = math.ceil(nq / qc) * (4 if w.nprobe <= 256 else 3)
    n += 1                   # query rotation
    # batched: two probe-list inversions (pair histograms, segment sums,
    # prefix, scatter, list scan, item table), query split, first-probe pass,
    # threshold, tensor-core scan, finalize, overflow re-scan; else one scan
    n += 12 + 1 + 1 + 1 + 1 + fin + 1 if batched else 1
    if w.rescore_bits:
        n += 2               # second rotation + rescore
    return n


def run_gpu(args):
    import torch
    import torch.distributed as dist

    from paper_2608_30384_gb300 import Index
    from paper_2608_30384_gb300 import binding as B

    ws, rank, local = dist_setup(args)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws > 1:
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl", device_id=dev)

    w = W.WORKLOADS[args.config]
    if args.nq:
        w = w.scaled(nq=args.nq)
    if args.score_bits:
        w = w.scaled(bits=args.score_bits)
    # the database is generated in 2^20-row blocks straight into the encoder,
    # so no configuration holds it in host memory
    A = W.assignment(w)
    C = W.ivf_centroids(w)
    Q = W.queries(w)
    nq = w.nq

    # index build (not timed as part of the step)
    ix = Index(torch.from_numpy(C).to(dev), w.bits, w.rescore_bits, lite=args.lite,
               reading=args.reading if w.rescore_bits else "B", full_vector=args.full_vector)
    ix.reserve(torch.from_numpy(A).to(dev))
    torch.cuda.synchronize()
    encode_s = 0.0
    exact = ExactTopK(Q[:args.recall], max(w.k_final, 20)) if args.recall else None
    for lo, X in W.row_blocks(w, 1 << 20):
        Xd = torch.from_numpy(X).to(dev)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        ix.encode(Xd, lo)
        ix.sync()
        encode_s += time.perf_counter() - t0
        del Xd
        if exact is not None:
            exact.add(X, lo)
    desc = ix.desc

    Qd = torch.from_numpy(Q).to(dev)
    probes = torch.empty((nq, w.nprobe), dtype=torch.int32, device=dev)
    cs = torch.empty((nq, w.nprobe), dtype=torch.float32, device=dev)
    qrot = torch.empty((nq, desc["padded_dim"]), dtype=torch.float32, device=dev)
    s1_ids = torch.empty((nq, w.k), dtype=torch.int64, device=dev)
    s1_sc = torch.empty((nq, w.k), dtype=torch.float32, device=dev)
    if w.rescore_bits:
        qrot2 = torch.empty((nq, desc["rescore_padded_dim"]), dtype=torch.float32, device=dev)
        f_ids = torch.empty((nq, w.k_final), dtype=torch.int64, device=dev)
        f_sc = torch.empty((nq, w.k_final), dtype=torch.float32, device=dev)
    h = ix.handle
    batched = (args.scan == "batched" or
               (args.scan == "auto" and nq * w.nprobe >= BATCH_MIN_QUERIES * w.P))
    scan_fn = B.rslm_scan_batched if batched else B.rslm_scan

    def step(ev=None):
        B.rslm_probe(h, Qd, w.nprobe, probes, cs)
        if ev is not None:
            ev[0].record()
        B.rslm_rotate_queries(h, 1, Qd, qrot)
        if ev is not None:
            ev[1].record()
        scan_fn(h, qrot, probes, cs, w.k, s1_ids, s1_sc)
        if ev is not None:
            ev[2].record()
        if w.rescore_bits:
            B.rslm_rotate_queries(h, 2, Qd, qrot2)
            B.rslm_rescore(h, qrot2, s1_ids, s1_sc, w.k_final, f_ids, f_sc)
        if ev is not None:
            ev[3].record()

    for _ in range(args.warmup):
        step()
    ix.sync()
    sizes = torch.bincount(torch.from_numpy(A).to(dev).long(), minlength=w.P)
    cand_per_step = int(sizes[probes.long()].sum().item())
    # codes + UE7M9 + UE4M12 scales (Rslm4Lite: the scales are inside the codes)
    bytes_per_cand = desc["code_bytes"] + (0 if args.lite else 4)

    E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    starts = [E() for _ in range(args.steps)]
    evs = [[E() for _ in range(4)] for _ in range(args.steps)]
    # an index that fits in L2 would be served from it by the next step:
    # overwrite a buffer larger than L2 between timed steps (not timed)
    small_index = scan_bytes_index(desc) + rescore_bytes_index(desc) < L2_BYTES
    flush = torch.empty(4 * L2_BYTES // 4, dtype=torch.float32, device=dev) if small_index else None
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler = ClockSampler(visible_gpu_index(local))
    sampler.start()
    time.sleep(0.3)
    B.rslm_profile_enable(h, True)
    for i in range(args.steps):
        if flush is not None:
            flush.fill_(float(i))
        starts[i].record()
        step(evs[i])
    torch.cuda.synchronize()
    clocks = sampler.stop()
    kern_ms, kern_n, kern_name = B.rslm_profile_read(h)
    B.rslm_profile_enable(h, False)
    if ws > 1:
        dist.barrier()
    step_ms = [starts[i].elapsed_time(evs[i][3]) for i in range(args.steps)]
    total_ms = sum(step_ms)
    probe_ms = sum(starts[i].elapsed_time(evs[i][0]) for i in range(args.steps)) / args.steps
    rot_ms = sum(evs[i][0].elapsed_time(evs[i][1]) for i in range(args.steps)) / args.steps
    scan_ms = sum(evs[i][1].elapsed_time(evs[i][2]) for i in range(args.steps)) / args.steps
    resc_ms = sum(evs[i][2].elapsed_time(evs[i][3]) for i in range(args.steps)) / args.steps
    ix.sync()
    total_ms = max_over_ranks(total_ms, ws, dev)
    ms_per_step = total_ms / args.steps
    value = job_throughput(cand_per_step, ws, args.steps, total_ms)

    hbm_peak, tensor_peak, peak_kind = load_peaks()

    # single-query (GEMV) regime: the first GEMV_QUERIES queries scanned by
    # scan_kernel, one CTA per query, no cross-query reuse inside the kernel;
    # judged by algorithmic code + scale bytes per kernel time against HBM
    gemv = None
    if rank == 0 and not args.no_gemv and scan_bytes_index(desc) >= L2_BYTES:
        ng = min(GEMV_QUERIES, nq)
        Qg = Qd[:ng].contiguous()
        pg = torch.empty((ng, w.nprobe), dtype=torch.int32, device=dev)
        cg = torch.empty((ng, w.nprobe), dtype=torch.float32, device=dev)
        qg = torch.empty((ng, desc["padded_dim"]), dtype=torch.float32, device=dev)
        g_ids = torch.empty((ng, w.k), dtype=torch.int64, device=dev)
        g_sc = torch.empty((ng, w.k), dtype=torch.float32, device=dev)
        B.rslm_probe(h, Qg, w.nprobe, pg, cg)
        B.rslm_rotate_queries(h, 1, Qg, qg)
        cand_g = int(sizes[pg.long()].sum().item())
        gflush = torch.empty(4 * L2_BYTES // 4, dtype=torch.float32, device=dev)
        for _ in range(3):
            B.rslm_scan(h, qg, pg, cg, w.k, g_ids, g_sc)
        torch.cuda.synchronize()
        gs = ClockSampler(visible_gpu_index(local))
        gs.start()
        time.sleep(0.3)
        B.rslm_profile_enable(h, True)
        for i in range(args.steps):
            gflush.fill_(float(i))  # L2 flushed between launches (not in the kernel's time)
            B.rslm_scan(h, qg, pg, cg, w.k, g_ids, g_sc)
        torch.cuda.synchronize()
        gclocks = gs.stop()
        g_ms, g_n, g_name = B.rslm_profile_read(h)
        B.rslm_profile_enable(h, False)
        ix.sync()
        del gflush
        g_avg = g_ms / max(1, g_n) / 1e3
        g_bytes = cand_g * bytes_per_cand
        g_ach = g_bytes / g_avg / 1e9
        g_trec = traffic_record(w.name + ("-lite" if args.lite else "") + "-gemv", g_name) \
            if not args.score_bits else None
        gemv = {"workload": f"first {ng} queries of {w.name}, single-query scan (no cross-query reuse)",
                "kernel": g_name, "bound": "hbm", "achieved": g_ach, "peak": hbm_peak, "unit": "GB/s",
                "frac": g_ach / hbm_peak, "peak_kind": peak_kind,
                "algorithmic_bytes": g_bytes, "bytes_per_candidate": bytes_per_cand, "candidates": cand_g,
                "candidates_per_s": cand_g / g_avg, "kernel_ms": g_avg * 1e3, "launches": g_n,
                "traffic": (g_trec["dram_bytes_per_candidate"] * cand_g) if g_trec else None,
                "l2": "flushed between launches", "clocks": gclocks}

    # end to end through the public one-call API with host buffers
    e2e = None
    if not args.no_e2e:
        Qh = torch.from_numpy(Q).pin_memory()
        Qd2 = torch.empty_like(Qd)
        o_ids = torch.empty((nq, w.k_final), dtype=torch.int64, device=dev)
        o_sc = torch.empty((nq, w.k_final), dtype=torch.float32, device=dev)
        h_ids = torch.empty((nq, w.k_final), dtype=torch.int64).pin_memory()
        h_sc = torch.empty((nq, w.k_final), dtype=torch.float32).pin_memory()

        def e2e_step():
            Qd2.copy_(Qh, non_blocking=True)
            B.rslm_search(h, Qd2, w.nprobe, w.k, bool(w.rescore_bits), w.k_final, o_ids, o_sc)
            h_ids.copy_(o_ids, non_blocking=True)
            h_sc.copy_(o_sc, non_blocking=True)

        for _ in range(max(1, min(args.warmup, 2))):
            e2e_step()
        torch.cuda.synchronize()
        a, b = E(), E()
        if ws > 1:
            dist.barrier()
        a.record()
        for _ in range(args.steps):
            e2e_step()
        b.record()
        torch.cuda.synchronize()
        ems = max_over_ranks(a.elapsed_time(b), ws, dev)
        ix.sync()
        e2e = {"value": job_throughput(cand_per_step, ws, args.steps, ems), "unit": UNIT,
               "h2d_bytes_per_step": int(Qh.numel() * 4),
               "d2h_bytes_per_step": int(h_ids.numel() * 8 + h_sc.numel() * 4),
               "ms_per_step": ems / args.steps}

    # recall diagnostic (untimed): the final top-k of the timed steps, and
    # one deeper search (40 results) of the same queries for Recall@20@y
    recall = None
    if exact is not None:
        n = args.recall
        final = (f_ids if w.rescore_bits else s1_ids)[:n].cpu().numpy()
        deep_ids, _ = ix.search(Qd[:n].contiguous(), w.nprobe, max(w.k, 40), k_final=40)
        ix.sync()
        recall = exact.recall(final, deep_ids.cpu().numpy())

    scan_bytes = cand_per_step * bytes_per_cand
    kern_avg_s = kern_ms / max(1, kern_n) / 1e3
    bits_tag = f"-{w.bits}bit" if args.score_bits and args.score_bits != W.WORKLOADS[w.name].bits else ""
    trec = traffic_record(w.name + bits_tag + ("-lite" if args.lite else ""), kern_name)
    traffic = (trec["dram_bytes_per_candidate"] * cand_per_step) if trec else None
    if kern_name.startswith("batched_"):
        # dense contraction: 2 D flops per candidate (the fp16 hi/lo split is
        # counted once); one launch scores the whole step's candidates
        flops = 2.0 * w.D * cand_per_step
        achieved = flops / kern_avg_s / 1e12
        roofline = {"bound": "tensor", "kernel": kern_name, "achieved": achieved,
                    "peak": tensor_peak, "unit": "TFLOP/s", "frac": achieved / tensor_peak,
                    "peak_kind": f"{peak_kind} burst dense bf16 (fp16 runs at the same rate; the kernel "
                                 f"runs a few ms inside the step)",
                    "traffic": traffic, "algorithmic_flops": flops,
                    "kernel_ms": kern_avg_s * 1e3, "launches": kern_n}
    else:
        achieved = scan_bytes / kern_avg_s / 1e9
        roofline = {"bound": "hbm", "kernel": kern_name, "achieved": achieved, "peak": hbm_peak,
                    "unit": "GB/s", "frac": achieved / hbm_peak, "peak_kind": peak_kind,
                    "traffic": traffic, "algorithmic_bytes": scan_bytes,
                    "kernel_ms": kern_avg_s * 1e3, "launches": kern_n}

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        nqs = min(SAMPLE_QUERIES[w.name], nq)
        index, cand, nrows = oracle_sample(w, A, C, Q, nqs, args.lite, args.reading, args.full_vector)
        cval, passes, dt = oracle_time(w, index, Q, nqs, cand, args.cpu_seconds)
        cpu = {"value": cval, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "sample": f"{nqs} of the {nq} queries of {w.name} ({cand} candidates per pass) x {passes} "
                         f"passes = {dt:.1f} s, float64 oracle index over the {nrows} rows of their "
                         f"probed partitions"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": workload_label(w, args.lite, args.reading, args.full_vector), "nq": nq, "nprobe": w.nprobe, "k": w.k,
                       "k_final": w.k_final, "score_bits": w.bits, "rescore_bits": w.rescore_bits,
                       "l2": (f"L2 flushed between timed steps (a {4 * L2_BYTES / 1e6:.0f} MB buffer "
                              f"overwritten, not timed): the {(scan_bytes_index(desc) + rescore_bytes_index(desc)) / 1e6:.0f}"
                              f" MB index fits in the 129 MB L2") if small_index else
                             (f"inputs larger than L2: {scan_bytes_index(desc) / 1e6:.0f} MB of codes "
                              f"and scales vs 129 MB L2"),
                       "parallelism": f"replica x{ws}",
                       "scan": "batched (partition-major, tensor cores)" if batched else
                               "single-query (shared-memory table)"},
            "qps": nq * ws / (ms_per_step / 1e3),
            "latency_ms": {"p50": float(np.percentile(step_ms, 50)), "p99": float(np.percentile(step_ms, 99)),
                           "steps": len(step_ms)},
            "logical_code_gbps": {
                "value": scan_bytes * ws / (ms_per_step / 1e3) / 1e9,
                "note": "codes + scales of every scored candidate per step time; a logical figure: in "
                        "the batched regime each partition's codes are read once per tile of up to 128 "
                        "of its queries and reused by all of them, so it exceeds the HBM bandwidth"},
            "stage_ms": {"probe": probe_ms, "rotate": rot_ms, "scan": scan_ms, "rescore": resc_ms},
            "candidates_per_step": cand_per_step,
            "encode_rows_per_s": w.N / encode_s,
            "roofline": roofline,
            "gemv": gemv,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": launches_per_step(w, nq, batched, finalize_launches(desc, args.lite)) * args.steps,
            "clocks": clocks,
            "recall": recall,
            # index event counters over the whole run (warm-up and timed
            # steps): queries answered by the exact re-scan fallback
            "events": ix.counters(),
        }
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.destroy_process_group()
    return 0


L2_BYTES = 129 * 1000 * 1000


def scan_bytes_index(desc) -> int:
    return int(desc["n_slots"]) * (int(desc["code_bytes"]) + 4)


def rescore_bytes_index(desc) -> int:
    return int(desc["n_slots"]) * (int(desc.get("rescore_code_bytes", 0)) + 4) if desc.get("rescore_bits") else 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
