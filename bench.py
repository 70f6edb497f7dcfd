#!/usr/bin/env python
"""Benchmark of the TurboQuant search path on GB300 (one JSON line on stdout).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--config scale|c2|tiny|filtered|sweep|idmap|prof] [--batches 1,1024] [--k 5]

Workload (default "scale"): N = 999,000 synthetic L2-normalised d = 1536
vectors (1,024-cluster Gaussian mixture, seed 42), rotated by a seeded Haar R
and encoded to 4-bit codes (767.2 MB packed) on the GPU; 10,000
perturbed-corpus queries; top-5 by inner product.  A step is one search of a
batch of B queries through tq_search: query rotation, the scan with fused
top-k, and the merge (Sec. II-B step 5).  Inputs are resident in HBM when the
timed region starts; the 767 MB corpus is larger than the 129 MB L2, so every
step streams it from HBM.  The headline `value` is queries/s at the first batch
size; every batch size measured is reported under "batches".

The default run also measures, compactly under "extra", the 100K workload
(batch 1 and 256, top-5 and top-10, encode), the filtered workload on that
corpus (Zipf tenants, T = 10/100/1000, with the over-fetch post-filter
baseline) and the bit-width sweep on the 999K corpus (b = 2/3/4/8, batch 256,
encode), each with its roofline (--no-extras skips them).

--impl reference times the CPU oracle (float64 numpy) on the host cores on a
bounded sample of the same workload.

Under torchrun (N > 1 ranks, one GPU each) the corpus is N x 999,000 rows, one
999,000-row shard per rank (rows [r N0, (r+1) N0) of the same seeded
generator), and the queries of rank 0 are broadcast once.  A step is then the
sharded search: tq_search on the rank's shard, an all-gather of every rank's
top-k (the exchange step), and tq_merge_topk.  Work per GPU is fixed (weak
scaling); `value` counts query x shard scans per second, summed over ranks.
The timed region is bracketed by barriers and the slowest rank's time is used.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

CONFIGS = {
    # name: corpus size, dim, bits, clusters, query pool, k, batch sizes
    "scale": dict(n=999_000, d=1536, bits=4, clusters=1024, pool=10_000, k=5, batches=[1, 1024]),
    "c2": dict(n=100_000, d=1536, bits=4, clusters=256, pool=1_000, k=10, batches=[1, 256]),
    "tiny": dict(n=10_000, d=1536, bits=4, clusters=64, pool=100, k=10, batches=[1, 100]),
    # profiling case: codes (192 MB) larger than L2, a few GB on the device at most
    "prof": dict(n=250_000, d=1536, bits=4, clusters=256, pool=2_048, k=5, batches=[1, 1024]),
    # filtered search: Zipf(1.1) tenants, allowlist of one tenant (10% of the
    # queries five), 64-vector filter blocks
    "filtered": dict(n=100_000, d=1536, bits=4, clusters=256, pool=1_000, k=10, batches=[1],
                     tenants=[10, 100, 1000], block=64),
    # id-mapped index: external ids, 1% of the rows deleted; same searches
    # with and without the id map
    "idmap": dict(n=999_000, d=1536, bits=4, clusters=1024, pool=2_048, k=5, batches=[1, 1024],
                  deleted_frac=0.01),
    # bit-width sweep: encode and batch-256 top-10 search at b = 2, 3, 4, 8
    "sweep": dict(n=999_000, d=1536, bits=4, clusters=1024, pool=2_000, k=10, batches=[256],
                  sweep_bits=[2, 3, 4, 8]),
}

RECALL_Q = 200       # queries whose Recall@k against exact kNN the bench reports
MMA_MIN_BATCH = 16  # tq_search's AUTO switch to the tensor-core scan (k <= 64)

METRIC = "queries/sec at 999Kx1536 4-bit top-5 (batch 1 / 1024); % of HBM / TC roofline"


# ------------------------------------------------------------------ helpers --
def log(*a):
    print(*a, file=sys.stderr, flush=True)


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p["bf16_tflops_sustained"]), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def source_hash(*files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def lookup_kernel(bits: int, n: int, d: int, k: int) -> str:
    """The lookup scan tq_search's AUTO path runs below the tensor-core batch
    size: the bulk-copy ring for 3-bit codes, else the register-fed byte-pair
    (4-bit) or per-code scan."""
    return "k_scan_ring" if bits == 3 else "k_scan_stream"


def recorded_traffic(kernel_file, profile_md: str, scale_to: int):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on
    the current kernel source (the summary records the source hash).  The
    summary is captured on a smaller corpus of `captured_n` vectors; traffic
    grows with the corpus, so it is scaled to `scale_to` vectors."""
    path = os.path.join(ROOT, "profiles", profile_md)
    if not os.path.exists(path):
        return None
    want = source_hash(*((kernel_file,) if isinstance(kernel_file, str) else kernel_file))
    got_hash, traffic, cap_n = None, None, None
    with open(path) as f:
        for line in f:
            if line.startswith("source_sha256_16:"):
                got_hash = line.split(":", 1)[1].strip()
            if line.startswith("dram_bytes_per_launch:"):
                traffic = float(line.split(":", 1)[1].strip())
            if line.startswith("captured_n:"):
                cap_n = int(line.split(":", 1)[1].strip())
    if got_hash != want or traffic is None or not cap_n:
        return None
    return traffic * scale_to / cap_n


class ClockSampler:
    """Samples SM clock and clock-event reasons during the timed region, via
    NVML (read-only queries), else `nvidia-smi -lms`."""

    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
               0x2: "applications_clocks_setting"}

    def __init__(self, pci_bus_id: str | None, index: int):
        self.samples, self.reasons, self.max_mhz = [], set(), None
        self._stop = threading.Event()
        self._nvml = None
        self._dev = ctypes.c_void_p()
        self._index = index
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                raise OSError("nvmlInit")
            ok = -1
            if pci_bus_id:
                ok = nv.nvmlDeviceGetHandleByPciBusId_v2(pci_bus_id.encode(), ctypes.byref(self._dev))
            if ok != 0:
                ok = nv.nvmlDeviceGetHandleByIndex_v2(index, ctypes.byref(self._dev))
            if ok != 0:
                raise OSError("nvml handle")
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(self._dev, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = mx.value
            self._nvml = nv
        except OSError:
            self._nvml = None

    def _loop_nvml(self):
        nv = self._nvml
        mhz = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        getr = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            nv.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if nv.nvmlDeviceGetClockInfo(self._dev, 1, ctypes.byref(mhz)) == 0:
                self.samples.append(mhz.value)
            if getr(self._dev, ctypes.byref(rs)) == 0:
                for bit, name in self.REASONS.items():
                    if rs.value & bit:
                        self.reasons.add(name)
            time.sleep(0.002)

    def _loop_smi(self):
        cmd = ["nvidia-smi", "-i", str(self._index), "--query-gpu=clocks.sm,clocks.max.sm,"
               "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
               "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
               "--format=csv,noheader,nounits", "-lms", "200"]
        try:
            self._proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, text=True)
        except OSError:
            return
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self._proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            try:
                self.samples.append(int(parts[0]))
                self.max_mhz = int(parts[1])
                for nm, v in zip(names, parts[2:]):
                    if v.lower().startswith("active"):
                        self.reasons.add(nm)
            except (ValueError, IndexError):
                pass
            if self._stop.is_set():
                break

    def __enter__(self):
        self._t = threading.Thread(target=self._loop_nvml if self._nvml else self._loop_smi, daemon=True)
        self._t.start()
        return self

    def __exit__(self, *exc):
        self._stop.set()
        if getattr(self, "_proc", None) is not None:
            self._proc.terminate()
        self._t.join(timeout=2)

    def summary(self):
        return {"sm_mhz": statistics.median(self.samples) if self.samples else None,
                "sm_max_mhz": self.max_mhz, "reasons": sorted(self.reasons),
                "samples": len(self.samples), "source": "nvml" if self._nvml else "nvidia-smi"}


# --------------------------------------------------------------- workloads --
def make_corpus(cfg, workers, shard=0):
    """Rows [shard n, (shard+1) n) of the seeded mixture corpus and the query
    pool drawn from them (shard 0 is the single-GPU workload)."""
    from paper_2607_16973_gb300 import synth
    t0 = time.time()
    n = cfg["n"]
    X = synth.mixture_rows(shard * n, (shard + 1) * n, cfg["d"], cfg["clusters"], workers=workers)
    src = synth.query_sources(n, cfg["pool"])
    Q = synth.perturb(X[src])
    log(f"[bench] generated corpus shard {shard} {X.shape} + {len(Q)} queries in {time.time() - t0:.1f}s")
    return X, Q


def cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count() or 1


def oracle_qps_sample(cfg, sample_rows: int, n_queries: int, seconds_cap: float = 30.0):
    """Times the oracle's search of single queries over a bounded sample of
    the corpus rows (encoded by the oracle itself) and scales to the full
    corpus.  Returns (qps_full, info)."""
    import oracle as O
    from paper_2607_16973_gb300 import synth
    d, bits, k = cfg["d"], cfg["bits"], cfg["k"]
    X = synth.mixture_rows(0, sample_rows, d, cfg["clusters"], workers=8)
    R = O.rotation(d, synth.SEED_ROTATION).astype(np.float32)
    cb = O.codebook(d, bits)
    enc = O.encode(X, R, cb.centroids32, cb.boundaries32, bits)
    Q = synth.perturb(X[synth.query_sources(sample_rows, n_queries)])
    times = []
    t_start = time.time()
    for q in range(n_queries):
        t0 = time.perf_counter()
        O.search(Q[q:q + 1], R, cb.centroids32, bits, enc.packed, enc.scale, k, d)
        times.append(time.perf_counter() - t0)
        if time.time() - t_start > seconds_cap:
            break
    per_q_sample = statistics.median(times)
    per_q_full = per_q_sample * cfg["n"] / sample_rows
    return 1.0 / per_q_full, {
        "sample": f"oracle search (float64 numpy) of {len(times)} single queries over the first "
                  f"{sample_rows} of {cfg['n']} corpus rows, median time scaled by {cfg['n']}/{sample_rows}",
        "per_query_s_sample": per_q_sample}


def arm_config(args, n, d, bits, k, batch, world):
    """The `config` object of the JSON line, the same for both arms."""
    return {"workload": f"{args.config}: N={n} d={d} {bits}-bit top-{k}, batch {batch}, "
                        f"codes {n * d * bits // 8 / 1e6:.1f} MB resident in HBM",
            "n": n, "d": d, "bits": bits, "k": k, "batch": batch,
            "l2": "inputs larger than L2 (corpus streamed from HBM every step)",
            "parallelism": "single GPU" if world == 1 else
            f"corpus sharded by rows over {world} GPUs ({n} rows each), all-gather of top-k + merge"}


# -------------------------------------------------------------- reference --
def run_reference(args, cfg, rank, world):
    if world > 1 and rank != 0:
        return
    import oracle as O
    from paper_2607_16973_gb300 import synth
    d, bits, k = cfg["d"], cfg["bits"], cfg["k"]
    sample_rows = min(cfg["n"], args.ref_sample)
    X = synth.mixture_rows(0, sample_rows, d, cfg["clusters"], workers=8)
    R = O.rotation(d, synth.SEED_ROTATION).astype(np.float32)
    cb = O.codebook(d, bits)
    enc = O.encode(X, R, cb.centroids32, cb.boundaries32, bits)
    Q = synth.perturb(X[synth.query_sources(sample_rows, max(args.steps + args.warmup, 1))])
    B = 1
    for i in range(args.warmup):
        O.search(Q[i:i + 1], R, cb.centroids32, bits, enc.packed, enc.scale, k, d)
    t0 = time.perf_counter()
    for i in range(args.steps):
        j = args.warmup + i
        O.search(Q[j:j + 1], R, cb.centroids32, bits, enc.packed, enc.scale, k, d)
    el = time.perf_counter() - t0
    scale_up = cfg["n"] / sample_rows
    per_step = el / max(args.steps, 1)          # measured: one query over the sample rows
    per_step_full = per_step * scale_up
    qps = B / per_step_full
    cores = cpu_threads()
    line = {
        "impl": "reference", "metric": METRIC, "value": qps, "unit": "queries/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_step * 1e3,
        "extrapolated_from": {"rows_per_step": sample_rows, "corpus_rows": cfg["n"], "factor": scale_up,
                              "ms_per_full_query": per_step_full * 1e3},
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": arm_config(args, cfg["n"], d, bits, k, B, world),
        "cpu_baseline": {"value": qps, "unit": "queries/s", "cores": cores, "kind": "oracle", **cpu_model(),
                         "sample": f"each step: oracle search of 1 query over the first {sample_rows} "
                                   f"rows, time scaled by {cfg['n']}/{sample_rows}"},
        "e2e": {"value": qps, "unit": "queries/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------- ours ----
def run_ours(args, cfg, rank, world):
    import torch
    import paper_2607_16973_gb300 as tq
    from paper_2607_16973_gb300 import shard, synth
    from paper_2607_16973_gb300.build import build

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
    build()
    tq.load()
    d, bits, k, n = cfg["d"], cfg["bits"], cfg["k"], cfg["n"]
    batches = [int(b) for b in args.batches.split(",")] if args.batches else cfg["batches"]
    if args.k:
        k = args.k
    if args.bits:
        bits = args.bits
    stream = torch.cuda.Stream(device=dev)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    # ---- index build: codebook + rotation on the host, encode on the GPU
    X, Qpool = make_corpus(cfg, workers=min(16, os.cpu_count() or 4), shard=rank)
    if world > 1:  # every rank searches rank 0's queries
        qb = torch.from_numpy(Qpool).to(dev)
        dist.broadcast(qb, src=0)
        Qpool = qb.cpu().numpy()
        del qb
    cen, bnd, _ = tq.codebook(d, bits)
    R = tq.rotation(d, synth.SEED_ROTATION)
    with torch.cuda.stream(stream):
        Xd = torch.from_numpy(X).to(dev, non_blocking=False)
        Rd = torch.from_numpy(R).to(dev)
        cd = torch.from_numpy(cen).to(dev)
        bd = torch.from_numpy(bnd).to(dev)
        codes = torch.empty((n, d * bits // 8), dtype=torch.uint8, device=dev)
        scale = torch.empty(n, dtype=torch.float32, device=dev)
        Qd = torch.from_numpy(Qpool).to(dev)
        plan = tq.encode_plan(Rd, stream=stream)  # the index's split of R (built once, like R itself)
    del X
    barrier()

    def enc_time(**kw):
        ts = []
        for i in range(3):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            tq.encode(Xd, Rd, cd, bd, bits, "norm", codes, scale, stream=stream, **kw)
            e1.record(stream)
            e1.synchronize()
            ts.append(e0.elapsed_time(e1))
        return min(ts[1:])
    ffma_ms = enc_time()             # the FFMA encoder, for comparison
    enc_ms = enc_time(plan=plan)     # the tensor-core encoder: the codes the searches use
    tq.encode_check(plan, stream=stream)
    # ground truth for Recall@k: exact float32 inner products of the first
    # RECALL_Q queries with the unquantised normalised corpus (torch matmul,
    # outside the timed regions; TF32 off)
    torch.backends.cuda.matmul.allow_tf32 = False
    nrec = min(RECALL_Q, len(Qpool))
    with torch.cuda.stream(stream):
        exact = torch.empty((nrec, k), dtype=torch.int64, device=dev)
        best = torch.full((nrec, k), float("-inf"), device=dev)
        for r0 in range(0, n, 1 << 18):
            sc = Qd[:nrec] @ Xd[r0:r0 + (1 << 18)].T
            v, i = torch.topk(torch.cat([best, sc], dim=1), k, dim=1)
            idx = torch.cat([exact, torch.arange(r0, r0 + sc.shape[1], device=dev).expand(nrec, -1)], dim=1)
            exact, best = torch.gather(idx, 1, i), v
    stream.synchronize()
    run_extras = world == 1 and args.config == "scale" and not args.no_extras
    if not run_extras:
        del Xd
    torch.cuda.empty_cache()
    log(f"[bench] encode {n} vectors: {enc_ms:.1f} ms ({n / enc_ms * 1e3:.3g} vec/s; FFMA encoder "
        f"{ffma_ms:.1f} ms)")

    pk = peaks()
    pci = None
    try:
        pr = torch.cuda.get_device_properties(dev)
        pci = f"{pr.pci_domain_id:08X}:{pr.pci_bus_id:02X}:{pr.pci_device_id:02X}.0"
    except Exception:
        pci = None
    results = {}
    tq.set_search_path(args.search_path)  # the timed batches' scans (AUTO unless asked)
    for B in batches:
        nbatches = max(1, len(Qpool) // B)
        ws = torch.empty(tq.search_workspace(B, n, d, bits, k), dtype=torch.uint8, device=dev)
        ids = torch.empty((B, k), dtype=torch.int64, device=dev)
        scs = torch.empty((B, k), dtype=torch.float32, device=dev)
        gids = torch.empty((B, k), dtype=torch.int64, device=dev)
        gscs = torch.empty((B, k), dtype=torch.float32, device=dev)

        def exchange():
            # the sharded search's exchange step: all-gather of every rank's
            # top-k (global ids) and the exact merge, queued on `stream`
            with torch.cuda.stream(stream):
                ci, cs = shard.gather_topk(ids, scs, rank * n)
                tq.merge_topk(ci, cs, k, out_ids=gids, out_scores=gscs, stream=stream)

        def step(i):
            j = (i % nbatches) * B
            tq.search(Qd[j:j + B], Rd, cd, bits, codes, scale, k, workspace=ws, out_ids=ids,
                      out_scores=scs, stream=stream)
            if world > 1:
                exchange()

        for i in range(args.warmup):
            step(i)
        # the timed region: back-to-back steps on `stream`, as a serving loop
        # runs them (the lookup scan overlaps the rotation's tail there)
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier()
        with ClockSampler(pci, local) as clk:
            t0.record(stream)
            for i in range(args.steps):
                step(args.warmup + i)
            t1.record(stream)
            t1.synchronize()
        barrier()
        ms = t0.elapsed_time(t1)
        if world > 1:
            tt = torch.tensor([ms], device=dev)
            dist.all_reduce(tt, op=dist.ReduceOp.MAX)
            ms = float(tt.item())
        # the scan kernel's duration: the same steps again, with the library
        # recording CUDA events on `stream` around each scan launch
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        for i in range(args.steps):
            tq.profile_events(*evs[i])
            step(args.warmup + i)
        tq.profile_events(None, None)
        stream.synchronize()
        scan_ms = statistics.mean(a.elapsed_time(b) for a, b in evs)
        qps = B * args.steps * world / (ms / 1e3)
        alg_bytes = n * (d * bits // 8 + 4)
        mma = bits in (2, 4, 8, 3) and k <= 64 and (args.search_path == "mma" or
                                                    (args.search_path == "auto" and B >= MMA_MIN_BATCH))
        if mma:
            # tensor-core scan: 2*n*d*B flops per launch against the dense fp16/bf16
            # peak (same rate); each launch is a few ms, timed alone: the burst figure
            flops = 2.0 * n * d * B
            achieved = flops / (scan_ms / 1e3) / 1e12
            peak = pk["bf16_tflops"]
            roof = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                    "frac": achieved / peak, "frac_of": pk["source"] + " burst bf16 (= fp16 dense rate)",
                    "frac_of_sustained": achieved / pk["bf16_tflops_sustained"],
                    "traffic": recorded_traffic("paper_2607_16973_gb300/csrc/tq_mma.cu", "k_scan_mma_250k_batch1024.md",
                                                scale_to=n),
                    "kernel": "k_scan_mma", "alg_flops_per_launch": flops, "kernel_ms": scan_ms,
                    "hbm_gbs_of_corpus": alg_bytes / (scan_ms / 1e3) / 1e9}
        else:
            # lookup scan (with its last CTA's merge): the corpus, codes + scales,
            # read once per launch
            achieved = alg_bytes / (scan_ms / 1e3) / 1e9
            kern = "k_scan_fold" if args.search_path == "lut_fold" else lookup_kernel(bits, n, d, k)
            if kern == "k_scan_fold":
                traffic = recorded_traffic(("paper_2607_16973_gb300/csrc/tq_fold.cu",
                                            "paper_2607_16973_gb300/csrc/tq_topk.cuh"), "k_scan_fold_250k_batch1.md",
                                           scale_to=n)
            elif kern == "k_scan_stream" and bits == 4 and args.search_path == "auto":
                traffic = recorded_traffic(("paper_2607_16973_gb300/csrc/tq_scan.cu",
                                            "paper_2607_16973_gb300/csrc/tq_topk.cuh"), "k_scan_stream_250k_batch1.md",
                                           scale_to=n)
            else:
                traffic = None
            roof = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                    "frac": achieved / pk["hbm_gbs"], "frac_of": pk["source"], "traffic": traffic,
                    "kernel": kern, "alg_bytes_per_launch": alg_bytes,
                    "kernel_ms": scan_ms, "frac_of_8tbs_nominal": achieved / 8000.0}
        # e2e through the C ABI with host buffers: tq_search_host queues the
        # query upload, the search and the result download on `stream`
        qh = torch.empty((B, d), dtype=torch.float32).pin_memory()
        qh.copy_(torch.from_numpy(Qpool[:B]))
        ih = torch.empty((B, k), dtype=torch.int64).pin_memory()
        sh = torch.empty((B, k), dtype=torch.float32).pin_memory()
        stg = torch.empty(tq.search_host_staging(B, d, k), dtype=torch.uint8, device=dev)
        qdev = torch.empty((B, d), dtype=torch.float32, device=dev)
        with torch.cuda.stream(stream):
            def e2e_step():
                if world == 1:
                    tq.search_from_host(qh, Rd, cd, bits, codes, scale, k, ih, sh, workspace=ws, staging=stg,
                                        stream=stream)
                else:
                    qdev.copy_(qh, non_blocking=True)
                    tq.search(qdev, Rd, cd, bits, codes, scale, k, workspace=ws, out_ids=ids,
                              out_scores=scs, stream=stream)
                    exchange()
                    ih.copy_(gids, non_blocking=True)
                    sh.copy_(gscs, non_blocking=True)

            for _ in range(max(1, args.warmup)):
                e2e_step()
            barrier()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(args.steps):
                e2e_step()
            b.record(stream)
            b.synchronize()
        e2e_ms = a.elapsed_time(b)
        # our kernels per step: the rotation (with its reduce from 16 queries on:
        # the tensor-core rotation), then the lookup scan (merged in its last
        # CTA) or query packing + tensor-core scan + merge; + the shard merge
        launches = (2 if B >= 16 else 1) + (3 if mma else 1) + (1 if world > 1 else 0)
        results[B] = {
            "value": qps, "ms_per_step": ms / args.steps, "roofline": roof, "clocks": clk.summary(),
            "gpu_launches": launches * args.steps,
            "e2e": {"value": B * args.steps * world / (e2e_ms / 1e3), "unit": "queries/s",
                    "h2d_bytes_per_step": B * d * 4, "d2h_bytes_per_step": B * k * 12},
        }
        log(f"[bench] B={B}: {qps:.4g} q/s, {ms / args.steps:.3f} ms/step, scan {scan_ms:.3f} ms "
            f"= {achieved:.0f} GB/s ({100 * achieved / pk['hbm_gbs']:.1f}% of {pk['source']} HBM)")
        del ws

    tq.set_search_path("auto")
    # Recall@k of both scan paths on the same queries
    recall = {"k": k, "queries": nrec,
              "exact": "float32 brute force over the unquantised normalised corpus"}
    for path in ("lut", "mma"):
        if path == "mma" and not (bits in (2, 3, 4, 8) and k <= 64):
            continue
        tq.set_search_path(path)
        try:
            with torch.cuda.stream(stream):
                got, _ = tq.search(Qd[:nrec], Rd, cd, bits, codes, scale, k, stream=stream)
            stream.synchronize()
        finally:
            tq.set_search_path("auto")
        hit = (got.unsqueeze(2) == exact.unsqueeze(1)).any(dim=2).float().sum(dim=1) / k
        recall[path] = float(hit.mean())
    log(f"[bench] Recall@{k} over {nrec} queries: {recall}")
    # Hit@k and MRR@20 against the exact top-1 (the RAG-quality metrics of
    # Sec. IV-E, Table III), from each path's top-20
    rag = {"queries": nrec, "exact_top1": "float32 brute force over the unquantised normalised corpus"}
    for path in ("lut", "mma"):
        if path == "mma" and bits not in (2, 3, 4, 8):
            continue
        tq.set_search_path(path)
        try:
            with torch.cuda.stream(stream):
                top20, _ = tq.search(Qd[:nrec], Rd, cd, bits, codes, scale, 20, stream=stream)
            stream.synchronize()
        finally:
            tq.set_search_path("auto")
        at = (top20 == exact[:, :1])                       # [nrec, 20]: where the exact top-1 sits
        found = at.any(dim=1)
        pos = torch.where(found, at.float().argmax(dim=1) + 1, torch.zeros_like(found, dtype=torch.int64))
        m = {f"hit@{kk}": float(at[:, :kk].any(dim=1).float().mean()) for kk in (1, 3, 5, 10)}
        m["mrr@20"] = float(torch.where(found, 1.0 / pos.clamp(min=1).float(), torch.zeros(1, device=dev)).mean())
        rag[path] = m
    log(f"[bench] RAG quality over {nrec} queries: {rag}")

    head = batches[0]
    r = results[head]
    line = {
        "metric": METRIC, "value": r["value"], "unit": "queries/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": r["ms_per_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded Gaussian-mixture corpus, perturbed-corpus queries)",
        "config": arm_config(args, n, d, bits, k, head, world),
        "roofline": r["roofline"], "clocks": r["clocks"], "e2e": r["e2e"],
        "search_path": args.search_path,
        "recall": recall,
        "rag_quality": rag,
        "gpu_launches": r["gpu_launches"],
        "batches": {str(b): {"value": v["value"], "ms_per_step": v["ms_per_step"],
                             "roofline": v["roofline"], "e2e": v["e2e"], "gpu_launches": v["gpu_launches"]}
                    for b, v in results.items()},
        "encode": {"value": n / enc_ms * 1e3, "unit": "vectors/s", "ms": enc_ms,
                   "path": "tensor core (TF32, three-product split)", "roofline": _roof_encode(n, d, enc_ms, pk),
                   "ffma": {"value": n / ffma_ms * 1e3, "unit": "vectors/s", "ms": ffma_ms,
                            "tflops": 2.0 * n * d * d / (ffma_ms / 1e3) / 1e12}},
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        qps_cpu, info = oracle_qps_sample(cfg, sample_rows=min(n, args.ref_sample), n_queries=5)
        line["cpu_baseline"] = {"value": qps_cpu, "unit": "queries/s", "cores": cpu_threads(),
                                "kind": "oracle", **cpu_model(), "sample": info["sample"]}
    if run_extras:
        # the other workloads, compactly: the 100K and filtered workloads and
        # the bit-width sweep, each with its roofline
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        line["extra"] = {"100k": extras_100k(torch, tq, dev, stream, pk, flush, steps=20),
                         "sweep": extras_sweep(torch, tq, dev, stream, pk, Xd, Rd, Qd, steps=10)}
        del Xd, flush
    if rank == 0:
        print(json.dumps(line), flush=True)


def _timed(fn, steps, warmup, stream):
    """Mean ms of fn() over `steps` calls after `warmup`, CUDA events on `stream`."""
    import torch
    for i in range(warmup):
        fn(i)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record(stream)
    for i in range(steps):
        fn(warmup + i)
    b.record(stream)
    b.synchronize()
    return a.elapsed_time(b) / steps


# --------------------------------------------------------- other workloads --
def cpu_model():
    """The host CPU's model name and core count (lscpu, else /proc/cpuinfo)."""
    name = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                name = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if not name:
        try:
            with open("/proc/cpuinfo") as f:
                for line in f:
                    if line.lower().startswith(("model name", "cpu model")):
                        name = line.split(":", 1)[1].strip()
                        break
        except OSError:
            pass
    return {"model": name or "unknown", "nproc": os.cpu_count()}


def _flushed_ms(torch, fn, steps, stream, flush):
    """Mean device time of fn() over `steps` calls on `stream`, each after a
    write of `flush` (larger than L2) that is not timed: for corpora that fit
    in L2, so that every call still reads them from HBM."""
    times = []
    for i in range(steps):
        flush.fill_(i & 255)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn(i)
        b.record(stream)
        times.append((a, b))
    stream.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in times)


def _scan_ms(torch, tq, fn, steps, stream, flush=None):
    """Mean duration of the scan kernel inside fn(), from the library's events."""
    evs = []
    for i in range(steps):
        if flush is not None:
            flush.fill_(i & 255)
        e = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
        tq.profile_events(*e)
        fn(i)
        evs.append(e)
    tq.profile_events(None, None)
    stream.synchronize()
    return statistics.mean(a.elapsed_time(b) for a, b in evs)


def _roof_hbm(alg_bytes, ms, pk, kernel):
    gbs = alg_bytes / (ms / 1e3) / 1e9
    return {"bound": "hbm", "achieved": gbs, "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": gbs / pk["hbm_gbs"],
            "frac_of": pk["source"], "traffic": None, "kernel": kernel, "alg_bytes_per_launch": alg_bytes,
            "kernel_ms": ms}


def _roof_tc(flops, ms, pk):
    tf = flops / (ms / 1e3) / 1e12
    return {"bound": "tensor", "achieved": tf, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
            "frac": tf / pk["bf16_tflops"], "frac_of": pk["source"] + " burst bf16 (= fp16 dense rate)",
            "traffic": None, "kernel": "k_scan_mma", "alg_flops_per_launch": flops, "kernel_ms": ms}


TF32_PER_BF16 = 1.1 / 2.25  # nominal dense TF32 / BF16 tensor rates of the GB300


def _roof_encode(n, d, ms, pk):
    """Roofline of the tensor-core encoder: three TF32 products per
    multiply-add of the rotation (2 n d^2 flops each), against the TF32
    peak taken as the measured burst bf16 peak times the nominal ratio."""
    flops = 3 * 2.0 * n * d * d
    tf = flops / (ms / 1e3) / 1e12
    peak = pk["bf16_tflops"] * TF32_PER_BF16
    return {"bound": "tensor", "achieved": tf, "peak": peak, "unit": "TFLOP/s", "frac": tf / peak,
            "frac_of": pk["source"] + " burst bf16 x 1.1/2.25 (TF32 dense rate)", "traffic": None,
            "kernel": "k_encode_tc", "alg_flops_per_launch": flops, "kernel_ms": ms,
            "rotation_tflops": 2.0 * n * d * d / (ms / 1e3) / 1e12}


def _recall(torch, ids, exact):
    """Mean |ids ∩ exact| / |exact| over queries (torch tensors [nq, k]; -1 is no result)."""
    hits = 0.0
    for g, e in zip(ids.tolist(), exact.tolist()):
        e = {v for v in e if v >= 0}
        hits += len({v for v in g if v >= 0} & e) / max(1, len(e))
    return hits / len(exact)


def extras_100k(torch, tq, dev, stream, pk, flush, steps):
    """The 100K workload (batch 1 and 256, top-5 and top-10, encode) and the
    filtered workload on the same corpus (Zipf tenants, T = 10, 100, 1000,
    batch 1, with the over-fetch post-filter baseline).  The corpus (77 MB of
    codes) fits in L2, so L2 is flushed before every timed search."""
    import oracle as O
    from paper_2607_16973_gb300 import synth
    cfg, fcfg = CONFIGS["c2"], CONFIGS["filtered"]
    n, d, bits = cfg["n"], cfg["d"], cfg["bits"]
    X = synth.mixture_corpus(n, d, cfg["clusters"], workers=min(16, os.cpu_count() or 4))
    src = synth.query_sources(n, cfg["pool"])
    Q = synth.perturb(X[src])
    cen, bnd, _ = tq.codebook(d, bits)
    R = tq.rotation(d, synth.SEED_ROTATION)
    nrec = min(RECALL_Q, len(Q))
    with torch.cuda.stream(stream):
        Xd, Qd, Rd, cd, bd = (torch.from_numpy(a).to(dev) for a in (X, Q, R, cen, bnd))
        plan = tq.encode_plan(Rd, stream=stream)
        codes, scale = tq.encode(Xd, Rd, cd, bd, bits, stream=stream, plan=plan)
        enc_ms = _flushed_ms(torch, lambda i: tq.encode(Xd, Rd, cd, bd, bits, "norm", codes, scale, stream=stream,
                                                        plan=plan), 3, stream, flush)
        exact_sc = Qd[:nrec] @ Xd.T                      # float32, TF32 off: [nrec, n]
    stream.synchronize()
    out = {"workload": f"N={n} d={d} {bits}-bit, {cfg['clusters']}-cluster mixture, {len(Q)} queries",
           "l2": "corpus fits in L2: flushed before every timed call",
           "encode": {"value": n / enc_ms * 1e3, "unit": "vectors/s", "ms": enc_ms,
                      "roofline": _roof_encode(n, d, enc_ms, pk)}}
    alg = n * (d * bits // 8 + 4)
    for B in (1, 256):
        for k in (5, 10):
            nb = max(1, len(Q) // B)
            ws = torch.empty(tq.search_workspace(B, n, d, bits, k), dtype=torch.uint8, device=dev)
            ids = torch.empty((B, k), dtype=torch.int64, device=dev)
            scs = torch.empty((B, k), dtype=torch.float32, device=dev)

            def fn(i):
                j = (i % nb) * B
                tq.search(Qd[j:j + B], Rd, cd, bits, codes, scale, k, workspace=ws, out_ids=ids, out_scores=scs,
                          stream=stream)
            with torch.cuda.stream(stream):
                for i in range(3):
                    fn(i)
                ms = _flushed_ms(torch, fn, steps, stream, flush)
                kms = _scan_ms(torch, tq, fn, steps, stream, flush)
                tq.set_search_path("lut" if B < MMA_MIN_BATCH else "auto")
                try:
                    got, _ = tq.search(Qd[:nrec], Rd, cd, bits, codes, scale, k, stream=stream)
                finally:
                    tq.set_search_path("auto")
                ex = torch.topk(exact_sc, k, dim=1)[1]
            stream.synchronize()
            roof = _roof_tc(2.0 * n * d * B, kms, pk) if B >= MMA_MIN_BATCH else _roof_hbm(alg, kms, pk,
                                                                                        "k_scan_stream")
            out[f"batch{B}_top{k}"] = {"value": B / ms * 1e3, "unit": "queries/s", "ms_per_step": ms,
                                       "roofline": roof, "recall": _recall(torch, got.cpu(), ex.cpu())}
            log(f"[bench] 100K batch {B} top-{k}: {B / ms * 1e3:.4g} q/s, scan {kms * 1e3:.1f} us")
    # filtered workload on the same corpus
    k, blk = fcfg["k"], fcfg["block"]
    rb = d * bits // 8
    filt_out = {}
    for T in fcfg["tenants"]:
        tid, values = synth.zipf_tenants(n, T)
        off, allow = synth.allowlists(src, tid, values)
        filt = tq.Filter(torch.from_numpy(tid.view(np.int32)).to(dev), block=blk, stream=stream)
        q_off = [torch.tensor([0, off[i + 1] - off[i]], dtype=torch.int64, device=dev) for i in range(len(Q))]
        q_ten = [torch.from_numpy(allow[off[i]:off[i + 1]].view(np.int32)).to(dev) for i in range(len(Q))]
        ws = torch.empty(tq.search_workspace(1, n, d, bits, k, filt), dtype=torch.uint8, device=dev)
        ids = torch.empty((1, k), dtype=torch.int64, device=dev)
        scs = torch.empty((1, k), dtype=torch.float32, device=dev)

        def fn(i):
            j = i % len(Q)
            tq.search(Qd[j:j + 1], Rd, cd, bits, codes, scale, k, filter=filt, allow_off=q_off[j],
                      allow_tenants=q_ten[j], workspace=ws, out_ids=ids, out_scores=scs, stream=stream)
        # share of the corpus each timed query skips (filter blocks without an allowed tenant)
        nblocks = (n + blk - 1) // blk
        tb = np.concatenate([tid, np.full(nblocks * blk - n, 0xFFFFFFFF, np.uint32)]).reshape(nblocks, blk)
        skip = [1.0 - np.isin(tb, allow[off[i % len(Q)]:off[i % len(Q) + 1]]).any(axis=1).mean()
                for i in range(steps)]
        with torch.cuda.stream(stream):
            for i in range(3):
                fn(i)
            ms = _flushed_ms(torch, fn, steps, stream, flush)
            kms = _scan_ms(torch, tq, fn, steps, stream, flush)
            # recall against exact kNN restricted to the allowed vectors, and the
            # over-fetch post-filter baseline (Sec. V-C, Table V)
            k_over = min(256, k * max(1, T // 10))
            ws_o = torch.empty(tq.search_workspace(1, n, d, bits, k_over), dtype=torch.uint8, device=dev)
            ids_o = torch.empty((1, k_over), dtype=torch.int64, device=dev)
            scs_o = torch.empty((1, k_over), dtype=torch.float32, device=dev)

            def fn_over(i):
                j = i % len(Q)
                tq.search(Qd[j:j + 1], Rd, cd, bits, codes, scale, k_over, workspace=ws_o, out_ids=ids_o,
                          out_scores=scs_o, stream=stream)
            ms_over = _flushed_ms(torch, fn_over, steps, stream, flush)
            over, _ = tq.search(Qd[:nrec], Rd, cd, bits, codes, scale, k_over, stream=stream)
            got = []
            for i in range(nrec):
                g, _ = tq.search(Qd[i:i + 1], Rd, cd, bits, codes, scale, k, filter=filt, allow_off=q_off[i],
                                 allow_tenants=q_ten[i], stream=stream)
                got.append(g)
            got = torch.cat(got)
        stream.synchronize()
        hits = pf_hits = 0.0
        over = over.cpu().numpy()
        for i in range(nrec):
            ok = np.isin(tid, allow[off[i]:off[i + 1]])
            sc = torch.where(torch.from_numpy(ok).to(dev), exact_sc[i], torch.tensor(float("-inf"), device=dev))
            ex = set(torch.topk(sc, min(k, int(ok.sum())))[1].tolist())
            hits += len(ex & set(got[i].tolist())) / max(1, len(ex))
            kept = [v for v in over[i] if v >= 0 and ok[v]][:k]
            pf_hits += len(ex & set(kept)) / max(1, len(ex))
        filt.close()
        live = (1.0 - float(np.mean(skip))) * alg + n * 4  # codes + scales of the blocks read, dense tenant ids
        filt_out[str(T)] = {"value": 1e3 / ms, "unit": "queries/s", "ms_per_query": ms,
                            "bytes_skipped_frac": float(np.mean(skip)), "recall": hits / nrec,
                            "roofline": _roof_hbm(live, kms, pk, "k_scan_stream (filtered)"),
                            "postfilter": {"overfetch_k": k_over, "recall": pf_hits / nrec, "ms_per_query": ms_over}}
        log(f"[bench] filtered T={T}: {1e3 / ms:.4g} q/s, scan {kms * 1e3:.1f} us, {np.mean(skip):.1%} skipped, "
            f"R@{k} {hits / nrec:.3f}, post-filter R@{k} {pf_hits / nrec:.3f}")
    out["filtered"] = {"workload": f"Zipf(1.1) tenants, block {blk}, batch 1, top-{k}, 10% of the queries allow 5",
                       "variants": filt_out}
    # the oracle on the host cores: its search of 3 single queries over the
    # whole 100K corpus, which it encodes itself
    enc = O.encode(X, R, cen, bnd, bits)
    t = []
    for q in range(3):
        t0 = time.perf_counter()
        O.search(Q[q:q + 1], R, cen, bits, enc.packed, enc.scale, 10, d)
        t.append(time.perf_counter() - t0)
    out["cpu_baseline"] = {"value": 1.0 / statistics.median(t), "unit": "queries/s", "cores": cpu_threads(),
                           "kind": "oracle", **cpu_model(),
                           "sample": "oracle search (float64 numpy) of 3 single queries over all 100,000 rows, "
                                     "top-10, median"}
    del Xd
    return out


def extras_sweep(torch, tq, dev, stream, pk, Xd, Rd, Qd, steps):
    """The bit-width sweep on the 999K corpus already on the device: encode at
    b = 2, 3, 4, 8 and batch-256 top-10 search at each width."""
    cfg = CONFIGS["sweep"]
    n, d, k, B = cfg["n"], cfg["d"], cfg["k"], cfg["batches"][0]
    nb = max(1, Qd.shape[0] // B)
    out = {"workload": f"N={n} d={d}, batch {B}, top-{k}; corpus larger than L2", "variants": {}}
    plan = tq.encode_plan(Rd, stream=stream)
    for bits in cfg["sweep_bits"]:
        cen, bnd, _ = tq.codebook(d, bits)
        cd, bd = torch.from_numpy(cen).to(dev), torch.from_numpy(bnd).to(dev)
        with torch.cuda.stream(stream):
            codes = torch.empty((n, d * bits // 8), dtype=torch.uint8, device=dev)
            scale = torch.empty(n, dtype=torch.float32, device=dev)
            enc = lambda i: tq.encode(Xd, Rd, cd, bd, bits, "norm", codes, scale, stream=stream, plan=plan)
            enc(0)
            enc_ms = _timed(enc, 3, 1, stream)
            ws = torch.empty(tq.search_workspace(B, n, d, bits, k), dtype=torch.uint8, device=dev)
            ids = torch.empty((B, k), dtype=torch.int64, device=dev)
            scs = torch.empty((B, k), dtype=torch.float32, device=dev)

            def fn(i):
                j = (i % nb) * B
                tq.search(Qd[j:j + B], Rd, cd, bits, codes, scale, k, workspace=ws, out_ids=ids, out_scores=scs,
                          stream=stream)
            ms = _timed(fn, steps, 2, stream)
            kms = _scan_ms(torch, tq, fn, min(steps, 5), stream)
        mma = bits in (2, 3, 4, 8)
        alg = n * (d * bits // 8 + 4)
        roof = _roof_tc(2.0 * n * d * B, kms, pk) if mma else _roof_hbm(alg, kms, pk, "k_scan_ring")
        out["variants"][str(bits)] = {"value": B / ms * 1e3, "unit": "queries/s", "ms_per_step": ms,
                                      "path": "tensor core" if mma else "lookup", "roofline": roof,
                                      "encode": {"value": n / enc_ms * 1e3, "unit": "vectors/s", "ms": enc_ms,
                                                 "roofline": _roof_encode(n, d, enc_ms, pk)}}
        log(f"[bench] sweep b={bits}: encode {n / enc_ms * 1e3:.3g} vec/s, batch {B}: {B / ms * 1e3:.4g} q/s")
        del codes, scale, ws
        torch.cuda.empty_cache()
    return out


def run_filtered(args, cfg):
    """Filtered search (allowlists of tenants) at batch 1 for each tenant
    count: queries/s, the share of code bytes the per-block tenant bitmaps
    skip, and Recall@k against exact filtered kNN."""
    import torch
    import paper_2607_16973_gb300 as tq
    from paper_2607_16973_gb300 import synth
    from paper_2607_16973_gb300.build import build
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    build()
    tq.load()
    n, d, bits, k, blk = cfg["n"], cfg["d"], cfg["bits"], args.k or cfg["k"], cfg["block"]
    stream = torch.cuda.Stream(device=dev)
    X = synth.mixture_corpus(n, d, cfg["clusters"], workers=min(16, os.cpu_count() or 4))
    src = synth.query_sources(n, cfg["pool"])
    Q = synth.perturb(X[src])
    cen, bnd, _ = tq.codebook(d, bits)
    R = tq.rotation(d, synth.SEED_ROTATION)
    Xd, Qd = torch.from_numpy(X).to(dev), torch.from_numpy(Q).to(dev)
    Rd, cd, bd = (torch.from_numpy(a).to(dev) for a in (R, cen, bnd))
    codes, scale = tq.encode(Xd, Rd, cd, bd, bits, plan=tq.encode_plan(Rd))
    torch.cuda.synchronize()
    torch.backends.cuda.matmul.allow_tf32 = False
    nrec = min(RECALL_Q, len(Q))
    exact_scores = Qd[:nrec] @ Xd.T                       # [nrec, n] float32, unquantised
    variants = {}
    steps = min(args.steps, len(Q) - args.warmup) if len(Q) > args.warmup else args.steps
    for T in cfg["tenants"]:
        tid, values = synth.zipf_tenants(n, T)
        off, allow = synth.allowlists(src, tid, values)
        filt = tq.Filter(torch.from_numpy(tid.view(np.int32)).to(dev), block=blk)
        # per-query CSR slices (offsets rebased to 0), on the device
        q_off = [torch.tensor([0, off[i + 1] - off[i]], dtype=torch.int64, device=dev) for i in range(len(Q))]
        q_ten = [torch.from_numpy(allow[off[i]:off[i + 1]].view(np.int32)).to(dev) for i in range(len(Q))]
        ws = torch.empty(tq.search_workspace(1, n, d, bits, k, filt), dtype=torch.uint8, device=dev)
        ids = torch.empty((1, k), dtype=torch.int64, device=dev)
        scs = torch.empty((1, k), dtype=torch.float32, device=dev)

        def step(i):
            j = i % len(Q)
            tq.search(Qd[j:j + 1], Rd, cd, bits, codes, scale, k, filter=filt, allow_off=q_off[j],
                      allow_tenants=q_ten[j], workspace=ws, out_ids=ids, out_scores=scs, stream=stream)

        with torch.cuda.stream(stream):
            ms = _timed(step, steps, args.warmup, stream)
        # share of code blocks skipped (no allowed tenant in the block)
        nblocks = (n + blk - 1) // blk
        pad = np.full(nblocks * blk - n, np.uint32(0xFFFFFFFF), np.uint32)
        tb = np.concatenate([tid, pad]).reshape(nblocks, blk)
        skipped = []
        for i in range(min(200, len(Q))):
            ok = np.isin(tb, allow[off[i]:off[i + 1]]).any(axis=1)
            skipped.append(1.0 - ok.mean())
        # Recall@k against exact kNN restricted to the allowed vectors
        hits = 0.0
        for i in range(nrec):
            mask = torch.from_numpy(np.isin(tid, allow[off[i]:off[i + 1]])).to(dev)
            sc = torch.where(mask, exact_scores[i], torch.tensor(float("-inf"), device=dev))
            ex = torch.topk(sc, min(k, int(mask.sum())))[1]
            with torch.cuda.stream(stream):
                got, _ = tq.search(Qd[i:i + 1], Rd, cd, bits, codes, scale, k, filter=filt, allow_off=q_off[i],
                                   allow_tenants=q_ten[i], stream=stream)
            stream.synchronize()
            g = got[0][got[0] >= 0]
            hits += float(torch.isin(g, ex).float().sum()) / max(1, len(ex))
        # the over-fetch post-filter baseline (Sec. V-C, Table V): an unfiltered
        # search of k * T/10 candidates (capped at tq_search's k <= 256), then the
        # allowed ones in order; timed as the unfiltered search it needs
        k_over = min(256, k * max(1, T // 10))
        ws_o = torch.empty(tq.search_workspace(1, n, d, bits, k_over), dtype=torch.uint8, device=dev)
        ids_o = torch.empty((1, k_over), dtype=torch.int64, device=dev)
        scs_o = torch.empty((1, k_over), dtype=torch.float32, device=dev)
        with torch.cuda.stream(stream):
            ms_o = _timed(lambda i: tq.search(Qd[i % len(Q):i % len(Q) + 1], Rd, cd, bits, codes, scale, k_over,
                                              workspace=ws_o, out_ids=ids_o, out_scores=scs_o, stream=stream),
                          steps, args.warmup, stream)
            over, _ = tq.search(Qd[:nrec], Rd, cd, bits, codes, scale, k_over, stream=stream)
        stream.synchronize()
        over = over.cpu().numpy()
        pf_hits = 0.0
        for i in range(nrec):
            ok = np.isin(tid[np.maximum(over[i], 0)], allow[off[i]:off[i + 1]]) & (over[i] >= 0)
            kept = torch.from_numpy(over[i][ok][:k]).to(dev)
            mask = torch.from_numpy(np.isin(tid, allow[off[i]:off[i + 1]])).to(dev)
            sc = torch.where(mask, exact_scores[i], torch.tensor(float("-inf"), device=dev))
            ex = torch.topk(sc, min(k, int(mask.sum())))[1]
            pf_hits += float(torch.isin(kept, ex).float().sum()) / max(1, len(ex))
        variants[str(T)] = {"value": 1e3 / ms, "ms_per_query": ms, "bytes_skipped_frac": float(np.mean(skipped)),
                            "recall": hits / nrec,
                            "postfilter": {"overfetch_k": k_over, "recall": pf_hits / nrec, "ms_per_query": ms_o}}
        log(f"[bench] filtered T={T}: {1e3 / ms:.4g} q/s, {ms * 1e3:.1f} us/query, "
            f"{100 * np.mean(skipped):.1f}% of code blocks skipped, R@{k} {hits / nrec:.3f}; "
            f"post-filter (k'={k_over}) R@{k} {pf_hits / nrec:.3f} at {ms_o * 1e3:.1f} us/query")
        filt.close()
    head = variants[str(cfg["tenants"][0])]
    line = {"metric": f"filtered queries/sec at {n // 1000}Kx{d} {bits}-bit top-{k} (batch 1)", "value": head["value"],
            "unit": "queries/s", "n_gpus": 1, "steps": steps, "warmup": args.warmup,
            "ms_per_step": head["ms_per_query"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": "synthetic (Gaussian mixture, Zipf(1.1) tenants in interleaved order)",
            "config": {"workload": f"filtered: N={n} d={d} {bits}-bit top-{k}, Zipf tenants T in {cfg['tenants']}, "
                                   f"block {blk}, 10% of queries allow 5 tenants", "n": n, "d": d, "bits": bits,
                       "k": k, "block": blk},
            "variants": variants, "gpu_launches": 4 * steps}
    print(json.dumps(line), flush=True)


def run_sweep(args, cfg):
    """Encode throughput and batch-B top-k search at each bit width."""
    import torch
    import paper_2607_16973_gb300 as tq
    from paper_2607_16973_gb300 import synth
    from paper_2607_16973_gb300.build import build
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    build()
    tq.load()
    n, d, k = cfg["n"], cfg["d"], args.k or cfg["k"]
    B = int(args.batches.split(",")[0]) if args.batches else cfg["batches"][0]
    stream = torch.cuda.Stream(device=dev)
    X, Qpool = make_corpus(cfg, workers=min(16, os.cpu_count() or 4))
    R = tq.rotation(d, synth.SEED_ROTATION)
    Xd, Rd, Qd = torch.from_numpy(X).to(dev), torch.from_numpy(R).to(dev), torch.from_numpy(Qpool).to(dev)
    del X
    nb = max(1, len(Qpool) // B)
    variants = {}
    plan = tq.encode_plan(Rd)
    for bits in cfg["sweep_bits"]:
        cen, bnd, _ = tq.codebook(d, bits)
        cd, bd = torch.from_numpy(cen).to(dev), torch.from_numpy(bnd).to(dev)
        codes = torch.empty((n, d * bits // 8), dtype=torch.uint8, device=dev)
        scale = torch.empty(n, dtype=torch.float32, device=dev)
        with torch.cuda.stream(stream):
            enc_ms = _timed(lambda i: tq.encode(Xd, Rd, cd, bd, bits, "norm", codes, scale, stream=stream,
                                                plan=plan), 3, 1, stream)
            ws = torch.empty(tq.search_workspace(B, n, d, bits, k), dtype=torch.uint8, device=dev)
            ids = torch.empty((B, k), dtype=torch.int64, device=dev)
            scs = torch.empty((B, k), dtype=torch.float32, device=dev)
            steps = max(1, min(args.steps, 10))
            ms = _timed(lambda i: tq.search(Qd[(i % nb) * B:(i % nb) * B + B], Rd, cd, bits, codes, scale, k,
                                            workspace=ws, out_ids=ids, out_scores=scs, stream=stream),
                        steps, min(args.warmup, 3), stream)
        path = "tensor core" if bits in (2, 3, 4, 8) and k <= 64 else "lookup"
        variants[str(bits)] = {"encode_vectors_per_s": n / enc_ms * 1e3, "encode_ms": enc_ms,
                               "value": B / ms * 1e3, "ms_per_step": ms, "path": path,
                               "codes_mb": n * d * bits / 8 / 1e6}
        log(f"[bench] sweep b={bits}: encode {n / enc_ms * 1e3:.3g} vec/s, search B={B} {B / ms * 1e3:.4g} q/s "
            f"({path})")
        del codes, scale, ws
        torch.cuda.empty_cache()
    head = variants[str(cfg["sweep_bits"][0])]
    line = {"metric": f"queries/sec at {n // 1000}Kx{d} top-{k} batch {B} by bit width; encode vectors/sec",
            "value": head["value"], "unit": "queries/s", "n_gpus": 1, "steps": max(1, min(args.steps, 10)),
            "warmup": min(args.warmup, 3), "ms_per_step": head["ms_per_step"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded Gaussian-mixture corpus, perturbed-corpus queries)",
            "config": {"workload": f"sweep: N={n} d={d} b in {cfg['sweep_bits']}, batch {B}, top-{k}", "n": n, "d": d,
                       "k": k, "batch": B},
            "variants": variants}
    print(json.dumps(line), flush=True)


def run_idmap(args, cfg):
    """Search over an id-mapped index (external uint64 ids, a share of the
    rows deleted) against the same search without the id map: the cost of
    the tombstone checks and the id mapping."""
    import torch
    import paper_2607_16973_gb300 as tq
    from paper_2607_16973_gb300 import synth
    from paper_2607_16973_gb300.build import build
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    build()
    tq.load()
    n, d, bits, k = cfg["n"], cfg["d"], cfg["bits"], args.k or cfg["k"]
    batches = [int(b) for b in args.batches.split(",")] if args.batches else cfg["batches"]
    stream = torch.cuda.Stream(device=dev)
    X, Qpool = make_corpus(cfg, workers=min(16, os.cpu_count() or 4))
    cen, bnd, _ = tq.codebook(d, bits)
    R = tq.rotation(d, synth.SEED_ROTATION)
    Xd = torch.from_numpy(X).to(dev)
    Rd, cd, bd, Qd = (torch.from_numpy(a).to(dev) for a in (R, cen, bnd, Qpool))
    codes, scale = tq.encode(Xd, Rd, cd, bd, bits, plan=tq.encode_plan(Rd))
    del Xd, X
    rng = np.random.default_rng(synth.SEED_QUERIES)
    ext = rng.choice(1 << 62, size=n, replace=False).astype(np.uint64)
    gone = rng.choice(n, int(cfg["deleted_frac"] * n), replace=False)
    m = tq.IdMap(n)
    m.add(ext, stream=stream)
    m.remove(ext[gone], stream=stream)
    torch.cuda.synchronize()
    variants = {}
    for B in batches:
        nb = max(1, len(Qpool) // B)
        ws = torch.empty(tq.search_workspace(B, n, d, bits, k), dtype=torch.uint8, device=dev)
        ids = torch.empty((B, k), dtype=torch.int64, device=dev)
        scs = torch.empty((B, k), dtype=torch.float32, device=dev)
        res = {}
        for name, im in (("plain", None), ("idmap", m)):
            with torch.cuda.stream(stream):
                res[name] = _timed(lambda i: tq.search(Qd[(i % nb) * B:(i % nb) * B + B], Rd, cd, bits, codes, scale,
                                                       k, workspace=ws, out_ids=ids, out_scores=scs, stream=stream,
                                                       idmap=im), args.steps, args.warmup, stream)
        # every returned id is a live external id
        with torch.cuda.stream(stream):
            got, _ = tq.search(Qd[:B], Rd, cd, bits, codes, scale, k, stream=stream, idmap=m)
        stream.synchronize()
        live = set(np.delete(ext, gone).view(np.int64).tolist())
        ok = all(v in live for v in got.cpu().numpy().reshape(-1).tolist() if v != -1)
        variants[str(B)] = {"value": B / res["idmap"] * 1e3, "ms_per_step": res["idmap"],
                            "plain_value": B / res["plain"] * 1e3, "plain_ms_per_step": res["plain"],
                            "overhead_frac": res["idmap"] / res["plain"] - 1.0, "results_live": ok}
        log(f"[bench] idmap B={B}: {B / res['idmap'] * 1e3:.4g} q/s with the id map, "
            f"{B / res['plain'] * 1e3:.4g} without ({100 * (res['idmap'] / res['plain'] - 1):+.1f}%), "
            f"results live: {ok}")
    m.close()
    head = variants[str(batches[0])]
    line = {"metric": f"queries/sec at {n // 1000}Kx{d} {bits}-bit top-{k} over an id-mapped index",
            "value": head["value"], "unit": "queries/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": head["ms_per_step"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": "synthetic (seeded Gaussian-mixture corpus, random external ids)",
            "config": {"workload": f"idmap: N={n} d={d} {bits}-bit top-{k}, {cfg['deleted_frac']:.0%} of the rows "
                                   f"deleted, batches {batches}", "n": n, "d": d, "bits": bits, "k": k},
            "variants": variants}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", choices=sorted(CONFIGS), default="scale")
    ap.add_argument("--batches", default=None, help="comma-separated batch sizes (first = headline)")
    ap.add_argument("--k", type=int, default=None)
    ap.add_argument("--bits", type=int, default=None, choices=[2, 3, 4, 8],
                    help="code width for the scale/c2/tiny/prof workloads (default: 4)")
    ap.add_argument("--ref-sample", type=int, default=50_000, help="corpus rows the oracle scans per step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--search-path", default="auto", choices=["auto", "lut", "lut_fixed", "lut_fold", "mma"],
                    help="scan kernels of the timed batches (tq_set_search_path; default: AUTO)")
    ap.add_argument("--no-extras", action="store_true",
                    help="scale workload only: skip the 100K, filtered and bit-width sweep lines under 'extra'")
    args = ap.parse_args()
    cfg = CONFIGS[args.config]
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        run_reference(args, cfg, rank, world)
        return
    if args.config in ("filtered", "sweep", "idmap"):
        if rank == 0:
            {"filtered": run_filtered, "sweep": run_sweep, "idmap": run_idmap}[args.config](args, cfg)
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        dist.init_process_group("nccl")
    run_ours(args, cfg, rank, world)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
