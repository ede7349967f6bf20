#!/usr/bin/env python3
"""Throughput of the GB300 retrieval hot path: queries/s at top-k and the
fraction of the roofline reached by the dominant kernel.

Headline workload (one step = one 4096-row upsert + one search call): the
scale case, 1,048,576 chunks x 768 bf16, a batch of 2048 queries, top-100
(the largest single-GPU workload; Sec. 5.1 shapes: 768-d embeddings, dense
retrieval with upserts between batches).  The same JSON line carries, under
"configs", the other workloads measured the same way: the tiny fp32 case
(1024 x 384, 16 queries), the paper-shaped dense search (32768 x 768, batches
of 1, 32 and 256, top-5), the clustered search (32768 x 1024, 4096 queries,
top-10) and the hybrid dense + BM25 search (32768 x 768, 1024 queries, top-5).
--config C [--batch Q] measures one workload alone.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Timing: W untimed steps, then K steps; before every step a 512 MiB buffer is
written (L2 flush, outside the timed events); each step is bracketed by CUDA
events on the launch stream and the steps are enqueued without waiting on the
host.  A second pass over the same steps, with the library's own events
around each of its kernels, times the search kernel for the roofline.  Under
torchrun every rank runs the same workloads on its own GPU (replicas), the
slowest rank's time counts and `value` adds the queries of all ranks.

Oracle leg (skipped with --no-cpu-baseline): on rank 0 the outputs of the
last timed step of every workload are checked against the CPU oracle on a
sample with rows in every 32-query group of every 128-query tile
("parity"), and the oracle itself is timed on a bounded sample of the
headline workload ("cpu_baseline").  --impl reference times the oracle alone
on the host cores (bounded samples of the same workload).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_08340_gb300 import workloads  # noqa: E402

L2_FLUSH_BYTES = 512 << 20
# Files that define the search kernel whose DRAM traffic profiles/ncu_traffic.json
# records; the hash covers their code with comments and blank space removed.
KERNEL_SOURCES = ["common.cuh", "search_tc.cuh", "search_tc.cu"]


def _code_only(text: str) -> str:
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def source_hash(read=None) -> str:
    h = hashlib.sha256()
    for name in KERNEL_SOURCES:
        path = os.path.join(ROOT, "paper_2608_08340_gb300", "csrc", name)
        text = read(name) if read else open(path, encoding="utf-8").read()
        h.update(_code_only(text).encode())
    return h.hexdigest()[:16]


HEADLINE = (4, 2048)
# The other workloads reported under "configs": (config, queries per step).
SUB_WORKLOADS = [(0, 16), (1, 1), (1, 32), (1, 256), (2, 4096), (3, 1024)]
TOL = 1e-4          # parity bar: absolute score tolerance (oracle/check.py rules)


def parse(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--config", type=int, default=None,
                   help="measure this workload alone (default: the scale workload as the "
                        "headline plus every other workload under \"configs\")")
    p.add_argument("--batch", type=int, default=None, help="queries per step (with --config)")
    p.add_argument("--n", type=int, default=None,
                   help="corpus rows (with --config; a smaller case of the same kernels, e.g. "
                        "for a profiler capture)")
    p.add_argument("--phases", action="store_true",
                   help="also record per-CTA global-timer stamps of the main search pass and "
                        "report their spread (\"phases\")")
    p.add_argument("--no-cpu-baseline", action="store_true",
                   help="skip the oracle leg (parity of the timed outputs and cpu_baseline)")
    p.add_argument("--block-n", type=int, default=0, help="tensor-core tile rows (0 = auto)")
    p.add_argument("--path", choices=["auto", "simt", "tc"], default="auto")
    p.add_argument("--pair", choices=["auto", "single", "pair", "dual"], default="auto",
                   help="tensor-core kernel: CTA pairs (M = 256 MMAs), single CTAs with one "
                        "query tile per unit, or dual mode (two query tiles per unit)")
    p.add_argument("--embed-tail", action="store_true",
                   help="time the embedding tail instead (masked mean pool + L2 normalise of "
                        "256 x 512 x 4096 bf16 hidden states, the Llama3-8B hidden size)")
    p.add_argument("--graph", action="store_true",
                   help="dense configs: run the searches on a side stream in graph mode "
                        "(repeated searches replay one captured CUDA graph)")
    p.add_argument("--index-ops", action="store_true",
                   help="time the index updates instead: append of 4096 rows, replacement of "
                        "4096 token bags (BM25 rebuilt), search over a knowledge + memory index")
    p.add_argument("--lex-gather", action="store_true",
                   help="config 3: gather BM25 in the search epilogue (OPRAG_OPT_LEX_GATHER) "
                        "instead of reading a materialised BM25 block")
    p.add_argument("--dense-first", type=int, default=0, metavar="N",
                   help="config 3 only: dense top-N, then the lexical rerank of those N "
                        "candidates (dense-first hybrid) instead of the full hybrid")
    return p.parse_args(argv)


def default_batch(cfg: int) -> int:
    return {0: 16, 1: 256, 2: 4096, 3: 1024, 4: 2048}[cfg]


def workload_name(cfg: int, w, dense_first: int = 0) -> str:
    base = {0: "tiny dense top-5", 1: "paper-shaped dense top-5", 2: "clustered dense top-10",
            3: "hybrid dense+BM25 top-5", 4: "scale dense top-100 with 4096-row upserts"}[cfg]
    if cfg == 3 and dense_first:
        base = f"dense-first hybrid top-5 (dense top-{dense_first}, lexical rerank)"
    return f"{base}: {w.n} x {w.d} {w.dtype}, {w.q} queries/step"


def workload_key(cfg: int, q: int) -> str:
    return f"cfg{cfg}_q{q}"


def config_dict(cfg: int, w, world: int, dense_first: int = 0) -> dict:
    """The `config` object of a bench line; the same for both arms."""
    return {"workload": workload_name(cfg, w, dense_first), "config_index": cfg,
            "n": w.n, "d": w.d, "q": w.q, "k": w.k, "parallelism": f"replicas{world}",
            "l2": f"flushed before every step ({L2_FLUSH_BYTES >> 20} MiB write)"}


def parity_rows(q: int, seed: int = 0) -> np.ndarray:
    """Rows to check against the oracle: every row of a batch of at most 64
    queries; otherwise one random row in every 32-query group of every
    128-query tile (each TMEM lane quarter of each tile)."""
    if q <= 64:
        return np.arange(q)
    rng = np.random.default_rng(seed)
    rows = []
    for lo in range(0, q, 32):
        rows.append(int(rng.integers(lo, min(q, lo + 32))))
    return np.asarray(rows, np.int64)


def upsert_sequence(warmup: int, steps: int, rounds: int = 4):
    """Upsert rounds applied before the last timed step's search, in order
    (step i upserts round i mod rounds; warm-up steps first)."""
    return [i % rounds for i in range(warmup)] + [i % rounds for i in range(steps)]


def slowest_replica(totals_ms, world: int, device):
    """Each timed total maximised over the ranks: the replicas run the same
    steps side by side, so the slowest one sets the job's time (identity for
    one rank).  Collective over the default process group."""
    if world <= 1:
        return [float(t) for t in totals_ms]
    import torch
    t = torch.tensor([float(x) for x in totals_ms], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(x) for x in t]


def job_rate(q: int, steps: int, world: int, total_ms: float) -> float:
    """Whole-job queries/s: every rank searched q queries per step."""
    return q * steps * world / (total_ms * 1e-3)


def sparse_terms(w) -> dict:
    """Postings (chunk, weight) pairs the lexical half must read: those of the
    distinct query terms (each read at least once), and the total visited
    over all queries (a term repeated in a query counts again)."""
    doc = np.repeat(np.arange(w.n, dtype=np.int64), np.diff(w.doc_indptr.astype(np.int64)))
    pairs = np.unique(doc * w.vocab + w.doc_terms.astype(np.int64))
    df = np.bincount(pairs % w.vocab, minlength=w.vocab)
    distinct = np.unique(w.q_terms)
    return {"postings_distinct_terms": int(df[distinct].sum()),
            "postings_visited": int(df[w.q_terms].sum()),
            "bytes_distinct_terms": int(df[distinct].sum()) * 8,
            "posting_bytes": 8}


def roofline_terms(w, cfg, dense_first: int = 0):
    """Algorithmic bytes and flops of one search call: the corpus and the
    queries read once (plus, for the hybrid search, the postings of the
    distinct query terms), and 2 q n d multiply-adds of the dense scores."""
    elem = 4 if w.dtype == "f32" else 2
    nbytes = w.n * w.d * elem + w.q * w.d * elem
    if cfg == 3 and not dense_first:
        nbytes += sparse_terms(w)["bytes_distinct_terms"]
    flops = 2.0 * w.q * w.n * w.d
    return nbytes, flops


def peaks():
    """(HBM GB/s, bf16 TFLOP/s burst, bf16 TFLOP/s sustained, source)."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            m = json.load(f)
        return (float(m["hbm_gbs"]), float(m["bf16_tflops"]),
                float(m.get("bf16_tflops_sustained", m["bf16_tflops"])), "measured")
    return 6800.0, 1900.0, 1700.0, "fallback"


def ncu_traffic(workload_key: str):
    """DRAM bytes per launch of the dominant kernel from the committed ncu
    summary, if it was taken on the current kernel sources."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        table = json.load(f)
    ent = table.get(workload_key)
    if not ent or ent.get("source_hash") != source_hash():
        return None
    return ent.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.out.flush()
        with open(self.out.name) as f:
            rows = [r.strip().split(", ") for r in f if r.strip()]
        os.unlink(self.out.name)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                smax.append(float(r[2]))
            except ValueError:
                continue
            for name, v in zip(names, r[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
                "samples": len(sm)}


class NvmlSampler:
    """Reads SM clock and clock-event reasons through NVML every 2 ms on a
    background thread (read-only queries; nothing is set)."""
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, torch_device: int):
        import ctypes
        import threading
        self.samples = []
        self.max_mhz = None
        self.error = None
        self._stop = threading.Event()
        self._thread = None
        try:
            import torch
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                raise RuntimeError("nvmlInit failed")
            self.lib = lib
            self.h = ctypes.c_void_p()
            props = torch.cuda.get_device_properties(torch_device)
            ok = False
            for attr in ("pci_domain_id", "pci_bus_id", "pci_device_id"):
                if not hasattr(props, attr):
                    break
            else:
                bus = f"{props.pci_domain_id:08x}:{props.pci_bus_id:02x}:{props.pci_device_id:02x}.0"
                ok = lib.nvmlDeviceGetHandleByPciBusId_v2(bus.encode(), ctypes.byref(self.h)) == 0
            if not ok and lib.nvmlDeviceGetHandleByIndex_v2(torch_device, ctypes.byref(self.h)) != 0:
                raise RuntimeError("no NVML handle")
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = float(mx.value)
            self.get_reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                lib.nvmlDeviceGetCurrentClocksThrottleReasons
        except Exception as e:  # noqa: BLE001
            self.error = str(e)

    def _run(self):
        import ctypes
        clk = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        while not self._stop.is_set():
            if self.lib.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(clk)) == 0:
                r = rs.value if self.get_reasons(self.h, ctypes.byref(rs)) == 0 else 0
                self.samples.append((float(clk.value), int(r)))
            self._stop.wait(0.002)

    def __enter__(self):
        import threading
        if self.error is None:
            self._thread = threading.Thread(target=self._run, daemon=True)
            self._thread.start()
        return self

    def __exit__(self, *exc):
        self._stop.set()
        if self._thread is not None:
            self._thread.join(timeout=2)

    def summary(self):
        if self.error is not None or not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [],
                    "samples": 0, "source": f"nvml unavailable: {self.error}"}
        reasons = set()
        for _, r in self.samples:
            for bit, name in self.REASONS.items():
                if r & bit:
                    reasons.add(name)
        return {"sm_mhz": statistics.median(c for c, _ in self.samples),
                "sm_max_mhz": self.max_mhz, "reasons": sorted(reasons),
                "samples": len(self.samples), "source": "nvml, 2 ms, timed region"}


# --------------------------------------------------------------------- ours

def _to_dev(a, dev):
    import torch
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev)
    return torch.from_numpy(a).to(dev)


def _to_pinned(a):
    import torch
    t = (torch.from_numpy(a.view(np.int16)).view(torch.bfloat16) if a.dtype == np.uint16
         else torch.from_numpy(a))
    return t.pin_memory()


def measure(args, cfg: int, batch: int, rank: int, world: int, local_rank: int,
            dense_first: int = 0, n: int | None = None):
    """Times one workload on this rank's GPU.  Returns (result, w, extra) on
    rank 0 (None elsewhere); extra holds the last timed step's outputs and
    what the oracle leg needs to rebuild the index it searched."""
    import torch
    from paper_2608_08340_gb300.index import Index

    dev = torch.device("cuda", local_rank)
    dense_first = dense_first if cfg == 3 else 0
    w = workloads.config(cfg, batch=batch, n=n)
    idx = Index(_to_dev(w.E_data, dev))
    if cfg == 3:
        idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
        idx.gather_lexical(bool(args.lex_gather))
        q_indptr = torch.from_numpy(w.q_indptr).to(dev)
        q_terms = torch.from_numpy(w.q_terms).to(dev)
    idx.force_block_n(args.block_n or None)
    idx.force_path(None if args.path == "auto" else args.path)
    idx.force_pair(None if args.pair == "auto" else args.pair)
    idx.reserve(w.q, w.k)
    use_graph = args.graph and cfg in (0, 1, 2)
    prev_stream = torch.cuda.current_stream()
    if use_graph:
        from paper_2608_08340_gb300 import _lib
        idx.set_option(_lib.OPRAG_OPT_GRAPH, 1)
        side = torch.cuda.Stream()
        side.wait_stream(prev_stream)
        torch.cuda.set_stream(side)              # every launch of the run goes to it
    idx.enable_timing(True)
    Q = _to_dev(w.Q_data, dev)
    Qh = _to_pinned(w.Q_data)
    ids = torch.empty((w.q, w.k), dtype=torch.int64, device=dev)
    scores = torch.empty((w.q, w.k), dtype=torch.float32, device=dev)
    ids_h = torch.empty((w.q, w.k), dtype=torch.int64).pin_memory()
    scores_h = torch.empty((w.q, w.k), dtype=torch.float32).pin_memory()
    ups = []
    if cfg == 4:
        for r in range(4):
            u_ids, u_rows = workloads.upsert_batch(w.n, w.d, 4096, r + 1, w.dtype)
            ups.append((u_ids, u_rows, _to_dev(u_rows, dev), _to_pinned(u_rows)))
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()      # the side stream in graph mode
    last = {}

    def step(i, host=False):
        if cfg == 4:
            u_ids, _, u_dev, u_host = ups[i % len(ups)]
            idx.upsert(u_ids, u_host if host else u_dev)
        if host:
            idx.search_host(Qh, w.k, out=(ids_h, scores_h))
        elif cfg == 3 and dense_first:
            last["out"] = idx.hybrid_search_dense_first(Q, q_indptr, q_terms, w.alpha,
                                                        dense_first, w.k)
        elif cfg == 3:
            last["out"] = idx.hybrid_search(Q, q_indptr, q_terms, w.alpha, w.k)
        else:
            idx.search(Q, w.k, out=(ids, scores))
            last["out"] = (ids, scores)

    # our kernels per step: search + merge; k > 32 over many tiles adds the
    # sampled first pass (search + merge); config 3 adds the BM25 pass
    # (dense-first: the rerank), config 4 the upsert scatter.
    for i in range(args.warmup):
        flush.zero_()
        step(i)
    torch.cuda.synchronize()
    idx.check()
    t = idx.last_timing()
    sampled = t["sample_ms"] > 0.0
    launches_per_step = 2 + (2 if sampled else 0) + (1 if cfg in (3, 4) else 0)

    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    # Timed steps: enqueued back to back (the host runs ahead of the device,
    # nothing waits between steps), each bracketed by CUDA events on the
    # launching stream; the L2 flush sits between the events of two steps.
    idx.enable_timing(False)
    marks = []
    with ClockSampler(local_rank) as smi, NvmlSampler(local_rank) as clocks:
        for i in range(args.steps):
            flush.zero_()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            step(i)
            b.record(stream)
            marks.append((a, b))
        torch.cuda.synchronize()
    step_ms = [a.elapsed_time(b) for a, b in marks]
    if world > 1:
        torch.distributed.barrier()
    idx.check()
    # The last timed step's outputs, kept for the oracle leg.
    out_ids, out_scores = (x.cpu().numpy() for x in last["out"])

    # Per-kernel breakdown (roofline): the same steps again with events around
    # each kernel of the search; these events also separate the launches, so
    # they are not used for the step time.
    idx.enable_timing(True)
    tim = {"search_ms": [], "merge_ms": [], "lexical_ms": [], "sample_ms": []}
    for i in range(min(args.steps, 50)):
        flush.zero_()
        step(i)
        t = idx.last_timing()              # waits for this step
        for key in tim:
            tim[key].append(t[key])
    idx.enable_timing(False)
    idx.check()

    phases = phase_breakdown(idx, step, flush, min(args.steps, 20)) if args.phases else None

    # What two CUDA events with nothing between them read after the same
    # flush: part of every event-timed kernel duration that is not the
    # kernel's work (reported beside the kernel time, not subtracted).
    ev_pair = []
    for _ in range(20):
        flush.zero_()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        b.record(stream)
        ev_pair.append((a, b))
    torch.cuda.synchronize()
    ev_pair_us = statistics.median(a.elapsed_time(b) for a, b in ev_pair) * 1e3

    # Warm-L2 figure, reported beside the flushed one: the same steps back to
    # back with no flush in between (a corpus under 129 MB stays in L2).
    warm_marks = []
    for i in range(min(args.steps, 50)):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        step(i)
        b.record(stream)
        warm_marks.append((a, b))
    torch.cuda.synchronize()
    warm_ms = [a.elapsed_time(b) for a, b in warm_marks]
    # Upsert alone (config 4): 4096 rows scattered into the resident index.
    upsert_ms = []
    if cfg == 4:
        for i in range(min(args.steps, 20)):
            _, _, u_dev, _ = ups[i % len(ups)]
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            idx.upsert(ups[i % len(ups)][0], u_dev)
            b.record(stream)
            upsert_ms.append((a, b))
        torch.cuda.synchronize()
        upsert_ms = [a.elapsed_time(b) for a, b in upsert_ms]
    idx.check()

    # end to end: host queries in, host results out, through the C ABI
    e2e_ms = []
    if cfg != 3:
        for i in range(args.warmup):
            step(i, host=True)
        for i in range(args.steps):
            flush.zero_()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            step(i, host=True)                 # synchronous call
            e2e_ms.append((time.perf_counter() - t0) * 1e3)
    else:
        # hybrid: copy queries and terms in, read results out, around the call
        for i in range(args.steps + args.warmup):
            flush.zero_()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            Qd = Qh.to(dev, non_blocking=True)
            qi = torch.from_numpy(w.q_indptr).to(dev, non_blocking=True)
            qt = torch.from_numpy(w.q_terms).to(dev, non_blocking=True)
            if dense_first:
                r_ids, r_sc = idx.hybrid_search_dense_first(Qd, qi, qt, w.alpha, dense_first,
                                                            w.k)
            else:
                r_ids, r_sc = idx.hybrid_search(Qd, qi, qt, w.alpha, w.k)
            ids_h.copy_(r_ids)
            scores_h.copy_(r_sc)
            torch.cuda.synchronize()
            if i >= args.warmup:
                e2e_ms.append((time.perf_counter() - t0) * 1e3)

    total_ms, e2e_total = slowest_replica([sum(step_ms), sum(e2e_ms)], world, dev)
    quality = None
    if dense_first and rank == 0:
        # Quality against the full hybrid search (Sec. 5.2 Recall@k; Jaccard
        # overlap of the two top-k sets), as the paper reports for this policy.
        f_ids, _ = idx.hybrid_search(Q, q_indptr, q_terms, w.alpha, w.k)
        d_ids, _ = idx.hybrid_search_dense_first(Q, q_indptr, q_terms, w.alpha, dense_first, w.k)
        f_ids, d_ids = f_ids.cpu().numpy(), d_ids.cpu().numpy()
        inter = [len(set(a) & set(b)) for a, b in zip(f_ids.tolist(), d_ids.tolist())]
        union = [len(set(a) | set(b)) for a, b in zip(f_ids.tolist(), d_ids.tolist())]
        quality = {"recall_at_k": float(np.mean(inter)) / w.k,
                   "jaccard": float(np.mean([i / u for i, u in zip(inter, union)])),
                   "vs": "full hybrid search on the same batch", "n_candidates": dense_first}
    path, launch = idx.last_path, idx.last_launch
    idx.close()
    if use_graph:
        torch.cuda.set_stream(prev_stream)
    del flush
    torch.cuda.empty_cache()
    if rank != 0:
        return None

    nbytes, flops = roofline_terms(w, cfg, dense_first)
    hbm, tflops_burst, tflops_sustained, peak_src = peaks()
    # The burst figure is for a kernel timed alone; when the timed loop kept
    # the GPU at its power cap (NVML reported sw_power_cap while it ran), the
    # sustained figure (the same GEMM back to back under the cap) applies.
    clk = clocks.summary()
    capped = "sw_power_cap" in clk.get("reasons", [])
    tflops = tflops_sustained if capped else tflops_burst
    t_kernel = statistics.mean(tim["search_ms"]) * 1e-3
    t_bytes = nbytes / (hbm * 1e9)
    t_flops = flops / (tflops * 1e12)
    if t_flops > t_bytes and w.dtype == "bf16":
        roof = {"bound": "tensor", "achieved": flops / t_kernel / 1e12, "peak": tflops,
                "unit": "TFLOP/s"}
    else:
        roof = {"bound": "hbm", "achieved": nbytes / t_kernel / 1e9, "peak": hbm, "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["peak_source"] = f"{peak_src} (MEASURED_PEAKS.json)" if peak_src == "measured" else peak_src
    if roof["bound"] == "tensor":
        roof["peak_kind"] = ("sustained: sw_power_cap active in the timed region" if capped
                             else "burst")
    roof["kernel"] = "tc_search_kernel" if path == "tc" else "simt_search_kernel"
    roof["kernel_ms_mean"] = statistics.mean(tim["search_ms"])
    roof["kernel_ms_median"] = statistics.median(tim["search_ms"])
    roof["event_pair_us"] = ev_pair_us
    roof["merge_ms_mean"] = statistics.mean(tim["merge_ms"])
    roof["merge_ms_median"] = statistics.median(tim["merge_ms"])
    if sampled:
        # k > 32: the first pass over every 32nd corpus tile and its merge,
        # timed apart from the main pass (the dominant kernel above)
        roof["sample_pass_ms_mean"] = statistics.mean(tim["sample_ms"])
        roof["sample_pass_ms_median"] = statistics.median(tim["sample_ms"])
        roof["sample_pass_ms_max"] = max(tim["sample_ms"])
    if cfg == 3 and not dense_first:
        roof["bm25_ms_mean"] = statistics.mean(tim["lexical_ms"])
        roof["sparse"] = sparse_terms(w)
    roof["algorithmic_bytes"] = nbytes
    roof["algorithmic_flops"] = flops
    # the whole step against the roofline of its algorithmic work
    roof["step_frac"] = max(t_bytes, t_flops) / (statistics.mean(step_ms) * 1e-3)
    roof["traffic"] = ncu_traffic(workload_key(cfg, w.q))

    queries_all = w.q * args.steps * world
    h2d = w.q * w.d * (2 if w.dtype == "bf16" else 4)
    if cfg == 4:
        h2d += 4096 * (w.d * 2 + 8)
    if cfg == 3:
        h2d += w.q_indptr.nbytes + w.q_terms.nbytes
    d2h = w.q * w.k * 12
    lex_form = None
    if cfg == 3 and not dense_first:
        lex_form = ("gathered in the search epilogue (no BM25 block)" if args.lex_gather else
                    "materialised q x n BM25 block read by the search epilogue")
    result = {
        "metric": f"queries/s at top-{w.k}", "value": job_rate(w.q, args.steps, world, total_ms),
        "unit": "queries/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": total_ms / args.steps,
        "ms_per_step_median": statistics.median(step_ms), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": config_dict(cfg, w, world, dense_first),
        "roofline": roof,
        "e2e": {"value": queries_all / (e2e_total * 1e-3), "unit": "queries/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "api": ("oprag_search_host" if cfg != 3 else
                        "oprag_hybrid_search_dense_first + torch copies" if dense_first else
                        "oprag_hybrid_search + torch copies")},
        "warm_l2": {"value": w.q / (statistics.median(warm_ms) * 1e-3), "unit": "queries/s",
                    "ms_per_step_median": statistics.median(warm_ms), "steps": len(warm_ms),
                    "l2": "not flushed between steps"},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": dict(clk, smi=smi.summary()),
        "path": path, "launch": launch, "graph_mode": bool(use_graph),
    }
    if upsert_ms:
        # Sec. 3.2 Op_upsert: 4096 rows of d bf16 plus their int64 ids per call.
        ub = 4096 * (w.d * 2 + 8)
        result["upsert"] = {"rows": 4096, "bytes": ub, "ms_median": statistics.median(upsert_ms),
                            "GB_per_s": ub / (statistics.median(upsert_ms) * 1e-3) / 1e9}
    if quality:
        result["quality"] = quality
    if phases:
        result["phases"] = phases
    if lex_form:
        result["lexical"] = lex_form
    extra = {"ids": out_ids, "scores": out_scores,
             "upserts": ([(ups[r][0], ups[r][1]) for r in upsert_sequence(args.warmup, args.steps)]
                         if cfg == 4 else [])}
    return result, w, extra


def phase_breakdown(idx, step, flush, n_steps: int) -> dict:
    """Per-CTA global-timer stamps of the main search pass over n_steps
    flushed steps: for each mark, the earliest, median and latest CTA in
    microseconds after the earliest CTA entry (median over the steps), next
    to the same steps' event-timed kernel duration."""
    idx.enable_phases(True)
    idx.enable_timing(True)
    per = {name: [] for name in idx.PHASES}
    ev = []
    for i in range(n_steps):
        flush.zero_()
        step(i)
        ev.append(idx.last_timing()["search_ms"] * 1e3)
        st = idx.last_phases()
        t0 = st[:, 0][st[:, 0] > 0].min()
        for m, name in enumerate(idx.PHASES):
            col = st[:, m]
            col = col[col > 0]
            if col.size:
                rel = (col - t0) / 1e3
                per[name].append((float(rel.min()), float(np.median(rel)), float(rel.max())))
    idx.enable_phases(False)
    idx.enable_timing(False)
    out = {"unit": "us after the first CTA entry (global timer); min / median / max over CTAs, "
                   "median over steps",
           "steps": n_steps, "ctas": int(st.shape[0]),
           "kernel_event_us_median": float(np.median(ev))}
    for name, v in per.items():
        if v:
            a = np.asarray(v)
            out[name] = [round(float(np.median(a[:, c])), 2) for c in range(3)]
    return out


def sub_entry(res: dict) -> dict:
    """The fields of a workload's line kept under the headline's "configs"."""
    keep = ("value", "unit", "ms_per_step", "ms_per_step_median", "roofline", "e2e", "clocks",
            "warm_l2", "parity", "gpu_launches", "path", "launch", "upsert", "metric", "phases",
            "lexical")
    out = {k: res[k] for k in keep if k in res}
    out["workload"] = res["config"]["workload"]
    return out


# --------------------------------------------------------------------- oracle leg

def parity_check(w, cfg: int, extra: dict, threads: int) -> dict:
    """The last timed step's outputs against the CPU oracle (oracle/check.py
    rules: scores within 1e-4, ids exact outside near-tie blocks) on the rows
    of parity_rows(); for the scale workload the oracle searches the index as
    the timed upserts left it."""
    import oracle
    from oracle import check

    rows = parity_rows(w.q, seed=cfg)
    E = w.E_data
    if extra["upserts"]:
        E = E.copy()
        for u_ids, u_rows in extra["upserts"]:
            oracle.upsert(E, u_ids, u_rows)
    Qs = w.Q_data[rows]
    if cfg == 3:
        qts = [w.q_terms[w.q_indptr[r]:w.q_indptr[r + 1]] for r in rows]
        qip = np.zeros(len(rows) + 1, np.int32)
        qip[1:] = np.cumsum([len(t) for t in qts])
        qtm = np.concatenate(qts).astype(np.int32)

        def fn(kout):
            return oracle.hybrid_search(E, Qs, w.doc_indptr, w.doc_terms, w.vocab, qip, qtm,
                                        w.alpha, kout, w.k1, w.b, nthreads=threads)
    else:
        def fn(kout):
            return oracle.search(E, Qs, kout, nthreads=threads)
    t0 = time.perf_counter()
    out = {"rows_checked": int(len(rows)), "of": int(w.q),
           "sample": ("every query" if len(rows) == w.q else
                      "one random query in every 32-query group of every 128-query tile"),
           "tol": TOL}
    try:
        o_ids, o_sc = check.topk_with_margin(fn, w.k, w.n, TOL)
        stats = check.check_topk(extra["ids"][rows], extra["scores"][rows], o_ids, o_sc, w.k,
                                 TOL, n=w.n, query_index=rows, label=workload_key(cfg, w.q))
        out.update(passed=True, exact_id_lists=stats["exact_id_lists"],
                   max_abs_score_err=stats["max_abs_score_err"])
    except check.TopkMismatch as e:
        out.update(passed=False, error=str(e)[:400])
    out["oracle_s"] = round(time.perf_counter() - t0, 2)
    return out


def oracle_queries_per_s(w, cfg, nq: int, threads: int, offset: int = 0):
    import oracle
    rows = (np.arange(nq) + offset) % w.q
    Qs = w.Q_data[rows]
    t0 = time.perf_counter()
    if cfg == 3:
        qts = [w.q_terms[w.q_indptr[r]:w.q_indptr[r + 1]] for r in rows]
        qip = np.zeros(nq + 1, np.int32)
        qip[1:] = np.cumsum([len(t) for t in qts])
        oracle.hybrid_search(w.E_data, Qs, w.doc_indptr, w.doc_terms, w.vocab, qip,
                             np.concatenate(qts).astype(np.int32), w.alpha, w.k, w.k1, w.b,
                             nthreads=threads)
    else:
        oracle.search(w.E_data, Qs, w.k, nthreads=threads)
    return nq / (time.perf_counter() - t0)


def cpu_baseline(w, cfg, budget_s: float = 12.0):
    """The oracle as it stands, on all host cores, on a bounded sample sized
    from a short pilot to about budget_s seconds."""
    threads = os.cpu_count() or 1
    pilot = threads
    rate = oracle_queries_per_s(w, cfg, pilot, threads)
    nq = int(min(max(pilot, rate * budget_s), 4 * w.q))
    nq = max(threads, nq // threads * threads)
    rate = oracle_queries_per_s(w, cfg, nq, threads, offset=pilot)
    return {"value": rate, "unit": "queries/s", "cores": threads, "kind": "oracle",
            "sample": f"{nq} queries of the same workload (rows taken cyclically), full "
                      f"fp64 scoring + full sort per query, {threads} threads"}


def run_reference(args):
    """The reference arm: the oracle (the CPU definition of the path) on the
    host cores, on bounded samples of the same workload and config as ours.
    The scale workload's step applies its 4096-row upsert to the oracle's
    array before searching, as ours does."""
    import oracle
    cfg = HEADLINE[0] if args.config is None else args.config
    batch = args.batch or (HEADLINE[1] if args.config is None else default_batch(cfg))
    w = workloads.config(cfg, batch=batch)
    threads = os.cpu_count() or 1
    E = w.E_data.copy() if cfg == 4 else w.E_data
    ups = [workloads.upsert_batch(w.n, w.d, 4096, r + 1, w.dtype) for r in range(4)] if cfg == 4 else []
    ww = workloads.Workload(w.name, w.dtype, w.k, E, w.Q_data, w.doc_indptr, w.doc_terms,
                            w.q_indptr, w.q_terms, w.vocab, w.k1, w.b, w.alpha)
    # each step: a bounded sample of the step's queries (whole run within minutes)
    pilot = oracle_queries_per_s(ww, cfg, threads, threads)
    per_step = int(max(threads, min(w.q, pilot * 2.0)) // threads * threads)

    def one(i, nq):
        if ups:
            u_ids, u_rows = ups[i % len(ups)]
            oracle.upsert(E, u_ids, u_rows)
        oracle_queries_per_s(ww, cfg, nq, threads, offset=i * nq)

    for i in range(args.warmup):
        one(i, threads)
    times, done = [], 0
    for i in range(args.steps):
        t0 = time.perf_counter()
        one(i, per_step)
        times.append(time.perf_counter() - t0)
        done += per_step
    value = done / sum(times)
    out = {
        "impl": "reference", "metric": f"queries/s at top-{w.k}", "value": value,
        "unit": "queries/s", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * sum(times) / len(times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_dict(cfg, w, args.gpus),
        "cpu_baseline": {"value": value, "unit": "queries/s", "cores": threads,
                         "kind": "oracle",
                         "sample": f"{per_step} queries per step of the {w.q}-query batch"
                                   + (", after the step's 4096-row upsert" if ups else "")},
        "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out))


def run_embed_tail(args):
    """Embedding tail (Sec. 4.3): rows/s and HBM roofline of oprag_embed_pool on a
    synthetic padded batch (lengths uniform in [T/4, T])."""
    import torch
    from paper_2608_08340_gb300.index import embed_pool

    torch.cuda.set_device(0)
    b, t, d = 256, 512, 4096
    g = torch.Generator(device="cuda").manual_seed(5000)
    hidden = torch.randn((b, t, d), generator=g, device="cuda").to(torch.bfloat16)
    rng = np.random.default_rng(5001)
    lens = rng.integers(t // 4, t + 1, b)
    mask = torch.from_numpy((np.arange(t)[None, :] < lens[:, None]).astype(np.uint8)).cuda()
    for _ in range(args.warmup):
        embed_pool(hidden, mask)
    torch.cuda.synchronize()
    marks = []
    for _ in range(args.steps):
        a = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        a.record()
        embed_pool(hidden, mask)
        e.record()
        marks.append((a, e))
    torch.cuda.synchronize()
    ms = [a.elapsed_time(e) for a, e in marks]
    t_step = statistics.mean(ms) * 1e-3
    # bytes the kernel must move: the unmasked hidden states, the mask, the output
    nbytes = int(lens.sum()) * d * 2 + b * t + b * d * 2
    hbm = peaks()[0]
    print(json.dumps({
        "metric": "embedded rows/s (masked mean pool + L2 normalise)", "value": b / t_step,
        "unit": "rows/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": statistics.mean(ms), "higher_is_better": True, "dtype": "bf16",
        "data": "synthetic", "scaling": "weak", "vs_baseline": None,
        "config": {"workload": f"embedding tail: {b} rows x {t} tokens x {d} bf16, lengths "
                               f"uniform in [{t // 4}, {t}]",
                   "l2": "input (1 GiB) larger than L2"},
        "roofline": {"bound": "hbm", "achieved": nbytes / t_step / 1e9, "peak": hbm,
                     "unit": "GB/s", "frac": nbytes / t_step / 1e9 / hbm,
                     "algorithmic_bytes": nbytes, "kernel": "embed_pool_kernel"},
        "gpu_launches": args.steps}))


def run_index_ops(args):
    """Index updates (Sec. 3.2 Op_upsert, Sec. 4.4 memory index): append
    (rows/s), token-bag replacement (wall time of the rebuild), and the
    knowledge + memory search against the knowledge search alone."""
    import torch
    from paper_2608_08340_gb300.index import Index, search_two

    torch.cuda.set_device(0)
    w = workloads.config(3, batch=256)
    dev = torch.device("cuda", 0)
    to_dev = lambda a: torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev)
    out = {}
    # append: a 32768-chunk index grows by 4096 rows per step
    rows = to_dev(workloads.upsert_batch(w.n, w.d, 4096, 1, "bf16")[1])
    idx = Index(to_dev(w.E_data))
    idx.append(rows)                             # first growth (doubling) outside the timing
    times = []
    for _ in range(args.steps):
        a = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        a.record()
        idx.append(rows)
        e.record()
        torch.cuda.synchronize()
        times.append(a.elapsed_time(e))
    out["append_4096_rows_ms"] = statistics.median(times)
    out["append_rows_per_s"] = 4096 / (statistics.median(times) * 1e-3)
    out["index_rows_after"] = idx.n
    idx.close()
    # token bags: 4096 chunks get new bags, BM25 rebuilt on the host and uploaded
    idx = Index(to_dev(w.E_data))
    idx.set_sparse(w.doc_indptr, w.doc_terms, w.vocab, w.k1, w.b)
    rng = np.random.default_rng(6000)
    ids = rng.choice(w.n, 4096, replace=False)
    bip = (w.doc_indptr[ids + 1] - w.doc_indptr[ids]).cumsum()
    bip = np.concatenate([[0], bip]).astype(np.int32)
    btm = rng.choice(w.doc_terms, int(bip[-1])).astype(np.int32)
    times = []
    for _ in range(max(3, args.steps // 10)):
        t0 = time.perf_counter()
        idx.update_sparse(ids, bip, btm)
        times.append((time.perf_counter() - t0) * 1e3)
    out["update_4096_bags_ms"] = statistics.median(times)
    idx.close()
    # knowledge (32768) + memory (8192) search of 256 queries against knowledge alone
    kn = Index(to_dev(w.E_data))
    mem_rows = workloads.config(1, n=8192, batch=1).E_data
    mem = Index(to_dev(mem_rows))
    stacked = Index(to_dev(np.concatenate([w.E_data, mem_rows])))
    Q = to_dev(workloads.config(1, batch=256).Q_data)
    for label, fn in (("search_knowledge_ms", lambda: kn.search(Q, w.k)),
                      ("search_two_ms", lambda: search_two(kn, mem, Q, w.k)),
                      ("search_stacked_40960_ms", lambda: stacked.search(Q, w.k))):
        for _ in range(args.warmup):
            fn()
        marks = []
        for _ in range(args.steps):
            a = torch.cuda.Event(enable_timing=True)
            e = torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            e.record()
            marks.append((a, e))
        torch.cuda.synchronize()
        out[label] = statistics.median(a.elapsed_time(e) for a, e in marks)
    print(json.dumps({"metric": "index update timings", "unit": "ms", "n_gpus": 1,
                      "steps": args.steps, "warmup": args.warmup, "data": "synthetic",
                      "config": {"workload": "32768 x 768 bf16 knowledge index, 8192-row memory "
                                             "index, 256 queries, 4096-row updates"},
                      "results": out}))


def main():
    args = parse()
    if args.embed_tail and args.impl == "ours":
        run_embed_tail(args)
        return
    if args.index_ops and args.impl == "ours":
        run_index_ops(args)
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            run_reference(args)
        return
    import torch
    torch.cuda.set_device(local_rank)
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    oracle_leg = not args.no_cpu_baseline and rank == 0
    threads = os.cpu_count() or 1
    if args.config is None:
        plan = [HEADLINE] + SUB_WORKLOADS
    else:
        plan = [(args.config, args.batch or default_batch(args.config))]
    head = None
    subs = {}
    for n_run, (cfg, batch) in enumerate(plan):
        res = measure(args, cfg, batch, rank, world, local_rank,
                      dense_first=args.dense_first if n_run == 0 else 0,
                      n=args.n if args.config is not None else None)
        if res is None:
            continue
        result, w, extra = res
        if oracle_leg:
            result["parity"] = parity_check(w, cfg, extra, threads)
            if n_run == 0:
                result["cpu_baseline"] = cpu_baseline(w, cfg)
        if n_run == 0:
            head = result
        else:
            subs[workload_key(cfg, batch)] = sub_entry(result)
        del w, extra
    if world > 1:
        torch.distributed.destroy_process_group()
    if head is None:
        return
    if subs:
        head["configs"] = subs
    print(json.dumps(head))


if __name__ == "__main__":
    main()
