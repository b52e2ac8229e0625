"""Throughput of the intent-driven parameter manager on one or more GB300s.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload mf|micro|complex|sgns|tiny_mf]
                    [--impl ours|reference]

A step is one clock of the whole job: every worker slot signals the intent of
the batch `lookahead` clocks ahead, reads and writes the rows of its current
batch (pull + push, or one fused training step that reads through the slot
map and pushes its delta rows), advances its clock; then one sync merges all
replica updates (the per-clock loop of Fig. 2).  Inputs are seeded synthetic
data resident in HBM before timing starts; the stores (9-26 GB) and per-step
row traffic exceed the 129 MB L2, so no flush is needed between steps.

Reported (one JSON line on rank 0): pulled + pushed keys/s (value), training
samples/s, per-operation device time and algorithmic GB/s, the roofline of
the dominant kernel against the measured HBM copy peak, the end-to-end rate
through the C ABI with pinned host buffers (host<->device copies timed), the
CPU oracle's rate on a bounded sample (one thread), SM clocks sampled during
the timed region, and the number of library kernels launched in it.  With the
MF workload (the default) the same line carries a `micro` record: the
parameter-access microbenchmark (100M keys x 64 floats, 2^20 Zipf(1.1) keys
per worker and clock, span 1) measured the same way, with pull, push and sync
against the HBM roofline (--micro-zipf adds other exponents as `micro_sweep`).

With --gpus N > 1 (torchrun) every rank runs an independent replica of the
workload on its own GPU: the path has no exchange step (replicas only).
"""
import argparse
import json
import math
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

# The CPU oracle baseline is a one-core figure: numpy's BLAS and OpenMP pools are held to one thread
# (set before numpy is imported; the GPU path does no numerical work on the host).
ORACLE_THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS",
                      "VECLIB_MAXIMUM_THREADS", "NUMEXPR_NUM_THREADS")
for _v in ORACLE_THREAD_VARS:
    os.environ[_v] = "1"

import numpy as np  # noqa: E402
import torch  # noqa: E402

from synth import hashgen  # noqa: E402
from synth import workloads as wl  # noqa: E402

METRIC = "pulled+pushed keys/s and training samples/s on 1 GB300; % of HBM roofline"

# DRAM bytes (read + write) of the push scatter kernels (push_chunks + push_combine) per pushed row, per
# workload, from the one-pass ncu captures summarised in profiles/ (each on a smaller case of the same
# workload, scaled by rows); a figure stands for the kernels only while their source is the one captured
# (source_digest: first 16 hex digits of the sha256 of their code without comments), otherwise the traffic
# is reported as null.
PUSH_SOURCES = ("paper_2206_00470_gb300/csrc/push.cu", "paper_2206_00470_gb300/csrc/rowgroup.cuh")
PUSH_TRAFFIC = {
    "mf": {"bytes_per_row": 79.106e6 / 65536, "sha256_16": "b7ebddd50ef3a39f"},   # profiles/push_scatter_mf_2Mx200K.md
    "micro": {"bytes_per_row": None, "sha256_16": None},
}


def source_digest(paths):
    """sha256 (16 hex digits) of CUDA sources with their // comments and blank lines removed, so that
    a change to comments alone does not retire a recorded capture."""
    import hashlib
    import re
    code = []
    for path in paths:
        with open(path) as f:
            text = f.read()
        lines = [re.sub(r"//.*$", "", ln).rstrip() for ln in text.splitlines()]
        code.append("\n".join(ln for ln in lines if ln.strip()))
    return hashlib.sha256("\n".join(code).encode()).hexdigest()[:16]


def recorded_traffic(workload, rows_per_launch):
    rec = PUSH_TRAFFIC.get(workload)
    if not rec or rec["bytes_per_row"] is None:
        return None
    try:
        digest = source_digest([os.path.join(ROOT, p) for p in PUSH_SOURCES])
    except OSError:
        return None
    if digest != rec["sha256_16"]:
        return None
    return rec["bytes_per_row"] * rows_per_launch


UNIT = "keys/s"


# ---------------------------------------------------------------------------
# distributed plumbing (timing only; the data path has no collective)
# ---------------------------------------------------------------------------
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def init_dist(ws, backend):
    if ws > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, ws, device):
    if ws == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x, ws, device):
    if ws == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)),
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# workloads
# ---------------------------------------------------------------------------
def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


class Micro:
    """Parameter-access microbenchmark: 100M keys x 64 fp32, Zipf keys, pull + push per worker."""

    def __init__(self, args, device):
        import dataclasses
        self.cfg = dataclasses.replace(wl.MICRO, batch=args.batch or wl.MICRO.batch,
                                       zipf_s=args.zipf if args.zipf is not None else wl.MICRO.zipf_s,
                                       span=args.span or wl.MICRO.span,
                                       num_keys=args.keys or wl.MICRO.num_keys)
        c = self.cfg
        self.device = device
        self.K, self.D, self.W = c.num_keys, c.value_len, c.workers
        self.lookahead, self.span = c.lookahead, c.span
        self.row = self.D * 4
        self.capacity = min(self.W * (c.span + 1) * c.batch, 80_000_000)
        self.samples_per_step = 0

    def config(self):
        c = self.cfg
        return {"workload": c.name, "num_keys": c.num_keys, "value_len": c.value_len,
                "workers": c.workers, "batch_per_worker": c.batch, "zipf_s": c.zipf_s,
                "intent_span": c.span, "lookahead": c.lookahead}

    def init_store(self):
        return hashgen.init_store_torch(self.K, self.D, self.D, self.cfg.seed, self.cfg.init_std,
                                        self.device, chunk_rows=1 << 22)

    def prepare(self, clocks):
        c = self.cfg
        self.keys = {}
        for cl in range(clocks + self.lookahead + 1):
            for w in range(self.W):
                self.keys[(w, cl)] = wl.micro_keys(c, w, cl, self.device).to(torch.int32)
        g = torch.Generator(device=self.device).manual_seed(c.seed + 5)
        self.deltas = [torch.randn((c.batch, self.D), generator=g, device=self.device) * c.delta_std
                       for _ in range(self.W)]
        self.out = torch.empty((c.batch, self.D), device=self.device)

    def start(self, pm):
        for w in range(self.W):
            for j in range(self.lookahead):
                pm.intent(w, self.keys[(w, j)], j, j + self.span)

    def step(self, pm, cl):
        for w in range(self.W):
            j = cl + self.lookahead
            pm.intent(w, self.keys[(w, j)], j, j + self.span)
            k = self.keys[(w, cl)]
            pm.pull(w, k, out=self.out)
            pm.push(w, k, self.deltas[w])
            pm.advance_clock(w)
        pm.sync()

    def keys_per_step(self):
        return 2 * self.W * self.cfg.batch     # pulled + pushed

    # host-buffer variant for the end-to-end number
    def prepare_host(self, clocks):
        self.hkeys = {(w, c): self.keys[(w, c)].cpu().pin_memory() for c in clocks
                      for w in range(self.W) if (w, c) in self.keys}
        self.hdeltas = [d.cpu().pin_memory() for d in self.deltas]
        self.hout = torch.empty((self.cfg.batch, self.D), pin_memory=True)

    def step_host(self, pm, cl):
        for w in range(self.W):
            j = cl + self.lookahead
            pm.intent(w, self.hkeys[(w, j)], j, j + self.span)
            k = self.hkeys[(w, cl)]
            pm.pull(w, k, out=self.hout)
            pm.push(w, k, self.hdeltas[w])
            pm.advance_clock(w)
        pm.sync()

    def host_bytes_per_step(self):
        b = self.cfg.batch
        h2d = self.W * (b * 4 * 3 + b * self.D * 4)   # intent keys, pull keys, push keys, deltas
        d2h = self.W * b * self.D * 4                  # pulled rows
        return h2d, d2h


class MF:
    """Matrix factorisation 10M x 1M, rank 100 + AdaGrad: fused MF step per worker per clock."""

    def __init__(self, args, device, cfg=None):
        import dataclasses
        if cfg is None:
            cfg = dataclasses.replace(wl.MF, rows=args.mf_rows or wl.MF.rows, cols=args.mf_cols or wl.MF.cols,
                                      batch=args.batch or wl.MF.batch)
        self.cfg = cfg
        c = self.cfg
        self.device = device
        self.K, self.D, self.W = c.num_keys, c.value_len, c.workers
        self.lookahead, self.span = c.lookahead, c.span
        self.row = self.D * 4
        # live replicas per worker: the distinct keys of one batch (2 per cell at most)
        self.capacity = min(self.W * self.K, self.W * 4 * c.batch, 80_000_000)
        self.samples_per_step = self.W * c.batch

    def config(self):
        c = self.cfg
        return {"workload": c.name, "rows": c.rows, "cols": c.cols, "rank": c.rank,
                "adagrad": c.adagrad, "workers": c.workers, "batch_per_worker": c.batch,
                "zipf_s": c.zipf_s, "lookahead": c.lookahead, "intent_span": c.span, "lr": c.lr}

    def init_store(self):
        c = self.cfg
        return hashgen.init_store_torch(self.K, self.D, c.rank, c.seed, c.init_std, self.device,
                                        chunk_rows=1 << 21)

    def prepare(self, clocks):
        c = self.cfg
        self.data = {}
        for cl in range(clocks + self.lookahead + 1):
            for w in range(self.W):
                r, co, v = wl.mf_batch(c, w, cl, self.device)
                self.data[(w, cl)] = (r.to(torch.int32), co.to(torch.int32), v,
                                      torch.cat([r, co]).to(torch.int32))
        self.loss = torch.zeros(self.W, dtype=torch.float64, device=self.device)

    def start(self, pm):
        for w in range(self.W):
            for j in range(self.lookahead):
                pm.intent(w, self.data[(w, j)][3], j, j + self.span)

    def step(self, pm, cl, data=None):
        c = self.cfg
        data = data or self.data
        for w in range(self.W):
            j = cl + self.lookahead
            pm.intent(w, data[(w, j)][3], j, j + self.span)
            r, co, v, _ = data[(w, cl)]
            pm.mf_step(w, r, co, v, c.rank, c.adagrad, c.lr, c.eps, loss_out=self.loss[w:w + 1])
            pm.advance_clock(w)
        pm.sync()

    def keys_per_step(self):
        return 4 * self.W * self.cfg.batch     # 2 rows read + 2 delta rows written per cell

    def step_alg_bytes(self):
        # per cell: keys + value in (12 B), 2 rows read, 2 delta rows + 2 keys written
        return self.W * self.cfg.batch * (12 + 4 * self.row + 8)

    def prepare_host(self, clocks):
        self.hdata = {(w, c): tuple(x.cpu().pin_memory() for x in self.data[(w, c)]) for c in clocks
                      for w in range(self.W) if (w, c) in self.data}
        self.hloss = torch.zeros(1, dtype=torch.float64, pin_memory=True)

    def step_host(self, pm, cl):
        c = self.cfg
        for w in range(self.W):
            j = cl + self.lookahead
            pm.intent(w, self.hdata[(w, j)][3], j, j + self.span)
            r, co, v, _ = self.hdata[(w, cl)]
            pm.mf_step(w, r, co, v, c.rank, c.adagrad, c.lr, c.eps, loss_out=self.hloss)
            pm.advance_clock(w)
        pm.sync()

    def host_bytes_per_step(self):
        b = self.cfg.batch
        h2d = self.W * (b * 8 + b * 4 + 2 * b * 4)    # rows+cols, values, intent keys
        d2h = self.W * 8                               # batch loss
        return h2d, d2h


class TinyMF(MF):
    """The tiny 1,000 x 500 rank-16 MF (plain SGD, W=4, batch 256): the parity configuration."""

    def __init__(self, args, device):
        super().__init__(args, device, cfg=wl.TINY_MF)
        self.capacity = self.K * self.W

    def init_store(self):
        c = self.cfg
        return hashgen.init_store_torch(self.K, self.D, c.rank, c.seed, c.init_std, self.device)

    def prepare(self, clocks):
        c = self.cfg
        data = wl.tiny_mf_dataset(c)
        self.data = {}
        for cl in range(clocks + self.lookahead + 1):
            for w in range(self.W):
                r, co, v = wl.tiny_mf_batch(c, data, w, cl % wl.tiny_mf_clocks(c, data[3]))
                self.data[(w, cl)] = (r.to(torch.int32).to(self.device), co.to(torch.int32).to(self.device),
                                      v.to(self.device), torch.cat([r, co]).to(torch.int32).to(self.device))
        self.loss = torch.zeros(self.W, dtype=torch.float64, device=self.device)


class ComplEx:
    """ComplEx KGE, 5M entities + 800 relations, 2x128 + AdaGrad, 100 negatives, batch 4,096."""

    def __init__(self, args, device):
        self.cfg = wl.COMPLEX
        c = self.cfg
        self.device = device
        self.K, self.D, self.W = c.num_keys, c.value_len, c.workers
        self.lookahead, self.span = c.lookahead, c.span
        self.row = self.D * 4
        per = c.batch * (3 + c.negatives)
        self.capacity = min(self.W * self.K, self.W * 2 * per, 40_000_000)
        self.samples_per_step = self.W * c.batch

    def config(self):
        c = self.cfg
        return {"workload": c.name, "entities": c.entities, "relations": c.relations,
                "complex_dim": c.half_dim, "adagrad": True, "negatives": c.negatives,
                "workers": c.workers, "batch_per_worker": c.batch, "zipf_entities": c.zipf_entities,
                "zipf_relations": c.zipf_relations, "lookahead": c.lookahead, "intent_span": c.span,
                "lr": c.lr}

    def init_store(self):
        c = self.cfg
        return hashgen.init_store_torch(self.K, self.D, c.theta_dim, c.seed, c.init_std, self.device,
                                        chunk_rows=1 << 20)

    def prepare(self, clocks):
        c = self.cfg
        self.data = {}
        for cl in range(clocks + self.lookahead + 1):
            for w in range(self.W):
                h, r, t, n = (x.to(torch.int32) for x in wl.complex_batch(c, w, cl, self.device))
                self.data[(w, cl)] = (h, r, t, n.reshape(-1), torch.cat([h, r, t, n.reshape(-1)]))
        self.loss = torch.zeros(self.W, dtype=torch.float64, device=self.device)

    def start(self, pm):
        for w in range(self.W):
            for j in range(self.lookahead):
                pm.intent(w, self.data[(w, j)][4], j, j + self.span)

    def step(self, pm, cl, data=None, loss=None):
        c = self.cfg
        data = data or self.data
        for w in range(self.W):
            j = cl + self.lookahead
            pm.intent(w, data[(w, j)][4], j, j + self.span)
            h, r, t, n, _ = data[(w, cl)]
            pm.complex_step(w, h, r, t, n, c.negatives, c.theta_dim, c.lr, c.eps,
                            loss_out=(self.loss[w:w + 1] if loss is None else loss))
            pm.advance_clock(w)
        pm.sync()

    def keys_per_step(self):
        return 2 * self.W * self.cfg.batch * (3 + self.cfg.negatives)

    def step_alg_bytes(self):
        c = self.cfg
        rows = c.batch * (3 + c.negatives)
        # keys in (4 B per row), every row read once and one delta row + key written per row
        return self.W * rows * (2 * self.row + 8)

    def prepare_host(self, clocks):
        self.hdata = {(w, cc): tuple(x.cpu().pin_memory() for x in self.data[(w, cc)]) for cc in clocks
                      for w in range(self.W) if (w, cc) in self.data}
        self.hloss = torch.zeros(1, dtype=torch.float64, pin_memory=True)

    def step_host(self, pm, cl):
        self.step(pm, cl, data=self.hdata, loss=self.hloss)

    def host_bytes_per_step(self):
        c = self.cfg
        rows = c.batch * (3 + c.negatives)
        return self.W * rows * 4 * 2, self.W * 8      # step keys + intent keys; batch loss


class SGNS:
    """Skip-gram with negative sampling, 700K vocabulary, dim 300, window 5, 25 negatives, batch 8,192."""

    def __init__(self, args, device):
        self.cfg = wl.SGNS
        c = self.cfg
        self.device = device
        self.K, self.D, self.W = c.num_keys, c.value_len, c.workers
        self.lookahead, self.span = c.lookahead, c.span
        self.row = self.D * 4
        self.n_ctx = 2 * c.window
        self.per = 1 + self.n_ctx * (1 + c.negatives)
        self.capacity = min(self.W * self.K, 40_000_000)
        self.samples_per_step = self.W * c.batch

    def config(self):
        c = self.cfg
        return {"workload": c.name, "vocab": c.vocab, "dim": c.dim, "window": c.window,
                "negatives": c.negatives, "workers": c.workers, "batch_centres_per_worker": c.batch,
                "zipf_s": c.zipf_s, "lookahead": c.lookahead, "intent_span": c.span, "lr": c.lr}

    def init_store(self):
        c = self.cfg
        return hashgen.init_store_torch(self.K, self.D, c.dim, c.seed, c.init_std, self.device,
                                        chunk_rows=1 << 20)

    def prepare(self, clocks):
        c = self.cfg
        V = c.vocab
        self.data = {}
        for cl in range(clocks + self.lookahead + 1):
            for w in range(self.W):
                cen, ctx, neg = wl.sgns_batch(c, w, cl, self.device)
                pres = ctx != wl.MISSING
                keys = torch.cat([cen, V + ctx[pres], V + neg[pres].reshape(-1)]).to(torch.int32)
                ctx32 = torch.where(pres, ctx, torch.full_like(ctx, 0xFFFFFFFF)).to(torch.int32)
                self.data[(w, cl)] = (cen.to(torch.int32), ctx32.reshape(-1), neg.reshape(-1).to(torch.int32),
                                      keys)
        self.loss = torch.zeros(self.W, dtype=torch.float64, device=self.device)

    def start(self, pm):
        for w in range(self.W):
            for j in range(self.lookahead):
                pm.intent(w, self.data[(w, j)][3], j, j + self.span)

    def step(self, pm, cl, data=None, loss=None):
        c = self.cfg
        data = data or self.data
        for w in range(self.W):
            j = cl + self.lookahead
            pm.intent(w, data[(w, j)][3], j, j + self.span)
            cen, ctx, neg, _ = data[(w, cl)]
            pm.sgns_step(w, cen, ctx, neg, self.n_ctx, c.negatives, c.vocab, c.dim, c.lr,
                         loss_out=(self.loss[w:w + 1] if loss is None else loss))
            pm.advance_clock(w)
        pm.sync()

    def keys_per_step(self):
        return 2 * self.W * self.cfg.batch * self.per

    def step_alg_bytes(self):
        # per centre: its rows read once, one delta row + key written per row
        return self.W * self.cfg.batch * self.per * (2 * self.row + 8)

    def prepare_host(self, clocks):
        self.hdata = {(w, cc): tuple(x.cpu().pin_memory() for x in self.data[(w, cc)]) for cc in clocks
                      for w in range(self.W) if (w, cc) in self.data}
        self.hloss = torch.zeros(1, dtype=torch.float64, pin_memory=True)

    def step_host(self, pm, cl):
        self.step(pm, cl, data=self.hdata, loss=self.hloss)

    def host_bytes_per_step(self):
        c = self.cfg
        return self.W * c.batch * self.per * 4 * 2, self.W * 8


WORKLOADS = {"micro": Micro, "mf": MF, "tiny_mf": TinyMF, "complex": ComplEx, "sgns": SGNS}


# ---------------------------------------------------------------------------
# algorithmic bytes: the minimum each operation must move (keys 4 B, row D*4 B)
# ---------------------------------------------------------------------------
def alg_bytes_per_step(wk, d, steps, relocate=False):
    """d: differences of the library counters over `steps` profiled steps.

    A distinct pushed key costs 4 rows when its target is a replica (value and pending updates, read and
    written) and 2 when it is main.  Always replicating, every key a worker pushes has a replica; with
    relocation the split is not counted, so every target is taken as main (a lower bound)."""
    row = wk.row
    per = {k: v / steps for k, v in d.items()}
    R, U = per["push_rows"], per["push_unique"]
    tgt = 2 * row if relocate else 4 * row
    out = {
        # read keys + scatter rows, and one row read per distinct key (+ its slot)
        "push": R * (4 + row) + U * (4 + tgt),
        # the scatter kernel alone also reads the sorted (key, position) pairs
        "push_kernel": R * (8 + row) + U * (4 + tgt),
        # main += pending (2 rows per key); read pending and clear it (2 rows per replica); val := main
        # (1 row per refreshed replica: all of them unless the refresh is versioned)
        "sync": per["sync_keys"] * 2 * row + per["sync_replicas"] * 2 * row + per["sync_refreshed"] * row,
        # destroy: read pending, read+write main; create: read main, write val and pending
        "advance": (per["created"] + per["destroyed"]) * 3 * row,
    }
    if isinstance(wk, Micro):
        B, W = wk.cfg.batch, wk.W
        out["pull"] = W * B * (4 + row) + U * (4 + row)
        out["pull_kernel"] = out["pull"]
        out["intent"] = W * B * 4 + U * 4
    else:
        out["step"] = wk.step_alg_bytes()
        out["intent"] = R * 4 + U * 4
    return out


COUNTERS = ("push_rows", "push_unique", "sync_keys", "sync_replicas", "sync_refreshed", "created", "destroyed",
            "relocations", "planned_pushes", "plan_misses", "early_advances", "early_undone")


def manager_options(args):
    """The parameter manager's placement, action timing, refresh and push-plan options, as named in
    `config`."""
    return {"placement": "relocate" if args.relocate else "replicate", "action_timing": args.timing,
            "refresh": "versioned" if args.delta_refresh else "full",
            "push_plans": not getattr(args, "no_push_plans", False),
            "early_events": not getattr(args, "no_early_events", False),
            "pull": "bulk copies through shared memory" if getattr(args, "pull_staging", False) else "registers"}


def run_ours(args, ws, rank, local, workload=None):
    from paper_2206_00470_gb300 import adapm
    workload = workload or args.workload
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    wk = WORKLOADS[workload](args, device)
    total_clocks = args.warmup + args.steps
    t0 = time.time()
    wk.prepare(total_clocks + 2 * args.steps + 2)
    init = wk.init_store()
    pm = adapm.ParameterManager(wk.K, wk.D, wk.W, replica_capacity=wk.capacity, init_values=init,
                                relocate=args.relocate, action_timing=args.timing,
                                delta_refresh=args.delta_refresh, push_plans=not args.no_push_plans,
                                pull_staging=getattr(args, "pull_staging", False),
                                early_events=not getattr(args, "no_early_events", False))
    del init
    torch.cuda.synchronize()
    setup_s = time.time() - t0

    # -- device-resident run ---------------------------------------------------
    wk.start(pm)
    for cl in range(args.warmup):
        wk.step(pm, cl)
    pm.wait()
    clocks = ClockSampler(local)
    start_ev, end_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(ws)
    torch.cuda.synchronize()
    l0 = adapm.kernel_launches()
    clocks.start()
    start_ev.record()
    for cl in range(args.warmup, total_clocks):
        wk.step(pm, cl)
    end_ev.record()
    torch.cuda.synchronize()
    launches = adapm.kernel_launches() - l0
    barrier(ws)
    ms = start_ev.elapsed_time(end_ev)
    pm.wait()
    stats = pm.stats()

    # -- per-operation device times (library events), same steps again ---------
    s0 = pm.stats()
    pm.profile_enable(True)
    pm.profile_read()
    for cl in range(total_clocks, total_clocks + args.steps):
        wk.step(pm, cl)
    prof = pm.profile_read()
    pm.profile_enable(False)
    s1 = pm.stats()
    pm.wait()
    clk = clocks.stop()          # sampled over the timed and the profiled pass

    # -- end to end through the C ABI with pinned host buffers -------------------
    e2e_ms = None
    if not args.no_e2e:
        base = total_clocks + args.steps
        wk.prepare_host(range(base, base + 1 + args.steps + wk.lookahead + 1))
        wk.step_host(pm, base)
        pm.wait()
        barrier(ws)
        torch.cuda.synchronize()
        t = time.perf_counter()
        for cl in range(base + 1, base + 1 + args.steps):
            wk.step_host(pm, cl)
        pm.wait()
        e2e_ms = (time.perf_counter() - t) * 1e3
        barrier(ws)
    pm.close()

    ms_max = max_over_ranks(ms, ws, device)
    keys_total = sum_over_ranks(wk.keys_per_step() * args.steps, ws, device)
    value = keys_total / (ms_max / 1e3)
    samples = sum_over_ranks(wk.samples_per_step * args.steps, ws, device) / (ms_max / 1e3)
    peak, peak_src = load_peaks()

    steps = args.steps
    delta = {k: s1[k] - s0[k] for k in COUNTERS}
    alg = alg_bytes_per_step(wk, delta, steps, args.relocate)
    ops = {}
    for name, (t_ms, calls) in prof.items():
        if calls == 0:
            continue
        d = {"ms_per_step": t_ms / steps, "calls_per_step": calls / steps}
        if name in alg and t_ms > 0:
            gbs = alg[name] / (t_ms / steps / 1e3) / 1e9
            d["alg_bytes_per_step"] = alg[name]
            d["alg_GBps"] = gbs
            d["frac_of_peak"] = gbs / peak
        ops[name] = d

    # dominant kernel: the library kernel (or fused kernel pair) with the largest time
    roofline = None
    cand = [(ops[n]["ms_per_step"], n) for n in ("push_kernel", "pull_kernel", "sync", "step")
            if n in ops and n in alg]
    if cand:
        t_ms, name = max(cand)
        calls = ops[name]["calls_per_step"]
        a = alg[name] / calls
        dur = t_ms / calls / 1e3
        ach = a / dur / 1e9
        traffic = None
        if name == "push_kernel":
            rows = (s1["push_rows"] - s0["push_rows"]) / steps / calls
            traffic = recorded_traffic(workload, rows)
        roofline = {"bound": "hbm", "kernel": name, "achieved": ach, "peak": peak,
                    "peak_source": peak_src, "unit": "GB/s", "frac": ach / peak,
                    "traffic": traffic, "alg_bytes_per_launch": a, "launch_ms": t_ms / calls}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "samples_per_s": samples if wk.samples_per_step else None,
        "config": dict(wk.config(), parallelism=f"replicas{ws}", **manager_options(args),
                       l2="inputs larger than L2 (no flush)"),
        "gpu_launches": int(launches),
        "clocks": clk,
        "roofline": roofline,
        "ops": ops,
        "stats": {k: stats[k] for k in ("live_replicas", "high_water", "capacity")},
        # replica management per step (profiled pass): what relocation saves against always replicating
        "replica_events_per_step": {k: delta[k] / steps for k in ("created", "destroyed", "sync_replicas",
                                                                   "sync_refreshed", "sync_keys", "relocations")},
        "push_plans_per_step": {k: delta[k] / steps for k in ("planned_pushes", "plan_misses")},
        "early_events_per_step": {k: delta[k] / steps for k in ("early_advances", "early_undone")},
        "setup_s": setup_s,
    }
    if e2e_ms is not None:
        e2e_max = max_over_ranks(e2e_ms, ws, device)
        h2d, d2h = wk.host_bytes_per_step()
        line["e2e"] = {"value": keys_total / (e2e_max / 1e3), "unit": UNIT,
                       "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}
    return line


# ---------------------------------------------------------------------------
# CPU oracle (reported baseline / reference arm)
# ---------------------------------------------------------------------------
def oracle_sample(workload, budget_s, args):
    """Time the CPU oracle on a bounded sample of the workload; returns (keys/s, samples/s, desc)."""
    from oracle import ParameterManagerOracle, steps as osteps
    from oracle import driver as odriver
    import dataclasses
    if workload == "micro":
        base = wl.MICRO
        cfg = dataclasses.replace(base, batch=1 << 13,
                                  zipf_s=args.zipf if args.zipf is not None else base.zipf_s,
                                  span=args.span or base.span)
        nclk = 24
        kmap = {}
        for cl in range(nclk + cfg.lookahead + 1):
            for w in range(cfg.workers):
                kmap[(w, cl)] = wl.micro_keys(cfg, w, cl, "cpu").numpy()
        touched = np.unique(np.concatenate(list(kmap.values())))
        rel = {k: np.searchsorted(touched, v) for k, v in kmap.items()}
        init = hashgen.init_rows_np(touched, cfg.value_len, cfg.value_len, cfg.seed, cfg.init_std)
        pm = ParameterManagerOracle(touched.size, cfg.value_len, cfg.workers, init, relocation=args.relocate,
                                    action_timing=args.timing, delta_refresh=args.delta_refresh)
        g = np.random.default_rng(0)
        deltas = (g.standard_normal((cfg.batch, cfg.value_len)) * cfg.delta_std).astype(np.float32)

        def work(w, cl):
            k = rel[(w, cl)]
            pm.pull(w, k)
            pm.push(w, k, deltas)

        keys_of = lambda w, cl: rel[(w, cl)]  # noqa: E731
        odriver.start(pm, cfg.workers, cfg.lookahead, cfg.span, keys_of)
        t = time.perf_counter()
        done = 0
        while done < nclk and time.perf_counter() - t < budget_s:
            odriver.clock(pm, cfg.workers, cfg.lookahead, cfg.span, done, keys_of, work)
            done += 1
        el = time.perf_counter() - t
        keys = done * cfg.workers * cfg.batch * 2
        desc = (f"{done} clocks of {cfg.workers} workers x {cfg.batch} Zipf({cfg.zipf_s}) keys of the "
                f"100M-key x 64 workload (store restricted to the {touched.size} touched keys)")
        return keys / el, None, desc
    if workload == "mf":
        cfg = dataclasses.replace(wl.MF, batch=2048)
        nclk = 24
        data = {}
        for cl in range(nclk + cfg.lookahead + 1):
            for w in range(cfg.workers):
                r, co, v = wl.mf_batch(cfg, w, cl, "cpu")
                data[(w, cl)] = (r.numpy(), co.numpy(), v.numpy())
        touched = np.unique(np.concatenate([np.concatenate([a, b]) for a, b, _ in data.values()]))
        rel = {k: (np.searchsorted(touched, a), np.searchsorted(touched, b), v)
               for k, (a, b, v) in data.items()}
        init = hashgen.init_rows_np(touched, cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
        pm = ParameterManagerOracle(touched.size, cfg.value_len, cfg.workers, init, relocation=args.relocate,
                                    action_timing=args.timing, delta_refresh=args.delta_refresh)

        def work(w, cl):
            a, b, v = rel[(w, cl)]
            return osteps.mf_step(pm, w, a, b, v, cfg.rank, cfg.lr, cfg.adagrad, cfg.eps)

        keys_of = lambda w, cl: np.concatenate(rel[(w, cl)][:2])  # noqa: E731
        odriver.start(pm, cfg.workers, cfg.lookahead, cfg.span, keys_of)
        t = time.perf_counter()
        done = 0
        while done < nclk and time.perf_counter() - t < budget_s:
            odriver.clock(pm, cfg.workers, cfg.lookahead, cfg.span, done, keys_of, work)
            done += 1
        el = time.perf_counter() - t
        cells = done * cfg.workers * cfg.batch
        desc = (f"{done} clocks of {cfg.workers} workers x {cfg.batch} cells of the 10M x 1M rank-100 "
                f"AdaGrad workload (store restricted to the {touched.size} touched keys)")
        return 4 * cells / el, cells / el, desc
    if workload == "tiny_mf":
        cfg = wl.TINY_MF
        data = wl.tiny_mf_dataset(cfg)
        nclk = wl.tiny_mf_clocks(cfg, data[3])
        init = hashgen.init_rows_np(np.arange(cfg.num_keys), cfg.value_len, cfg.rank, cfg.seed, cfg.init_std)
        pm = ParameterManagerOracle(cfg.num_keys, cfg.value_len, cfg.workers, init, relocation=args.relocate,
                                    action_timing=args.timing, delta_refresh=args.delta_refresh)
        bt = {(w, c): [x.numpy() for x in wl.tiny_mf_batch(cfg, data, w, c)]
              for w in range(cfg.workers) for c in range(nclk + cfg.lookahead + 1)}

        def work(w, cl):
            a, b, v = bt[(w, cl)]
            return osteps.mf_step(pm, w, a, b, v, cfg.rank, cfg.lr, cfg.adagrad)

        keys_of = lambda w, cl: np.concatenate(bt[(w, cl)][:2])  # noqa: E731
        odriver.start(pm, cfg.workers, cfg.lookahead, cfg.span, keys_of)
        t = time.perf_counter()
        done = 0
        while done < nclk and time.perf_counter() - t < budget_s:
            odriver.clock(pm, cfg.workers, cfg.lookahead, cfg.span, done, keys_of, work)
            done += 1
        el = time.perf_counter() - t
        cells = sum(bt[(w, c)][0].size for w in range(cfg.workers) for c in range(done))
        return 4 * cells / el, cells / el, f"{done} clocks of the tiny MF workload (all {cfg.workers} workers)"
    if workload in ("complex", "sgns"):
        base = wl.COMPLEX if workload == "complex" else wl.SGNS
        cfg = dataclasses.replace(base, batch=32 if workload == "complex" else 16)
        nclk = 12
        batches = {}
        for cl in range(nclk + cfg.lookahead + 1):
            for w in range(cfg.workers):
                if workload == "complex":
                    batches[(w, cl)] = [x.numpy() for x in wl.complex_batch(cfg, w, cl)]
                else:
                    batches[(w, cl)] = [x.numpy() for x in wl.sgns_batch(cfg, w, cl)]

        def keys_full(b):
            if workload == "complex":
                return np.concatenate([b[0], b[1], b[2], b[3].reshape(-1)])
            pres = b[1] != wl.MISSING
            return np.concatenate([b[0], cfg.vocab + b[1][pres], cfg.vocab + b[2][pres].reshape(-1)])

        touched = np.unique(np.concatenate([keys_full(b) for b in batches.values()]))
        theta = cfg.theta_dim if workload == "complex" else cfg.dim
        init = hashgen.init_rows_np(touched, cfg.value_len, theta, cfg.seed, cfg.init_std)
        pm = ParameterManagerOracle(touched.size, cfg.value_len, cfg.workers, init, relocation=args.relocate,
                                    action_timing=args.timing, delta_refresh=args.delta_refresh)
        rel = lambda x: np.searchsorted(touched, x)  # noqa: E731

        if workload == "complex":
            def work(w, cl):
                h, r, t_, n = batches[(w, cl)]
                return osteps.complex_step(pm, w, rel(h), rel(r), rel(t_), rel(n), theta, cfg.lr, cfg.eps)
            per = 3 + cfg.negatives
        else:
            # the store is relabelled: a token's output row is found through its relabelled key
            class Relabelled:
                def __init__(self, inner):
                    self.inner = inner

                def pull(self, w, keys):
                    return self.inner.pull(w, rel(np.asarray(keys)))

                def push(self, w, keys, d):
                    return self.inner.push(w, rel(np.asarray(keys)), d)

            rpm = Relabelled(pm)

            def work(w, cl):
                cen, ctx, neg = batches[(w, cl)]
                return osteps.sgns_step(rpm, w, cen, ctx, neg, cfg.vocab, cfg.lr)
            per = 1 + 2 * cfg.window * (1 + cfg.negatives)

        keys_of = lambda w, cl: rel(keys_full(batches[(w, cl)]))  # noqa: E731
        odriver.start(pm, cfg.workers, cfg.lookahead, cfg.span, keys_of)
        t = time.perf_counter()
        done = 0
        while done < nclk and time.perf_counter() - t < budget_s:
            odriver.clock(pm, cfg.workers, cfg.lookahead, cfg.span, done, keys_of, work)
            done += 1
        el = time.perf_counter() - t
        samples = done * cfg.workers * cfg.batch
        desc = (f"{done} clocks of {cfg.workers} workers x {cfg.batch} samples of the {base.name} workload "
                f"(store restricted to the {touched.size} touched keys)")
        return 2 * samples * per / el, samples / el, desc
    raise ValueError(workload)


def host_cpu():
    """The host CPU the oracle ran on: machine, model (from /proc/cpuinfo when it names one) and core count."""
    import platform
    model = None
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                key = ln.split(":")[0].strip().lower()
                if key in ("model name", "cpu model", "hardware") and ":" in ln:
                    model = ln.split(":", 1)[1].strip()
                    break
                if key == "cpu part" and model is None:
                    model = "CPU part " + ln.split(":", 1)[1].strip()
    except OSError:
        pass
    return {"machine": platform.machine(), "model": model, "nproc": os.cpu_count()}


def cpu_baseline(args):
    threads = torch.get_num_threads()
    torch.set_num_threads(1)              # the oracle's batch generators run on the host too
    try:
        v, s, desc = oracle_sample(args.workload, args.cpu_budget, args)
    finally:
        torch.set_num_threads(threads)
    return {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": desc,
            "samples_per_s": s, "host_threads_available": os.cpu_count(),
            "threads": {"torch": 1, **{k: os.environ.get(k) for k in ORACLE_THREAD_VARS}},
            "host": host_cpu()}


def run_reference(args, ws, rank):
    if rank != 0:
        return None
    base = cpu_baseline(args)
    line = {
        "impl": "reference", "metric": METRIC, "value": base["value"], "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": dict(WORKLOADS[args.workload](args, None).config(), parallelism="replicas1",
                       **manager_options(args), l2="inputs larger than L2 (no flush)"),
        "reference_kind": "CPU oracle (plain Python/numpy, 1 core)",
        "cpu_baseline": base,
        "e2e": {"value": base["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    return line


MICRO_KEYS = ("value", "unit", "ms_per_step", "config", "gpu_launches", "clocks", "roofline", "ops", "e2e",
              "stats", "replica_events_per_step", "push_plans_per_step", "early_events_per_step", "setup_s")


def micro_args(args, zipf):
    """The microbenchmark's default shape (B = 2^20 keys per worker and clock, span 1, 100M keys) at
    Zipf exponent `zipf`, with the run's steps, warm-up and manager options."""
    a = argparse.Namespace(**vars(args))
    a.workload, a.batch, a.zipf, a.span, a.keys = "micro", None, zipf, None, None
    return a


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="mf", choices=sorted(WORKLOADS))
    ap.add_argument("--batch", type=int, default=None)
    ap.add_argument("--zipf", type=float, default=None)
    ap.add_argument("--span", type=int, default=None)
    ap.add_argument("--keys", type=int, default=None, help="micro: key-space size (default 1e8)")
    ap.add_argument("--mf-rows", type=int, default=None, help="mf: rows (default 10M)")
    ap.add_argument("--mf-cols", type=int, default=None, help="mf: columns (default 1M)")
    ap.add_argument("--micro-zipf", type=lambda x: [float(v) for v in x.split(",") if v], default=[1.1],
                    help="with the MF workload, also run the 100M-key microbenchmark at these Zipf exponents "
                         "(comma-separated; the first is reported as 'micro', the rest as 'micro_sweep'; "
                         "empty string: none)")
    ap.add_argument("--cpu-budget", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--relocate", action="store_true",
                    help="relocate a key to its only worker with active intent instead of always replicating")
    ap.add_argument("--delta-refresh", action="store_true",
                    help="versioned refresh: sync leaves a sole holder's value when nobody else wrote the key")
    ap.add_argument("--pull-staging", action="store_true",
                    help="pull rows through shared memory with bulk copies instead of through registers")
    ap.add_argument("--no-push-plans", action="store_true",
                    help="sort every push itself instead of using the sort made for its intent")
    ap.add_argument("--no-early-events", action="store_true",
                    help="compute each advance's refcount events in the advance instead of beside the pull/push")
    ap.add_argument("--timing", default="start", choices=["start", "adaptive", "signal"],
                    help="act on an intent at its start clock, by Algorithm 1 at each sync, or when signalled")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    ws, rank, local = dist_env()
    if args.impl == "reference":
        if ws > 1:
            init_dist(ws, "gloo")
        line = run_reference(args, ws, rank)
        if line is not None:
            print(json.dumps(line), flush=True)
        return
    init_dist(ws, "nccl")
    # the oracle baseline runs on the host before any CUDA work (rank 0, N=1 only)
    base = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        base = cpu_baseline(args)
    line = run_ours(args, ws, rank, local)
    if args.workload == "mf" and args.micro_zipf:
        # the parameter-access microbenchmark (100M keys x 64 floats, 2^20 Zipf keys per worker and
        # clock, span 1) in the same run: pull, push and sync against the HBM roofline
        sweep = []
        for z in args.micro_zipf:
            torch.cuda.empty_cache()          # the library allocates with cudaMalloc, not torch's cache
            rec = run_ours(micro_args(args, z), ws, rank, local, "micro")
            sweep.append({k: rec[k] for k in MICRO_KEYS if k in rec})
        line["micro"] = sweep[0]
        if len(sweep) > 1:
            line["micro_sweep"] = sweep[1:]
    if rank == 0:
        line["cpu_baseline"] = base
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
