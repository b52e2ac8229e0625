"""The five synthetic workloads and their per-(worker, clock) batches.

Every batch is a pure function of (seed, worker, clock) and the backend, so a
test can regenerate any clock's batch without replaying earlier ones.  Shapes
and distributions follow the paper's workloads (App. C task details) scaled
to one GPU:

  tiny_mf  1,000 x 500 matrix, rank 16, 20,000 uniform cells, W=4, batch 256
  mf       10M x 1M matrix, rank 100 (+ AdaGrad), cells with Zipf(1.1) rows
           and columns, W=8, batch 65,536
  complex  ComplEx, 5M entities + 800 relations, 2x128 (+ AdaGrad), Zipf(1.0)
           entities, Zipf(1.2) relations, 100 uniform negative tails,
           W=8, batch 4,096 triples
  sgns     skip-gram, vocabulary 700K, dim 300, Zipf(1.0) token stream,
           window 5, 25 negatives from unigram^0.75, W=8, batch 8,192 centres
  micro    100M keys x 64 floats, batches of 2^14..2^20 Zipf keys, W=8

Key layout (one key space per store): MF rows [0, R), columns [R, R+C);
ComplEx entities [0, E), relations [E, E+800); SGNS input vectors [0, V),
output vectors [V, 2V); micro [0, 1e8).

Planted MF factors come from the counter hash (hashgen), so the value of a
cell is reproducible for any subset of cells on any backend.  Uniform draws
(Zipf ranks, noise, negatives) use a torch.Generator seeded per
(seed, worker, clock, stream); CPU and CUDA generators give different
streams, so parity tests generate on the CPU and copy to the GPU.
"""
import dataclasses
import math

import torch

from . import hashgen
from .zipf import ranks_to_keys, zipf_ranks

MISSING = -1   # context slot without a token (SGNS near a shard edge)


def _mix(*parts):
    v = 0x2545F491
    for p in parts:
        v = (v * 0x9E3779B1 + (int(p) & 0xFFFFFFFFFFFF) + 0x7F4A7C15) % (1 << 61)
        v ^= v >> 29
    return v % (1 << 62)


def batch_generator(seed, worker, clock, stream, device="cpu"):
    g = torch.Generator(device=device)
    g.manual_seed(_mix(seed, worker, clock, stream))
    return g


# ---------------------------------------------------------------------------
# configurations
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class MFConfig:
    name: str
    rows: int
    cols: int
    rank: int
    adagrad: bool
    workers: int
    batch: int
    lookahead: int
    span: int
    lr: float
    init_std: float
    noise_std: float
    zipf_s: float            # 0 = uniform rows/cols
    total_cells: int
    epochs: int = 1
    eps: float = 1e-8
    seed: int = 0

    @property
    def num_keys(self):
        return self.rows + self.cols

    @property
    def value_len(self):
        return 2 * self.rank if self.adagrad else self.rank

    @property
    def planted_std(self):
        # each planted product u*.w* then has unit variance
        return self.rank ** -0.25


@dataclasses.dataclass
class ComplExConfig:
    name: str
    entities: int
    relations: int
    half_dim: int            # complex dimension: theta row = [re(half) | im(half)]
    workers: int
    batch: int
    negatives: int
    lookahead: int
    span: int
    lr: float
    init_std: float
    zipf_entities: float
    zipf_relations: float
    total_triples: int
    eps: float = 1e-8
    seed: int = 0

    @property
    def num_keys(self):
        return self.entities + self.relations

    @property
    def theta_dim(self):
        return 2 * self.half_dim

    @property
    def value_len(self):
        return 2 * self.theta_dim    # theta + AdaGrad accumulator


@dataclasses.dataclass
class SGNSConfig:
    name: str
    vocab: int
    dim: int
    workers: int
    batch: int               # centre tokens per worker per clock
    window: int
    negatives: int
    lookahead: int
    span: int
    lr: float
    init_std: float
    zipf_s: float
    neg_power: float
    total_tokens: int
    seed: int = 0

    @property
    def num_keys(self):
        return 2 * self.vocab

    @property
    def value_len(self):
        return self.dim

    @property
    def shard_len(self):
        return self.total_tokens // self.workers


@dataclasses.dataclass
class MicroConfig:
    name: str
    num_keys: int
    value_len: int
    workers: int
    batch: int
    zipf_s: float
    span: int
    delta_std: float
    init_std: float
    lookahead: int = 1
    seed: int = 0


TINY_MF = MFConfig(name="tiny_mf", rows=1000, cols=500, rank=16, adagrad=False, workers=4,
                   batch=256, lookahead=2, span=1, lr=0.05, init_std=0.1, noise_std=0.01,
                   zipf_s=0.0, total_cells=20000, epochs=5)
MF = MFConfig(name="mf_10Mx1M_r100", rows=10_000_000, cols=1_000_000, rank=100, adagrad=True,
              workers=8, batch=65536, lookahead=4, span=1, lr=0.05, init_std=0.1, noise_std=0.1,
              zipf_s=1.1, total_cells=500_000_000)
COMPLEX = ComplExConfig(name="complex_5M", entities=5_000_000, relations=800, half_dim=128,
                        workers=8, batch=4096, negatives=100, lookahead=2, span=1, lr=0.1,
                        init_std=0.1, zipf_entities=1.0, zipf_relations=1.2,
                        total_triples=20_000_000)
SGNS = SGNSConfig(name="sgns_700K", vocab=700_000, dim=300, workers=8, batch=8192, window=5,
                  negatives=25, lookahead=3, span=1, lr=0.05, init_std=0.1, zipf_s=1.0,
                  neg_power=0.75, total_tokens=100_000_000)
MICRO = MicroConfig(name="micro_100Mx64", num_keys=100_000_000, value_len=64, workers=8,
                    batch=1 << 20, zipf_s=1.1, span=1, delta_std=1e-3, init_std=0.1)


# ---------------------------------------------------------------------------
# microbenchmark
# ---------------------------------------------------------------------------

def micro_keys(cfg, worker, clock, device="cpu", batch=None):
    """Keys P_c of worker `worker` at clock `clock` (int64, may repeat)."""
    b = cfg.batch if batch is None else batch
    g = batch_generator(cfg.seed, worker, clock, 1, device)
    r = zipf_ranks(b, cfg.num_keys, cfg.zipf_s, g, device)
    return ranks_to_keys(r, cfg.num_keys, cfg.seed)


def micro_deltas(cfg, worker, clock, n, device="cpu", dyadic=False):
    """Push delta rows for a batch of n keys: N(0, delta_std), or dyadic."""
    if dyadic:
        # multiples of 2^-10 in [-1/16, 1/16]: sums of up to 2^17 stay exact in fp32
        rows = torch.arange(n, dtype=torch.int64, device=device).view(-1, 1)
        cols = torch.arange(cfg.value_len, dtype=torch.int64, device=device).view(1, -1)
        return hashgen.dyadic_torch(rows + (clock * 64 + worker) * (1 << 22), cols,
                                    cfg.seed + 1, half_range=64)
    g = batch_generator(cfg.seed, worker, clock, 2, device)
    return torch.randn((n, cfg.value_len), generator=g, device=device) * cfg.delta_std


# ---------------------------------------------------------------------------
# matrix factorisation
# ---------------------------------------------------------------------------

def mf_planted_rows(cfg, keys, side, device="cpu"):
    """Planted factor rows (float32, rank columns) of MF keys; side 0 rows, 1 cols."""
    keys = keys.to(torch.int64).view(-1, 1)
    cols = torch.arange(cfg.rank, dtype=torch.int64, device=keys.device).view(1, -1)
    return hashgen.normal_ih4_torch(keys, cols, cfg.seed + 1000, cfg.planted_std, salt=7 + side)


def mf_cell_values(cfg, rows, cols, g):
    """value = planted u*_row . w*_col + N(0, noise_std)."""
    u = mf_planted_rows(cfg, rows, 0)
    w = mf_planted_rows(cfg, cols, 1)
    v = (u.double() * w.double()).sum(1)
    noise = torch.randn(rows.shape[0], generator=g, device=rows.device, dtype=torch.float64)
    return (v + cfg.noise_std * noise).to(torch.float32)


def tiny_mf_dataset(cfg):
    """All cells of the tiny MF config and each worker's visiting order.

    Returns (rows, cols, vals, per_worker_streams) where per_worker_streams[w]
    is the int64 tensor of cell indices visited by worker w over all epochs
    (cells partitioned to workers by row, reshuffled every epoch).
    """
    g = torch.Generator().manual_seed(_mix(cfg.seed, 11))
    rows = torch.randint(0, cfg.rows, (cfg.total_cells,), generator=g)
    cols = torch.randint(0, cfg.cols, (cfg.total_cells,), generator=g)
    vals = mf_cell_values(cfg, rows, cols, g)
    owner = rows % cfg.workers
    streams = []
    for w in range(cfg.workers):
        mine = torch.nonzero(owner == w).view(-1)
        parts = []
        for e in range(cfg.epochs):
            gw = torch.Generator().manual_seed(_mix(cfg.seed, 12, w, e))
            parts.append(mine[torch.randperm(mine.numel(), generator=gw)])
        streams.append(torch.cat(parts))
    return rows, cols, vals, streams


def tiny_mf_clocks(cfg, streams):
    return max(math.ceil(s.numel() / cfg.batch) for s in streams)


def tiny_mf_batch(cfg, data, worker, clock):
    """(row_keys, col_keys, vals) of one worker's batch; empty when it ran out."""
    rows, cols, vals, streams = data
    idx = streams[worker][clock * cfg.batch:(clock + 1) * cfg.batch]
    return rows[idx], cols[idx] + cfg.rows, vals[idx]


def mf_batch(cfg, worker, clock, device="cpu", batch=None):
    """One batch of the large MF config: cells whose row r satisfies r % W == worker.

    Rows and columns are Zipf(s) ranks mapped through seeded bijections;
    drawing rows until `batch` of them belong to the worker is the same as
    partitioning a global Zipf stream of cells by row.
    Returns (row_keys, col_keys, vals) with col keys offset by cfg.rows.
    """
    b = cfg.batch if batch is None else batch
    g = batch_generator(cfg.seed, worker, clock, 3, device)
    got = []
    have = 0
    while have < b:
        r = ranks_to_keys(zipf_ranks(2 * cfg.workers * (b - have) + 64, cfg.rows, cfg.zipf_s, g,
                                     device), cfg.rows, cfg.seed + 1)
        r = r[r % cfg.workers == worker]
        got.append(r)
        have += r.numel()
    rows = torch.cat(got)[:b]
    cols = ranks_to_keys(zipf_ranks(b, cfg.cols, cfg.zipf_s, g, device), cfg.cols, cfg.seed + 2)
    vals = mf_cell_values(cfg, rows, cols, g)
    return rows, cols + cfg.rows, vals


# ---------------------------------------------------------------------------
# ComplEx knowledge-graph embeddings
# ---------------------------------------------------------------------------

def complex_batch(cfg, worker, clock, device="cpu", batch=None):
    """(heads, rels, tails, neg_tails[b, negatives]) as keys (relations offset by E)."""
    b = cfg.batch if batch is None else batch
    g = batch_generator(cfg.seed, worker, clock, 4, device)
    heads = ranks_to_keys(zipf_ranks(b, cfg.entities, cfg.zipf_entities, g, device),
                          cfg.entities, cfg.seed + 1)
    tails = ranks_to_keys(zipf_ranks(b, cfg.entities, cfg.zipf_entities, g, device),
                          cfg.entities, cfg.seed + 1)
    rels = ranks_to_keys(zipf_ranks(b, cfg.relations, cfg.zipf_relations, g, device),
                         cfg.relations, cfg.seed + 2) + cfg.entities
    negs = torch.randint(0, cfg.entities, (b, cfg.negatives), generator=g, device=device)
    return heads, rels, tails, negs


# ---------------------------------------------------------------------------
# skip-gram with negative sampling
# ---------------------------------------------------------------------------

def _sgns_tokens(cfg, worker, chunk, device):
    """Tokens of one 'batch'-long chunk of worker `worker`'s contiguous shard."""
    g = batch_generator(cfg.seed, worker, chunk, 5, device)
    r = zipf_ranks(cfg.batch, cfg.vocab, cfg.zipf_s, g, device)
    return ranks_to_keys(r, cfg.vocab, cfg.seed + 1)


def sgns_batch(cfg, worker, clock, device="cpu"):
    """(centres[b], contexts[b, 2*window], negatives[b, 2*window, n_neg]).

    Centres are the shard positions [clock*b, (clock+1)*b); context slot j
    holds the token at offset (-window..-1, 1..window)[j], or MISSING outside
    the shard.  Negatives are unigram^neg_power draws (the analytic Zipf
    frequency of each rank raised to neg_power, i.e. Zipf(s*neg_power)).
    Token keys are input vectors; callers add cfg.vocab for output vectors.
    """
    b = cfg.batch
    n_chunks = cfg.shard_len // b
    if clock >= n_chunks:                       # this worker's shard is used up: idle
        e = torch.empty(0, dtype=torch.int64, device=device)
        return e, e.view(0, 2 * cfg.window), e.view(0, 2 * cfg.window, cfg.negatives)
    parts = []
    for ch in (clock - 1, clock, clock + 1):
        if 0 <= ch < n_chunks:
            parts.append(_sgns_tokens(cfg, worker, ch, device))
        else:
            parts.append(torch.full((b,), MISSING, dtype=torch.int64, device=device))
    toks = torch.cat(parts)                      # positions (clock-1)*b .. (clock+2)*b
    centres = toks[b:2 * b]
    offs = [o for o in range(-cfg.window, cfg.window + 1) if o != 0]
    pos = torch.arange(b, 2 * b, device=device).view(-1, 1) + torch.tensor(offs, device=device).view(1, -1)
    contexts = toks[pos]
    g = batch_generator(cfg.seed, worker, clock, 6, device)
    nr = zipf_ranks(b * len(offs) * cfg.negatives, cfg.vocab, cfg.zipf_s * cfg.neg_power, g, device)
    negs = ranks_to_keys(nr, cfg.vocab, cfg.seed + 1).view(b, len(offs), cfg.negatives)
    return centres, contexts, negs
