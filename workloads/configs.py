"""Seeded synthetic workloads shaped like the paper's embedding tables.

Each config builds (a) the preload key list of the table, in preload order, and
(b) for each step the batch of int64 lookup keys (duplicates allowed, in
occurrence order) plus per-lookup fp32 gradients.  Generation is untimed and
holds none of the store's arithmetic; the same arrays feed the CUDA library and
the oracle.

Shapes (MLKV Table 2 lists the paper's datasets; these stand in for them, no
dataset is available):
  tiny   100,000 distinct keys from [0, 2^40), dim 16, 10 steps x 4,096
         Zipf(1.05) lookups, grads N(0, 0.01), Adagrad lr 0.1.
  dlrm   Criteo-shaped: 26 tables x 4,000,000 rows, dim 128, key t*2^32+row,
         65,536 samples x 26 one-hot Zipf(1.2) lookups, grads N(0, 1e-3), lr 0.01.
  kg     Freebase86M-shaped: 80,000,000 entities + 15,000 relations, dim 100,
         50,000 triples (heads, tails Zipf(0.9), relations uniform) plus 1,000
         uniform negatives per 1,000-triple chunk, grads N(0, 1e-3), lr 0.1.
  gnn    Papers100M-shaped: 100,000,000 nodes, dim 64, 8,192 uniform seeds with
         2-hop fanout 10 then 25 over a Chung-Lu power-law graph, grads
         N(0, 1e-3), lr 0.05.
  tiered 400,000,000 rows, dim 128, 1,048,576 Zipf(1.1) lookups, grads N(0, 1e-3).
  ycsb   a YCSB-shaped key-value mix (MLKV Section 4.5: 50% reads, 50% writes,
         uniform or skewed keys): 50,000,000 records of 256 fp32 (1 KiB),
         batches of 1,048,576 operations, each a Get or a Put by a seeded coin,
         keys Zipf(0.99) ("ycsb") or uniform ("ycsb-uniform"), written values
         N(0, 0.01).
The second parameter of N(., .) is the standard deviation.
"""
from dataclasses import dataclass, field

import numpy as np

from .zipf import ZipfSampler, scatter_bijection

BASE_SEED = 20250402
RELATION_BASE = 1 << 62


def _rng(*words) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([BASE_SEED, *[int(w) for w in words]]))


@dataclass
class StoreConfig:
    name: str
    index: int
    dim: int
    n_keys: int          # distinct keys preloaded into the table
    batch: int           # lookups per step
    steps: int
    lr: float
    grad_sigma: float
    eps: float = 1e-8
    state_init: float = 0.0
    init_lo: float = -0.01
    init_hi: float = 0.01
    hbm_cache_rows: int = 0
    _cache: dict = field(default_factory=dict, repr=False)

    @property
    def seed(self) -> int:
        return BASE_SEED * 16 + self.index

    @property
    def capacity(self) -> int:
        return self.n_keys

    # --- preload -----------------------------------------------------------
    def preload_keys(self, start: int = 0, stop: int | None = None) -> np.ndarray:
        stop = self.n_keys if stop is None else min(stop, self.n_keys)
        return self._preload(start, stop)

    def _preload(self, start, stop):
        return np.arange(start, stop, dtype=np.int64)

    # --- per step ----------------------------------------------------------
    def batch_keys(self, step: int) -> np.ndarray:
        raise NotImplementedError

    def grads(self, step: int, n: int | None = None) -> np.ndarray:
        """Per-lookup gradients N(0, sigma) as float32 [batch, dim] (host)."""
        n = self.batch if n is None else n
        g = _rng(self.index, step, 7).standard_normal((n, self.dim), dtype=np.float32)
        g *= np.float32(self.grad_sigma)
        return g


    def grads_device(self, step: int, device, n: int | None = None):
        """Per-lookup gradients N(0, sigma) as a float32 [n, dim] CUDA tensor, from
        torch's device generator seeded by (config, step): for full-size batches,
        whose host generation would take seconds a step.  Tests copy the rows they
        need to the host, so both sides see the same array."""
        import torch

        n = self.batch if n is None else n
        gen = torch.Generator(device=device)
        gen.manual_seed(self.seed * 1000 + 977 + step)
        return torch.randn((n, self.dim), generator=gen, device=device, dtype=torch.float32) * self.grad_sigma


class TinyConfig(StoreConfig):
    def _keyset(self):
        if "keyset" not in self._cache:
            rng = _rng(self.index, 1 << 30)
            keys = np.empty(0, np.int64)
            while len(keys) < self.n_keys:
                draw = rng.integers(0, 1 << 40, size=self.n_keys, dtype=np.int64)
                allk = np.concatenate([keys, draw])
                _, first = np.unique(allk, return_index=True)
                keys = allk[np.sort(first)]
            self._cache["keyset"] = keys[: self.n_keys]
        return self._cache["keyset"]

    def _preload(self, start, stop):
        return self._keyset()[start:stop].copy()

    def batch_keys(self, step: int) -> np.ndarray:
        rng = _rng(self.index, step, 3)
        ranks = ZipfSampler(self.n_keys, 1.05).sample(rng, self.batch)
        return self._keyset()[ranks - 1]


class DlrmConfig(StoreConfig):
    tables: int = 26
    rows_per_table: int = 4_000_000
    alpha: float = 1.2

    def _preload(self, start, stop):
        i = np.arange(start, stop, dtype=np.int64)
        t, r = np.divmod(i, self.rows_per_table)
        return (t << 32) + r

    def _maps(self):
        if "maps" not in self._cache:
            self._cache["maps"] = [scatter_bijection(self.rows_per_table, _rng(self.index, 100 + t))
                                   for t in range(self.tables)]
            self._cache["zipf"] = ZipfSampler(self.rows_per_table, self.alpha)
        return self._cache["maps"], self._cache["zipf"]

    def batch_keys(self, step: int) -> np.ndarray:
        maps, zipf = self._maps()
        samples = self.batch // self.tables
        out = np.empty((samples, self.tables), np.int64)
        for t in range(self.tables):
            ranks = zipf.sample(_rng(self.index, step, 3, t), samples)
            out[:, t] = (np.int64(t) << 32) + maps[t](ranks)
        return out.reshape(-1)  # sample-major: the 26 lookups of a sample are adjacent


class KgConfig(StoreConfig):
    entities: int = 80_000_000
    relations: int = 15_000
    triples: int = 50_000
    chunk: int = 1_000
    neg_per_chunk: int = 1_000
    alpha: float = 0.9

    def _preload(self, start, stop):
        i = np.arange(start, stop, dtype=np.int64)
        return np.where(i < self.entities, i, RELATION_BASE + (i - self.entities))

    def batch_keys(self, step: int) -> np.ndarray:
        if "map" not in self._cache:
            self._cache["map"] = scatter_bijection(self.entities, _rng(self.index, 100))
            self._cache["zipf"] = ZipfSampler(self.entities, self.alpha)
        emap, zipf = self._cache["map"], self._cache["zipf"]
        heads = emap(zipf.sample(_rng(self.index, step, 3, 0), self.triples))
        tails = emap(zipf.sample(_rng(self.index, step, 3, 1), self.triples))
        rels = RELATION_BASE + _rng(self.index, step, 3, 2).integers(0, self.relations, self.triples)
        nneg = (self.triples // self.chunk) * self.neg_per_chunk
        negs = _rng(self.index, step, 3, 3).integers(0, self.entities, nneg)
        return np.concatenate([heads, rels, tails, negs]).astype(np.int64)


class GnnConfig(StoreConfig):
    nodes: int = 100_000_000
    seeds: int = 8_192
    fanouts: tuple = (10, 25)
    degree_exponent: float = 2.1

    def batch_keys(self, step: int) -> np.ndarray:
        # Chung-Lu power-law graph whose degree density falls as k^-2.1, i.e.
        # node weights w with Pareto tail P(W > x) = x^-(2.1 - 1).  In a
        # Chung-Lu graph the neighbours of any node are drawn with probability
        # proportional to w.  With the weights given by their quantiles,
        # w_(r) = (r / N)^(-1/1.1) for the r-th heaviest node, so a draw
        # proportional to w is Zipf(1/1.1) over weight ranks; a fixed bijection
        # places the ranks among node ids.  Sampling is with replacement.
        if "map" not in self._cache:
            self._cache["map"] = scatter_bijection(self.nodes, _rng(self.index, 100))
            self._cache["zipf"] = ZipfSampler(self.nodes, 1.0 / (self.degree_exponent - 1.0))
        nmap, zipf = self._cache["map"], self._cache["zipf"]
        seeds = _rng(self.index, step, 3, 0).integers(0, self.nodes, self.seeds)
        parts = [seeds]
        frontier = self.seeds
        for h, f in enumerate(self.fanouts):
            frontier *= f
            parts.append(nmap(zipf.sample(_rng(self.index, step, 3, 1 + h), frontier)))
        return np.concatenate(parts).astype(np.int64)


class TieredConfig(StoreConfig):
    alpha: float = 1.1

    def batch_keys(self, step: int) -> np.ndarray:
        if "map" not in self._cache:
            self._cache["map"] = scatter_bijection(self.n_keys, _rng(self.index, 100))
            self._cache["zipf"] = ZipfSampler(self.n_keys, self.alpha)
        return self._cache["map"](self._cache["zipf"].sample(_rng(self.index, step, 3), self.batch))


@dataclass
class YcsbConfig(StoreConfig):
    """Batches of Get and Put operations over the preloaded records.  A batch's
    Gets read the records as they were before the batch; its Puts then write
    (the later of two Puts of a key wins)."""
    read_fraction: float = 0.5
    alpha: float = 0.99  # 0: uniform keys

    def _keys(self, step: int) -> np.ndarray:
        rng = _rng(self.index, step, 3)
        if self.alpha == 0.0:
            return rng.integers(0, self.n_keys, self.batch, dtype=np.int64)
        if "map" not in self._cache:
            self._cache["map"] = scatter_bijection(self.n_keys, _rng(self.index, 100))
            self._cache["zipf"] = ZipfSampler(self.n_keys, self.alpha)
        return self._cache["map"](self._cache["zipf"].sample(rng, self.batch))

    def ops(self, step: int):
        """(keys read, keys written, values written [n, dim] float32), in batch order."""
        keys = self._keys(step)
        read = _rng(self.index, step, 9).random(self.batch) < self.read_fraction
        w = keys[~read]
        vals = _rng(self.index, step, 11).standard_normal((len(w), self.dim), dtype=np.float32)
        vals *= np.float32(self.grad_sigma)
        return keys[read], w, vals

    def batch_keys(self, step: int) -> np.ndarray:
        return self._keys(step)


def tiny():
    return TinyConfig("tiny", 0, dim=16, n_keys=100_000, batch=4_096, steps=10, lr=0.1,
                      grad_sigma=0.01)


def dlrm():
    return DlrmConfig("dlrm", 1, dim=128, n_keys=26 * 4_000_000, batch=65_536 * 26, steps=50,
                      lr=0.01, grad_sigma=1e-3)


def kg():
    return KgConfig("kg", 2, dim=100, n_keys=80_000_000 + 15_000, batch=200_000, steps=50,
                    lr=0.1, grad_sigma=1e-3)


def gnn():
    return GnnConfig("gnn", 3, dim=64, n_keys=100_000_000, batch=8_192 * (1 + 10 + 250),
                     steps=30, lr=0.05, grad_sigma=1e-3)


def tiered():
    return TieredConfig("tiered", 4, dim=128, n_keys=400_000_000, batch=1_048_576, steps=20,
                        lr=0.01, grad_sigma=1e-3, hbm_cache_rows=120 * 10**9 // 1024)


def ycsb():
    return YcsbConfig("ycsb", 5, dim=256, n_keys=50_000_000, batch=1_048_576, steps=20, lr=0.0,
                      grad_sigma=0.01, alpha=0.99)


def ycsb_uniform():
    return YcsbConfig("ycsb-uniform", 6, dim=256, n_keys=50_000_000, batch=1_048_576, steps=20, lr=0.0,
                      grad_sigma=0.01, alpha=0.0)


ALL = {"tiny": tiny, "dlrm": dlrm, "kg": kg, "gnn": gnn, "tiered": tiered, "ycsb": ycsb,
       "ycsb-uniform": ycsb_uniform}


def scaled(cfg: StoreConfig, key_scale: int, batch_scale: int) -> StoreConfig:
    """Same distributions on a smaller table and batch (for oracle-sized tests)."""
    import copy
    c = copy.copy(cfg)
    c._cache = {}
    if isinstance(c, DlrmConfig):
        c.rows_per_table = max(1, c.rows_per_table // key_scale)
        c.n_keys = c.tables * c.rows_per_table
        c.batch = max(c.tables, (c.batch // batch_scale) // c.tables * c.tables)
    elif isinstance(c, KgConfig):
        c.entities = max(1, c.entities // key_scale)
        c.triples = max(c.chunk, c.triples // batch_scale // c.chunk * c.chunk)
        c.n_keys = c.entities + c.relations
        c.batch = c.triples * 3 + (c.triples // c.chunk) * c.neg_per_chunk
    elif isinstance(c, GnnConfig):
        c.nodes = max(1, c.nodes // key_scale)
        c.n_keys = c.nodes
        c.seeds = max(1, c.seeds // batch_scale)
        c.batch = c.seeds * (1 + c.fanouts[0] + c.fanouts[0] * c.fanouts[1])
    else:
        c.n_keys = max(1, c.n_keys // key_scale)
        c.batch = max(1, c.batch // batch_scale)
    return c
