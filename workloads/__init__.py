"""Seeded synthetic input generators shared by the tests and the benchmark.

They hold none of the store's arithmetic: keys, key sets and gradients only.
"""
from .configs import (ALL, BASE_SEED, RELATION_BASE, StoreConfig, YcsbConfig, dlrm, gnn, kg, scaled, tiered,
                      tiny, ycsb, ycsb_uniform)
from .zipf import ZipfSampler, scatter_bijection

__all__ = ["ALL", "BASE_SEED", "RELATION_BASE", "StoreConfig", "YcsbConfig", "ZipfSampler", "dlrm", "gnn", "kg",
           "scaled", "scatter_bijection", "tiered", "tiny", "ycsb", "ycsb_uniform"]
