"""Device-resident synthetic paged key/value caches for decode attention.

One layer's cache of a batch of sequences in the layout of include/wq4_attn.h
(fp16 [num_pages][n_kv_heads][page_size][head_dim]), with its page table,
lengths, queries and output buffer.  Keys, values and queries are drawn on
the device by the seeded sum4 generator (wq4_synth_sum4), one stream per
tensor, so any page can be regenerated on the host with ``synth.sum4_fp16``
for checking; page tables and lengths come from ``synth``.  torch provides
the device memory; the attention itself runs through the C ABI.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

from . import synth
from . import wq4 as _w
from .model import SHAPES, ModelShape


@dataclass(frozen=True)
class AttnWorkload:
    """Decode attention of one layer: shape, batch, length range, page size."""
    name: str
    shape: ModelShape
    batch: int
    len_lo: int
    len_hi: int
    page_size: int = 16

    def lens(self, seed: int) -> np.ndarray:
        return synth.seq_lens(seed, self.batch, self.len_lo, self.len_hi)


# Llama-3.1-8B-shaped (32 q + 8 kv heads of 128) and 3B-shaped (24 + 8) layers,
# 32 sequences with context lengths uniform on [1, 8192], pages of 16 tokens.
ATTN_WORKLOADS = {
    "attn-8b": AttnWorkload("attn-8b", SHAPES["8b"], 32, 1, 8192),
    "attn-3b": AttnWorkload("attn-3b", SHAPES["3b"], 32, 1, 8192),
    "attn-8b-b1": AttnWorkload("attn-8b-b1", SHAPES["8b"], 1, 4096, 4096),
}


class PagedAttentionLayer:
    """A synthetic paged cache, queries and output of one layer on the device."""

    def __init__(self, shape: ModelShape, lens, page_size: int = 16, seed: int = 0, layer: int = 0,
                 spare_pages: int = 0, device=None):
        import torch
        self.shape, self.page_size, self.seed, self.layer = shape, page_size, seed, layer
        self.lens = np.asarray(lens, np.int32)
        self.batch = len(self.lens)
        dev = torch.device("cuda") if device is None else torch.device(device)
        Hkv, D, P = shape.n_kv_heads, shape.head_dim, page_size
        need = (self.lens.astype(np.int64) + P - 1) // P
        self.num_pages = int(need.sum()) + spare_pages
        n = self.num_pages * Hkv * P * D
        self.k = torch.empty((self.num_pages, Hkv, P, D), dtype=torch.int16, device=dev)
        self.v = torch.empty_like(self.k)
        _w.wq4_synth_sum4(self.k, 0, n, seed, self.sid(synth.KIND_K))
        _w.wq4_synth_sum4(self.v, 0, n, seed, self.sid(synth.KIND_V))
        self.table_host = synth.page_table(seed, self.lens, P, self.num_pages, layer=layer)
        self.table = torch.from_numpy(self.table_host).to(dev)
        self.lens_dev = torch.from_numpy(self.lens.copy()).to(dev)
        Hq = shape.n_q_heads
        self.q = torch.empty((self.batch, Hq * D), dtype=torch.int16, device=dev)
        _w.wq4_synth_sum4(self.q, 0, self.batch * Hq * D, seed, self.sid(synth.KIND_Q))
        self.out = torch.empty((self.batch, Hq * D), dtype=torch.int16, device=dev)
        self.scale = 1.0 / math.sqrt(D)
        nbytes = _w.wq4_paged_attention_workspace_bytes(self.batch, Hq, Hkv, D)
        if nbytes == 0:
            raise ValueError(f"unsupported attention geometry {shape} batch {self.batch}")
        self.workspace = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
        self.cache = _w.kv_cache_desc(self.k, self.v, self.table, P)

    def sid(self, kind: int) -> int:
        return synth.stream_id(kind, self.layer, 0)

    def run(self, stream=None, check: bool = True) -> int:
        Hq, D = self.shape.n_q_heads, self.shape.head_dim
        return _w.wq4_paged_attention(self.cache, self.q, Hq * D, self.lens_dev, self.out, Hq * D, self.batch, Hq,
                                      self.scale, self.workspace, self.workspace.numel(), stream, check=check)

    # --- sizes ------------------------------------------------------------
    def kv_bytes(self) -> int:
        """Key and value bytes the call must read (the cached tokens only)."""
        sh = self.shape
        return int(self.lens.astype(np.int64).sum()) * sh.n_kv_heads * sh.head_dim * 2 * 2

    def algorithmic_bytes(self) -> int:
        """Keys and values, plus the queries read and the outputs written."""
        sh = self.shape
        return self.kv_bytes() + 2 * 2 * self.batch * sh.n_q_heads * sh.head_dim

    # --- host copies for checking ------------------------------------------
    def host_pages(self, pages):
        """(k, v) fp16 bits [len(pages)][n_kv_heads][page_size][head_dim], regenerated on the host."""
        sh = self.shape
        per = sh.n_kv_heads * self.page_size * sh.head_dim
        ks, vs = [], []
        for p in pages:
            ks.append(synth.sum4_fp16(self.seed, self.sid(synth.KIND_K), int(p) * per, per))
            vs.append(synth.sum4_fp16(self.seed, self.sid(synth.KIND_V), int(p) * per, per))
        shp = (len(pages), sh.n_kv_heads, self.page_size, sh.head_dim)
        return np.stack(ks).reshape(shp), np.stack(vs).reshape(shp)

    def host_sequence(self, b: int):
        """Inputs of sequence b alone, on the host: (q row, k, v, page table [1][n], lens [1])
        with the sequence's pages renumbered 0..n-1."""
        sh = self.shape
        T = int(self.lens[b])
        n = (T + self.page_size - 1) // self.page_size
        k, v = self.host_pages(self.table_host[b, :n])
        q = synth.sum4_fp16(self.seed, self.sid(synth.KIND_Q), b * sh.n_q_heads * sh.head_dim,
                            sh.n_q_heads * sh.head_dim)
        return q[None, :], k, v, np.arange(max(n, 1), dtype=np.int32)[None, :], np.array([T], np.int32)
