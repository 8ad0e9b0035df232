"""Device-resident synthetic decoders and their layer tables.

Shapes follow the 1-8B 4-bit models the paper decodes (Section 3, Table 1:
Llama-3.1-8B and Phi-3.5-mini; Section 1: a 4-bit 3B model).  Weights are drawn on the device
by the seeded generator (wq4_synth_*), one stream per (layer, projection,
codes|scales), so any row block can be regenerated on the host with
``synth.matrix`` for checking.  torch provides the device memory; every
computation goes through the C ABI.
"""
from __future__ import annotations

import weakref
from dataclasses import dataclass

import numpy as np

from . import synth
from . import wq4 as _w


@dataclass(frozen=True)
class ModelShape:
    name: str
    num_layers: int
    hidden: int
    ffn: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    vocab: int

    @property
    def n_qkv(self) -> int:
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim

    def mats(self, layer: int):
        """(name, N, K, projection index) of one layer's projections."""
        H, F = self.hidden, self.ffn
        return [("qkv", self.n_qkv, H, synth.MAT_QKV), ("o", H, H, synth.MAT_O),
                ("gate_up", 2 * F, H, synth.MAT_GATE_UP), ("down", H, F, synth.MAT_DOWN)]

    def weight_count(self) -> int:
        per_layer = sum(N * K for _, N, K, _ in self.mats(0))
        return self.num_layers * per_layer + self.vocab * self.hidden

    def weight_bytes(self) -> int:
        """Packed codes (0.5 B) + fp16 scales (1/16 B) per weight."""
        return self.weight_count() * 9 // 16


# 3B-shaped: hidden 3072, 24 q + 8 kv heads of 128, FFN 8192, 28 layers.
SHAPE_3B = ModelShape("3b", 28, 3072, 8192, 24, 8, 128, 128256)
# 8B-shaped (Llama-3.1-8B): hidden 4096, 32 q + 8 kv heads, FFN 14336, 32 layers.
SHAPE_8B = ModelShape("8b", 32, 4096, 14336, 32, 8, 128, 128256)
# Phi-3.5-mini-shaped (the paper's other Table 1 model, 3.8B; dimensions of its
# public model configuration): hidden 3072, 32 q + 32 kv heads of 96 (full
# multi-head attention), FFN 8192, 32 layers, vocabulary 32064.
SHAPE_PHI = ModelShape("phi3.5", 32, 3072, 8192, 32, 32, 96, 32064)
SHAPES = {"3b": SHAPE_3B, "8b": SHAPE_8B, "phi3.5": SHAPE_PHI}


def fill_matrix(W, s, N: int, K: int, seed: int, layer: int, mat: int, symmetric: bool = False,
                stream=None) -> None:
    _w.wq4_synth_codes(W, 0, N * K // 8, seed, synth.stream_id(synth.KIND_CODES, layer, mat), symmetric, stream)
    _w.wq4_synth_scales(s, 0, N * K // 32, seed, synth.stream_id(synth.KIND_SCALES, layer, mat),
                        synth.SCALE_LO, synth.SCALE_HI, stream)


def _release_plan(table) -> None:
    import torch
    torch.cuda.synchronize()          # a batched plan's graph may still run
    _w.wq4_chain_plan_destroy(table)


class DecodeModel:
    """A synthetic decoder resident in device memory plus its wq4 layer table.

    symmetric: codes drawn on 0..14 (the default, zero-mean q - 7, so that deep
    chains stay within fp16) or, with False, uniform on 0..15 (every code value,
    including 15, reaches every kernel; fine for a few layers)."""

    def __init__(self, shape: ModelShape, batch: int = 1, seed: int = 0, eps: float = 1e-5, device=None,
                 symmetric: bool = True, step: bool = False):
        import torch
        self.shape, self.batch, self.seed, self.eps = shape, batch, seed, eps
        self.symmetric = symmetric
        self.step = step           # workspace sized for wq4_decode_step as well
        dev = torch.device("cuda") if device is None else torch.device(device)
        self.weights = []          # per layer: dict name -> (W tensor, s tensor)
        self._keep = []
        layers = (_w.wq4_layer * shape.num_layers)()
        for l in range(shape.num_layers):
            d = {}
            for name, N, K, mat in shape.mats(l):
                W = torch.empty((N, K // 8), dtype=torch.int32, device=dev)
                s = torch.empty((N, K // 32), dtype=torch.int16, device=dev)
                fill_matrix(W, s, N, K, seed, l, mat, symmetric=symmetric)
                d[name] = (W, s)
                setattr(layers[l], name, _w.wq4_mat(W.data_ptr(), s.data_ptr()))
            self.weights.append(d)
        V, H = shape.vocab, shape.hidden
        W = torch.empty((V, H // 8), dtype=torch.int32, device=dev)
        s = torch.empty((V, H // 32), dtype=torch.int16, device=dev)
        fill_matrix(W, s, V, H, seed, shape.num_layers, synth.MAT_LM_HEAD, symmetric=symmetric)
        self.lm_head = (W, s)
        self._layers = layers
        t = _w.wq4_layer_table()
        t.num_layers, t.hidden, t.ffn = shape.num_layers, shape.hidden, shape.ffn
        t.n_q_heads, t.n_kv_heads, t.head_dim = shape.n_q_heads, shape.n_kv_heads, shape.head_dim
        t.vocab, t.batch, t.rms_eps = shape.vocab, batch, eps
        t.layers = layers
        t.lm_head = _w.wq4_mat(W.data_ptr(), s.data_ptr())
        nbytes = _w.wq4_chain_workspace_bytes(t)
        if nbytes == 0:
            raise ValueError(f"invalid chain shape {shape} batch {batch}")
        if step:
            nbytes = _w.wq4_decode_step_workspace_bytes(t)
            if nbytes == 0:
                raise ValueError(f"decode step unsupported for {shape} batch {batch}")
        self.workspace = torch.zeros(nbytes + 256, dtype=torch.uint8, device=dev)
        base = self.workspace.data_ptr()
        aligned = (base + 255) // 256 * 256
        self._ws_offset = aligned - base
        t.workspace = aligned
        t.workspace_bytes = nbytes
        self.table = t
        # the library caches a plan per table: release it with the model, before
        # its buffers can come back at the same addresses under another table
        fin = weakref.finalize(self, _release_plan, t)
        fin.atexit = False

    # --- decoding -------------------------------------------------------
    def decode(self, x, logits, stream=None, check=True) -> int:
        return _w.wq4_decode_chain(self.table, x, logits, stream, check=check)

    def decode_host(self, x_host: np.ndarray, logits_host: np.ndarray, stream=None) -> int:
        return _w.wq4_decode_chain_host(self.table, x_host, logits_host, stream)

    def decode_step(self, caches: "StepCaches", x, logits, stream=None, check=True) -> int:
        """One decode step with attention over `caches` (wq4_decode_step)."""
        return _w.wq4_decode_step(self.table, caches.desc, x, logits, stream, check=check)

    def decode_step_host(self, caches: "StepCaches", x_host: np.ndarray, logits_host: np.ndarray,
                         stream=None) -> int:
        return _w.wq4_decode_step_host(self.table, caches.desc, x_host, logits_host, stream)

    def destroy_plan(self) -> None:
        _w.wq4_chain_plan_destroy(self.table)

    # --- inspection -----------------------------------------------------
    def trace(self, layer: int):
        """fp16 bit arrays (numpy uint16 [batch][len]) of one layer's stages."""
        off = _w.wq4_chain_trace_offsets(self.table, layer)
        sh, B = self.shape, self.batch
        lens = dict(x_in=sh.hidden, qkv=sh.n_qkv, o=sh.hidden, x_mid=sh.hidden,
                    gate_up=2 * sh.ffn, act=sh.ffn, down=sh.hidden, x_out=sh.hidden)
        if self.step:
            lens.update(q_rot=sh.hidden, k_rot=sh.n_kv_heads * sh.head_dim, attn=sh.hidden)
        out = {}
        for name, n in lens.items():
            o = getattr(off, name)
            if layer == sh.num_layers and name != "x_in":
                continue
            o += self._ws_offset
            buf = self.workspace[o:o + 2 * B * n]
            out[name] = buf.cpu().numpy().view(np.uint16).reshape(B, n)
        return out

    def host_rows(self, layer: int, name: str, row_start: int, nrows: int):
        """Rows of one projection regenerated on the host (uint32 W, uint16 s)."""
        sh = self.shape
        if name == "lm_head":
            N, K, mat, lay = sh.vocab, sh.hidden, synth.MAT_LM_HEAD, sh.num_layers
        else:
            (N, K, mat), lay = [(N, K, m) for nm, N, K, m in sh.mats(layer) if nm == name][0], layer
        return synth.matrix(self.seed, N, K, lay, mat, row_start, nrows, symmetric=self.symmetric)


class StepCaches:
    """The paged key/value caches of every layer of a decode step, on the
    device: one page table shared by the layers (sequence b holds
    positions[b] + 1 tokens after the step, pages drawn from a seeded
    permutation of the pool), a cache pool per layer filled with the seeded
    sum4 values, and the rows' positions (tokens already cached)."""

    def __init__(self, shape: ModelShape, positions, page_size: int = 16, seed: int = 0, spare_pages: int = 0,
                 rope_theta: float = 500000.0, device=None):
        import math
        import torch
        dev = torch.device("cuda") if device is None else torch.device(device)
        self.shape, self.page_size, self.seed = shape, page_size, seed
        self.positions = np.asarray(positions, np.int32)
        self.batch = len(self.positions)
        Hkv, D, P = shape.n_kv_heads, shape.head_dim, page_size
        lens = self.positions.astype(np.int64) + 1
        need = (lens + P - 1) // P
        self.num_pages = int(need.sum()) + spare_pages
        self.table_host = synth.page_table(seed, lens, P, self.num_pages)
        self.table = torch.from_numpy(self.table_host).to(dev)
        self.pos_dev = torch.from_numpy(self.positions.copy()).to(dev)
        n = self.num_pages * Hkv * P * D
        self.k, self.v = [], []
        descs = (_w.wq4_kv_cache * shape.num_layers)()
        for l in range(shape.num_layers):
            k = torch.empty((self.num_pages, Hkv, P, D), dtype=torch.int16, device=dev)
            v = torch.empty_like(k)
            _w.wq4_synth_sum4(k, 0, n, seed, synth.stream_id(synth.KIND_K, l, 0))
            _w.wq4_synth_sum4(v, 0, n, seed, synth.stream_id(synth.KIND_V, l, 0))
            self.k.append(k)
            self.v.append(v)
            descs[l] = _w.kv_cache_desc(k, v, self.table, P)
        self._descs = descs
        self.rope_theta = rope_theta
        self.scale = 1.0 / math.sqrt(D)
        self.desc = _w.wq4_decode_attn(descs, self.pos_dev.data_ptr(), rope_theta, self.scale)

    def cache_bytes_read(self) -> int:
        """Key and value bytes one step reads from the caches: every cached
        token of every sequence and layer (the new token's row comes from the
        projection)."""
        sh = self.shape
        return int(self.positions.astype(np.int64).sum()) * sh.n_kv_heads * sh.head_dim * 2 * 2 * sh.num_layers

    def host_cache(self, layer: int):
        """(k, v) fp16 bits [num_pages][n_kv_heads][page_size][head_dim] as they are now on the device."""
        return (self.k[layer].cpu().numpy().view(np.uint16), self.v[layer].cpu().numpy().view(np.uint16))
