"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle.

This module holds no arithmetic of the method (no unpacking, no dequantization,
no dot products): it only draws random bits and turns them into the input
arrays, so that the oracle and the CUDA path can be fed identical bytes.

Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014), used counter-style so that any element of
any stream can be produced independently:

    mix64(z)        = the SplitMix64 output function
                      (xor-shift 30, multiply, xor-shift 27, multiply,
                      xor-shift 31, with the published multipliers)
    key(seed, sid)  = mix64(seed * GAMMA + sid * SID_MUL)          (mod 2^64)
    u64(key, i)     = mix64(key + (i + 1) * GAMMA)                 (mod 2^64)

Streams (sid) name one tensor each; see ``stream_id``.

Drawn tensors (the distributions of the 1-8B 4-bit decode workloads):
  * packed codes: uint32 words; word 2m is the low half and word 2m+1 the high
    half of u64(m), so every 4-bit code is uniform on 0..15.  The symmetric
    draw then turns every code 15 into 7: codes 0..14 with mean 7, the range
    of symmetric 4-bit quantisation (|q - 7| <= 7) and zero-mean weights as in
    trained models.  Whole synthetic models use it (with codes uniform on
    0..15, q - 7 has mean 1/2 and the fp16 activations of a deep chain
    overflow); single-matrix tests use the full range;
  * scales: fp16_RNE(lo + (hi - lo) * u), u = (u64(i) >> 11) * 2^-53,
    evaluated in fp64 as one multiply then one add, lo = 0.005, hi = 0.02;
  * activations: fp16_RNE(sqrt(-2 ln u1) * cos(2 pi u2)) (Box-Muller) with
    u1 = ((u64(2i) >> 11) + 1) * 2^-53 and u2 = (u64(2i+1) >> 11) * 2^-53;
  * attention queries, keys and values ("sum4"): the four 16-bit fields of
    u64(i) summed, centred and scaled, fp16_RNE((a + b + c + d - 131070) *
    2^-15): an Irwin-Hall(4) approximation of a normal draw with standard
    deviation 2/sqrt(3) and range [-4, 4].  Integer arithmetic and one
    rounding, so the device generator reproduces it bit for bit;
  * page tables: the pages of a pool in the order of an argsort of u64 draws
    (a random permutation), handed out to the sequences in turn; sequence
    lengths lo + u64(i) mod (hi - lo + 1).

The CUDA library carries a device implementation of the first two draws (for
weight matrices too large to generate on the host in reasonable time); the
tests check it against this module bit for bit.  Activations are always drawn
here and copied.
"""
from __future__ import annotations

import numpy as np

GAMMA = 0x9E3779B97F4A7C15
SID_MUL = 0xD1B54A32D192ED03
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB
MASK64 = (1 << 64) - 1

SCALE_LO = 0.005
SCALE_HI = 0.02

# kinds of stream
KIND_CODES = 0
KIND_SCALES = 1
KIND_X = 2
KIND_Q = 3
KIND_K = 4
KIND_V = 5
KIND_PAGES = 6
KIND_LENS = 7

# projection index within a layer
MAT_QKV, MAT_O, MAT_GATE_UP, MAT_DOWN, MAT_LM_HEAD = 0, 1, 2, 3, 4


def stream_id(kind: int, layer: int = 0, mat: int = 0) -> int:
    """Stream number of one tensor: kind (codes/scales/x), layer, projection."""
    return (kind & 0xFF) | ((mat & 0xFF) << 8) | ((layer & 0xFFFF) << 16)


def _mix64_scalar(z: int) -> int:
    z &= MASK64
    z = ((z ^ (z >> 30)) * _M1) & MASK64
    z = ((z ^ (z >> 27)) * _M2) & MASK64
    return z ^ (z >> 31)


def _mix64(z: np.ndarray) -> np.ndarray:
    z = z.copy()
    z ^= z >> np.uint64(30)
    z *= np.uint64(_M1)
    z ^= z >> np.uint64(27)
    z *= np.uint64(_M2)
    z ^= z >> np.uint64(31)
    return z


def key(seed: int, sid: int) -> int:
    return _mix64_scalar((seed * GAMMA + sid * SID_MUL) & MASK64)


def u64(k: int, start: int, count: int) -> np.ndarray:
    """u64(k, i) for i in [start, start + count)."""
    i = np.arange(start, start + count, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (i + np.uint64(1)) * np.uint64(GAMMA) + np.uint64(k)
    return _mix64(z)


def fold15(words: np.ndarray) -> np.ndarray:
    """Every 4-bit field equal to 15 becomes 7 (bit 3 cleared where all four
    bits are set)."""
    w = words.astype(np.uint32)
    m = w & (w >> np.uint32(1)) & (w >> np.uint32(2)) & (w >> np.uint32(3)) & np.uint32(0x11111111)
    return w ^ (m << np.uint32(3))


def codes_words(seed: int, sid: int, word_start: int, nwords: int, symmetric: bool = False) -> np.ndarray:
    """Packed-code words [word_start, word_start + nwords) of a stream (uint32).

    word_start and nwords must be even (two words per 64-bit draw)."""
    if word_start % 2 or nwords % 2:
        raise ValueError("codes are drawn two words at a time")
    v = u64(key(seed, sid), word_start // 2, nwords // 2)
    w = v.view(np.uint32).copy()  # little endian: low half first
    return fold15(w) if symmetric else w


def scales_fp16(seed: int, sid: int, start: int, count: int,
                lo: float = SCALE_LO, hi: float = SCALE_HI) -> np.ndarray:
    """Scales [start, start + count) of a stream, as fp16 bit patterns (uint16)."""
    v = u64(key(seed, sid), start, count)
    u = (v >> np.uint64(11)).astype(np.float64) * 2.0 ** -53
    s = np.float64(lo) + np.float64(hi - lo) * u
    return s.astype(np.float16).view(np.uint16)


def normal_fp16(seed: int, sid: int, count: int) -> np.ndarray:
    """count N(0,1) draws rounded to fp16, as bit patterns (uint16)."""
    v = u64(key(seed, sid), 0, 2 * count)
    u1 = ((v[0::2] >> np.uint64(11)).astype(np.float64) + 1.0) * 2.0 ** -53
    u2 = (v[1::2] >> np.uint64(11)).astype(np.float64) * 2.0 ** -53
    z = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)
    return z.astype(np.float16).view(np.uint16)


def matrix(seed: int, N: int, K: int, layer: int = 0, mat: int = 0,
           row_start: int = 0, nrows: int | None = None, symmetric: bool = False):
    """Rows [row_start, row_start + nrows) of one N x K packed matrix.

    Returns (W uint32 [nrows][K/8], s uint16 [nrows][K/32]).  Row blocks of
    the same matrix are consistent with the whole, so a sample of rows of a
    large matrix can be regenerated on the host."""
    if nrows is None:
        nrows = N - row_start
    wpr, gpr = K // 8, K // 32
    W = codes_words(seed, stream_id(KIND_CODES, layer, mat), row_start * wpr, nrows * wpr, symmetric)
    s = scales_fp16(seed, stream_id(KIND_SCALES, layer, mat), row_start * gpr, nrows * gpr)
    return W.reshape(nrows, wpr), s.reshape(nrows, gpr)


def activations(seed: int, batch: int, K: int, layer: int = 0) -> np.ndarray:
    """x fp16 bits [batch][K] ~ N(0,1)."""
    return normal_fp16(seed, stream_id(KIND_X, layer, 0), batch * K).reshape(batch, K)


def sum4_fp16(seed: int, sid: int, start: int, count: int) -> np.ndarray:
    """Elements [start, start + count) of a sum4 stream, fp16 bit patterns."""
    v = u64(key(seed, sid), start, count)
    m = np.uint64(0xFFFF)
    c = ((v & m) + ((v >> np.uint64(16)) & m) + ((v >> np.uint64(32)) & m) + (v >> np.uint64(48))).astype(np.int64)
    return ((c - 131070).astype(np.float64) * 2.0 ** -15).astype(np.float16).view(np.uint16)


def seq_lens(seed: int, batch: int, lo: int, hi: int, layer: int = 0) -> np.ndarray:
    """Sequence lengths uniform on [lo, hi] (int32 [batch])."""
    v = u64(key(seed, stream_id(KIND_LENS, layer, 0)), 0, batch)
    return (lo + (v % np.uint64(hi - lo + 1)).astype(np.int64)).astype(np.int32)


def page_table(seed: int, lens, page_size: int, num_pages: int, pt_stride: int | None = None,
               layer: int = 0) -> np.ndarray:
    """Page table int32 [batch][pt_stride]: sequence b gets ceil(len_b / page_size)
    pages, taken in turn from a random permutation of the pool; unused entries
    are -1.  num_pages must cover every sequence's pages."""
    lens = np.asarray(lens, np.int64)
    need = (lens + page_size - 1) // page_size
    if int(need.sum()) > num_pages:
        raise ValueError("page pool too small")
    width = int(need.max()) if pt_stride is None else pt_stride
    order = np.argsort(u64(key(seed, stream_id(KIND_PAGES, layer, 0)), 0, num_pages), kind="stable")
    table = np.full((len(lens), max(width, 1)), -1, np.int32)
    off = 0
    for b, n in enumerate(need):
        table[b, :n] = order[off:off + n]
        off += int(n)
    return table


def kv_cache(seed: int, num_pages: int, n_kv_heads: int, page_size: int, head_dim: int, layer: int = 0):
    """Key and value caches, fp16 bits [num_pages][n_kv_heads][page_size][head_dim] (sum4)."""
    n = num_pages * n_kv_heads * page_size * head_dim
    shape = (num_pages, n_kv_heads, page_size, head_dim)
    k = sum4_fp16(seed, stream_id(KIND_K, layer, 0), 0, n).reshape(shape)
    v = sum4_fp16(seed, stream_id(KIND_V, layer, 0), 0, n).reshape(shape)
    return k, v


def queries(seed: int, batch: int, n_q_heads: int, head_dim: int, layer: int = 0) -> np.ndarray:
    """Queries fp16 bits [batch][n_q_heads * head_dim] (sum4)."""
    return sum4_fp16(seed, stream_id(KIND_Q, layer, 0), 0, batch * n_q_heads * head_dim).reshape(batch, -1)
