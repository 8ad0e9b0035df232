"""Oracle for the 4-bit weight-streaming GEMV and the decode-chain glue.

TEST INFRASTRUCTURE ONLY: only the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import this package.  The product library
(``paper_2412_15803_gb300``) never imports it, and the two share no code.

The arithmetic lives in ``wq4_oracle.c`` (the GEMV and the chain glue) and
``attention_oracle.c`` (decode attention over a paged key/value cache), plain
C, fp64, single-threaded; this module compiles them with gcc and wraps them
with ctypes and numpy.  Every
array is passed as raw bit patterns: fp16 values travel as uint16.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRCS = [os.path.join(_HERE, "wq4_oracle.c"), os.path.join(_HERE, "attention_oracle.c")]
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")

# -ffp-contract=off keeps "acc += w * x" a rounded multiply then a rounded
# add on every host (aarch64 gcc would otherwise fuse it into an fma).
CFLAGS = ["-O2", "-std=c99", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared"]


def build(force: bool = False) -> str:
    """Compile the oracle into oracle/_build/liboracle.so (gcc)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and all(os.path.getmtime(_LIB_PATH) >= os.path.getmtime(f) for f in _SRCS)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", *CFLAGS, *_SRCS, "-o", tmp, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        I = ctypes.c_int
        I64 = ctypes.c_int64
        D = ctypes.c_double
        _lib.wq4o_half_to_double.argtypes = [ctypes.c_uint16]
        _lib.wq4o_half_to_double.restype = D
        _lib.wq4o_double_to_half.argtypes = [D]
        _lib.wq4o_double_to_half.restype = ctypes.c_uint16
        _lib.wq4o_half_to_double_array.argtypes = [P, P, I64]
        _lib.wq4o_double_to_half_array.argtypes = [P, P, I64]
        _lib.wq4o_ulp16.argtypes = [D]
        _lib.wq4o_ulp16.restype = D
        _lib.wq4o_code.argtypes = [P, I, I, I]
        _lib.wq4o_code.restype = I
        _lib.wq4o_pack.argtypes = [P, P, I, I]
        _lib.wq4o_unpack.argtypes = [P, P, I, I, P, P]
        _lib.wq4o_gemv.argtypes = [P, P, P, I, I, I, P, P, P, P]
        _lib.wq4o_rms_factor.argtypes = [P, I, D]
        _lib.wq4o_rms_factor.restype = D
        _lib.wq4o_rms_normalize.argtypes = [P, I, D, P]
        _lib.wq4o_silu_mul.argtypes = [P, P, I, P, P]
        _lib.wq4o_add_fp16.argtypes = [P, P, I, P]
        _lib.wq4o_paged_attention.argtypes = [P, I, P, P, I, I, P, I, P, I, I, I, I, D, P, P, P]
        _lib.wq4o_paged_attention.restype = I
        _lib.wq4o_kv_append.argtypes = [P, P, I, P, P, I, I, P, I, P, I, I, I]
        _lib.wq4o_kv_append.restype = I
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


# ------------------------------------------------------------------- fp16 --

def half_to_double(h) -> np.ndarray:
    h = _c(h, np.uint16)
    out = np.empty(h.shape, np.float64)
    lib().wq4o_half_to_double_array(_p(h), _p(out), h.size)
    return out


def double_to_half(v) -> np.ndarray:
    v = _c(v, np.float64)
    out = np.empty(v.shape, np.uint16)
    lib().wq4o_double_to_half_array(_p(v), _p(out), v.size)
    return out


def ulp16(v: float) -> float:
    return lib().wq4o_ulp16(float(v))


def ulp16_array(v) -> np.ndarray:
    return np.array([ulp16(t) for t in np.ravel(v)]).reshape(np.shape(v))


# ----------------------------------------------------------------- format --

def pack(q) -> np.ndarray:
    """codes uint8 [N][K] -> packed uint32 [N][K/8]."""
    q = _c(q, np.uint8)
    N, K = q.shape
    W = np.empty((N, K // 8), np.uint32)
    lib().wq4o_pack(_p(q), _p(W), N, K)
    return W


def unpack(W, s, K: int):
    """-> (codes uint8 [N][K], w fp64 [N][K] = (q - 7) * s)."""
    W = _c(W, np.uint32)
    s = _c(s, np.uint16)
    N = W.shape[0]
    q = np.empty((N, K), np.uint8)
    w = np.empty((N, K), np.float64)
    lib().wq4o_unpack(_p(W), _p(s), N, K, _p(q), _p(w))
    return q, w


def gemv(W, s, x, r=None):
    """The GEMV definition.  W uint32 [N][K/8], s fp16 bits [N][K/32],
    x fp16 bits [batch][K], r optional fp64 [batch] RMS factors.

    Returns (y fp64 [batch][N], A fp64 [batch][N], y16 fp16 bits [batch][N])."""
    W = _c(W, np.uint32)
    s = _c(s, np.uint16)
    x = _c(x, np.uint16)
    if x.ndim == 1:
        x = x[None, :]
    N = W.shape[0]
    batch, K = x.shape
    assert W.shape == (N, K // 8) and s.shape == (N, K // 32)
    rr = None if r is None else _c(r, np.float64).reshape(batch)
    y = np.empty((batch, N), np.float64)
    A = np.empty((batch, N), np.float64)
    y16 = np.empty((batch, N), np.uint16)
    lib().wq4o_gemv(_p(W), _p(s), _p(x), N, K, batch, _p(rr), _p(y), _p(A), _p(y16))
    return y, A, y16


def tolerance(y_ref, A):
    """Per-element bound |y_gpu - y_ref| <= 1e-3 * A + ulp16(|y_ref|)."""
    return 1e-3 * np.asarray(A) + ulp16_array(np.abs(y_ref))


# ------------------------------------------------------------------- glue --

def rms_factor(v, eps: float) -> float:
    v = _c(v, np.uint16)
    return lib().wq4o_rms_factor(_p(v), v.size, float(eps))


def rms_normalize(u, eps: float) -> np.ndarray:
    """fp16 bits of fp16_RNE(r(u) * u), r(u) = 1 / sqrt(mean(u^2) + eps), per row."""
    u = np.atleast_2d(_c(u, np.uint16))
    v = np.empty(u.shape, np.uint16)
    for b in range(u.shape[0]):
        row = np.ascontiguousarray(u[b])
        out = np.empty(row.shape, np.uint16)
        lib().wq4o_rms_normalize(_p(row), row.size, float(eps), _p(out))
        v[b] = out
    return v


def rope(x, positions, head_dim: int, theta: float):
    """Rotary position embedding of the heads of each row (the paper names no
    positional encoding; its models, Llama-3.1 and Phi-3.5, rotate q and k).
    Reading: within each head, the adjacent pair (x_2i, x_2i+1) is the
    complex number x_2i + i x_2i+1 multiplied by exp(i pos w_i), with
    w_i = theta^(-2i / head_dim) and pos = positions[b] (the token's place in
    its sequence).  Inputs are fp16 bits [batch][n_heads * head_dim]; the
    rotation is exact in fp64 on the fp16 values and rounded once.

    Returns (fp64 [batch][n], fp16 bits [batch][n])."""
    x = np.atleast_2d(_c(x, np.uint16))
    batch, n = x.shape
    assert n % head_dim == 0 and head_dim % 2 == 0
    pos = np.asarray(positions, np.float64).reshape(batch, 1, 1)
    i = np.arange(head_dim // 2, dtype=np.float64)
    w = np.power(float(theta), -2.0 * i / head_dim)            # [head_dim / 2]
    ang = pos * w[None, None, :]                                # [batch][1][head_dim / 2]
    c, s = np.cos(ang), np.sin(ang)
    v = half_to_double(x).reshape(batch, n // head_dim, head_dim // 2, 2)
    re, im = v[..., 0], v[..., 1]
    out = np.stack([re * c - im * s, re * s + im * c], axis=-1).reshape(batch, n)
    return out, double_to_half(out)


def silu_mul(g, u):
    """-> (m fp64, m16 fp16 bits) with m = silu(g) * u."""
    g = _c(g, np.uint16)
    u = _c(u, np.uint16)
    m = np.empty(g.shape, np.float64)
    m16 = np.empty(g.shape, np.uint16)
    lib().wq4o_silu_mul(_p(g), _p(u), g.size, _p(m), _p(m16))
    return m, m16


def add_fp16(a, b) -> np.ndarray:
    a = _c(a, np.uint16)
    b = _c(b, np.uint16)
    z = np.empty(a.shape, np.uint16)
    lib().wq4o_add_fp16(_p(a), _p(b), a.size, _p(z))
    return z


# -------------------------------------------------------------- attention --

def paged_attention(q, k_cache, v_cache, page_table, seq_lens, scale: float, n_q_heads: int):
    """Decode attention over a paged cache (definition in attention_oracle.c).

    q          fp16 bits [batch][>= n_q_heads * head_dim] (row stride = q.shape[1])
    k_cache,
    v_cache    fp16 bits [num_pages][n_kv_heads][page_size][head_dim]
    page_table int32 [batch][pt_stride]
    seq_lens   int32 [batch]

    Returns (o fp64, A fp64, o16 fp16 bits), each [batch][n_q_heads][head_dim]."""
    q = _c(q, np.uint16)
    k_cache = _c(k_cache, np.uint16)
    v_cache = _c(v_cache, np.uint16)
    page_table = _c(np.atleast_2d(page_table), np.int32)
    seq_lens = _c(seq_lens, np.int32)
    num_pages, n_kv, page_size, head_dim = k_cache.shape
    assert v_cache.shape == k_cache.shape
    batch = seq_lens.shape[0]
    q2 = q.reshape(batch, -1)
    o = np.empty((batch, n_q_heads, head_dim), np.float64)
    A = np.empty_like(o)
    o16 = np.empty(o.shape, np.uint16)
    rc = lib().wq4o_paged_attention(_p(q2), q2.shape[1], _p(k_cache), _p(v_cache), num_pages, page_size,
                                    _p(page_table), page_table.shape[1], _p(seq_lens), batch, n_q_heads, n_kv,
                                    head_dim, float(scale), _p(o), _p(A), _p(o16))
    if rc != 0:
        raise ValueError("paged_attention: bad page id or head grouping")
    return o, A, o16


def kv_append(new_k, new_v, k_cache, v_cache, page_table, positions):
    """Writes each sequence's new key/value rows into the cache (in place).

    new_k, new_v fp16 bits [batch][>= n_kv_heads * head_dim]; the caches are
    modified in place.  Raises on a bad position or page id (after writing the
    other sequences)."""
    new_k = _c(new_k, np.uint16)
    new_v = _c(new_v, np.uint16)
    assert k_cache.flags.c_contiguous and v_cache.flags.c_contiguous
    assert k_cache.dtype == np.uint16 and v_cache.dtype == np.uint16
    page_table = _c(np.atleast_2d(page_table), np.int32)
    positions = _c(positions, np.int32)
    num_pages, n_kv, page_size, head_dim = k_cache.shape
    batch = positions.shape[0]
    nk = new_k.reshape(batch, -1)
    nv = new_v.reshape(batch, -1)
    assert nk.shape == nv.shape
    rc = lib().wq4o_kv_append(_p(nk), _p(nv), nk.shape[1], _p(k_cache), _p(v_cache), num_pages, page_size,
                              _p(page_table), page_table.shape[1], _p(positions), batch, n_kv, head_dim)
    if rc != 0:
        raise ValueError("kv_append: bad position or page id")


# Tolerance of the attention output.  The GPU path rounds each softmax weight
# to fp16 (relative error <= 2^-11) before the value product and sums the same
# rounded weights into the normaliser, so each normalised weight is off by at
# most about 2 * 2^-11 of itself; fp32 score and accumulation errors add
# < 1e-4 for scale * sum|q k| <= 64 and sequences of <= 64K tokens.  The bound
# 2e-3 * A covers both with margin; ulp16(|o|) covers the final rounding.
ATTN_REL = 2e-3


def attention_tolerance(o_ref, A):
    """Per-element bound |o_gpu - o_ref| <= 2e-3 * A + ulp16(|o_ref|)."""
    return ATTN_REL * np.asarray(A) + ulp16_array(np.abs(o_ref))
