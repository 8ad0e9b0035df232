"""Python binding of the wq4 C ABI (include/wq4.h): argument marshalling only.

Every function here has the name of the C entry point it calls; tensors are
passed as raw device (or host) addresses, every computation runs in the CUDA
library.  Loading fails loudly when libwq4.so is missing: there is no other
implementation to fall back to.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

WQ4_OK = 0
WQ4_ERR_INVALID = -1
WQ4_ERR_ALIGN = -2
WQ4_ERR_UNSUPPORTED = -3
WQ4_ERR_CUDA = -4
WQ4_ERR_TIMEOUT = -5
WQ4_MAX_BATCH = 32

_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_U64 = ctypes.c_uint64
_SZ = ctypes.c_size_t


class Wq4Error(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} failed: {status} ({wq4_status_string(status)})")
        self.status = status


class wq4_mat(ctypes.Structure):
    _fields_ = [("W", _P), ("s", _P)]


class wq4_layer(ctypes.Structure):
    _fields_ = [("qkv", wq4_mat), ("o", wq4_mat), ("gate_up", wq4_mat), ("down", wq4_mat)]


class wq4_layer_table(ctypes.Structure):
    _fields_ = [("num_layers", _I), ("hidden", _I), ("ffn", _I), ("n_q_heads", _I),
                ("n_kv_heads", _I), ("head_dim", _I), ("vocab", _I), ("batch", _I),
                ("rms_eps", ctypes.c_float), ("layers", ctypes.POINTER(wq4_layer)),
                ("lm_head", wq4_mat), ("workspace", _P), ("workspace_bytes", _SZ)]


class wq4_kv_cache(ctypes.Structure):
    _fields_ = [("k", _P), ("v", _P), ("num_pages", _I), ("n_kv_heads", _I), ("page_size", _I),
                ("head_dim", _I), ("page_table", _P), ("page_table_stride", _I)]


class wq4_chain_trace(ctypes.Structure):
    _fields_ = [(n, _SZ) for n in ("x_in", "qkv", "o", "x_mid", "gate_up", "act", "down", "x_out",
                                   "q_rot", "k_rot", "attn")]


class wq4_decode_attn(ctypes.Structure):
    _fields_ = [("layers", ctypes.POINTER(wq4_kv_cache)), ("positions", _P), ("rope_theta", ctypes.c_double),
                ("scale", ctypes.c_float)]


_lib = None


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Loads libwq4.so (building it first when asked and it is stale)."""
    global _lib
    if _lib is not None:
        return _lib
    if build_if_missing:
        _build.build()
    if not os.path.exists(_build.LIB):
        raise RuntimeError(f"libwq4.so not found at {_build.LIB}: build it with "
                           "`python -m paper_2412_15803_gb300.build`")
    L = ctypes.CDLL(_build.LIB)
    L.wq4_gemv.argtypes = [_P, _P, _P, _P, _I, _I, _I, _P]
    L.wq4_gemm.argtypes = [_P, _P, _P, _P, _I, _I, _I, _P]
    L.wq4_unpack_debug.argtypes = [_P, _P, _P, _P, _I, _I, _P]
    L.wq4_pack_host.argtypes = [_P, _P, _I, _I]
    L.wq4_status_string.argtypes = [_I]
    L.wq4_status_string.restype = ctypes.c_char_p
    L.wq4_device_status.argtypes = [_P, ctypes.POINTER(_I)]
    L.wq4_chain_workspace_bytes.argtypes = [ctypes.POINTER(wq4_layer_table)]
    L.wq4_chain_workspace_bytes.restype = _SZ
    L.wq4_decode_chain.argtypes = [ctypes.POINTER(wq4_layer_table), _P, _P, _P]
    L.wq4_decode_chain_host.argtypes = [ctypes.POINTER(wq4_layer_table), _P, _P, _P]
    L.wq4_decode_chain_noalloc.argtypes = [ctypes.POINTER(wq4_layer_table), _P, _P, _P]
    L.wq4_chain_plan_destroy.argtypes = [ctypes.POINTER(wq4_layer_table)]
    L.wq4_chain_path.argtypes = [ctypes.POINTER(wq4_layer_table), _I]
    L.wq4_chain_trace_offsets.argtypes = [ctypes.POINTER(wq4_layer_table), _I,
                                          ctypes.POINTER(wq4_chain_trace)]
    L.wq4_test_chain_waits.argtypes = [_U64, _I]
    L.wq4_test_gemv_path.argtypes = [_I]
    L.wq4_decode_step_workspace_bytes.argtypes = [ctypes.POINTER(wq4_layer_table)]
    L.wq4_decode_step_workspace_bytes.restype = _SZ
    L.wq4_decode_step.argtypes = [ctypes.POINTER(wq4_layer_table), ctypes.POINTER(wq4_decode_attn), _P, _P, _P]
    L.wq4_decode_step_host.argtypes = [ctypes.POINTER(wq4_layer_table), ctypes.POINTER(wq4_decode_attn), _P, _P, _P]
    L.wq4_synth_codes.argtypes = [_P, _I64, _I64, _U64, _U64, _I, _P]
    L.wq4_synth_scales.argtypes = [_P, _I64, _I64, _U64, _U64, ctypes.c_double, ctypes.c_double, _P]
    L.wq4_synth_sum4.argtypes = [_P, _I64, _I64, _U64, _U64, _P]
    L.wq4_paged_attention_workspace_bytes.argtypes = [_I, _I, _I, _I]
    L.wq4_paged_attention_workspace_bytes.restype = _SZ
    L.wq4_paged_attention.argtypes = [ctypes.POINTER(wq4_kv_cache), _P, _I, _P, _P, _I, _I, _I, ctypes.c_float,
                                      _P, _SZ, _P]
    L.wq4_kv_append.argtypes = [ctypes.POINTER(wq4_kv_cache), _P, _P, _I, _P, _I, _P]
    _lib = L
    return L


# names every C entry point of include/*.h (checked by the tests)
EXPORTED = ["wq4_gemv", "wq4_gemm", "wq4_unpack_debug", "wq4_pack_host", "wq4_status_string",
            "wq4_device_status", "wq4_chain_workspace_bytes", "wq4_decode_chain",
            "wq4_decode_chain_host", "wq4_decode_chain_noalloc", "wq4_chain_plan_destroy", "wq4_chain_path",
            "wq4_chain_trace_offsets",
            "wq4_test_chain_waits", "wq4_test_gemv_path", "wq4_decode_step_workspace_bytes", "wq4_decode_step", "wq4_decode_step_host",
            "wq4_synth_codes", "wq4_synth_scales", "wq4_synth_sum4",
            "wq4_paged_attention_workspace_bytes", "wq4_paged_attention", "wq4_kv_append"]


def _ptr(t) -> int | None:
    """Address of a torch tensor / numpy array, or an int passed through."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if hasattr(t, "data_ptr"):
        return t.data_ptr()
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    raise TypeError(f"cannot take the address of {type(t)}")


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(fn: str, rc: int) -> int:
    if rc != WQ4_OK:
        raise Wq4Error(fn, rc)
    return rc


def wq4_status_string(status: int) -> str:
    return load().wq4_status_string(int(status)).decode()


def wq4_gemv(W, scales, x, y, N: int, K: int, batch: int, stream=None, check: bool = True) -> int:
    rc = load().wq4_gemv(_ptr(W), _ptr(scales), _ptr(x), _ptr(y), N, K, batch, _stream(stream))
    return _check("wq4_gemv", rc) if check else rc


def wq4_gemm(W, scales, x, y, N: int, K: int, M: int, stream=None, check: bool = True) -> int:
    rc = load().wq4_gemm(_ptr(W), _ptr(scales), _ptr(x), _ptr(y), N, K, M, _stream(stream))
    return _check("wq4_gemm", rc) if check else rc


def wq4_unpack_debug(W, scales, w_out, q_out, N: int, K: int, stream=None, check: bool = True) -> int:
    rc = load().wq4_unpack_debug(_ptr(W), _ptr(scales), _ptr(w_out), _ptr(q_out), N, K, _stream(stream))
    return _check("wq4_unpack_debug", rc) if check else rc


def wq4_pack_host(q: np.ndarray) -> np.ndarray:
    q = np.ascontiguousarray(q, dtype=np.uint8)
    N, K = q.shape
    W = np.empty((N, K // 8), np.uint32)
    _check("wq4_pack_host", load().wq4_pack_host(q.ctypes.data, W.ctypes.data, N, K))
    return W


def wq4_device_status(stream=None) -> int:
    flags = _I(0)
    rc = load().wq4_device_status(_stream(stream), ctypes.byref(flags))
    if rc not in (WQ4_OK, WQ4_ERR_TIMEOUT):
        raise Wq4Error("wq4_device_status", rc)
    return flags.value


def wq4_chain_workspace_bytes(table: wq4_layer_table) -> int:
    return load().wq4_chain_workspace_bytes(ctypes.byref(table))


def wq4_decode_chain(table: wq4_layer_table, x, logits, stream=None, check: bool = True) -> int:
    rc = load().wq4_decode_chain(ctypes.byref(table), _ptr(x), _ptr(logits), _stream(stream))
    return _check("wq4_decode_chain", rc) if check else rc


def wq4_decode_chain_host(table: wq4_layer_table, x_host, logits_host, stream=None, check: bool = True) -> int:
    rc = load().wq4_decode_chain_host(ctypes.byref(table), _ptr(x_host), _ptr(logits_host), _stream(stream))
    return _check("wq4_decode_chain_host", rc) if check else rc


def wq4_decode_chain_noalloc(table: wq4_layer_table, x, logits, stream=None, check: bool = True) -> int:
    rc = load().wq4_decode_chain_noalloc(ctypes.byref(table), _ptr(x), _ptr(logits), _stream(stream))
    return _check("wq4_decode_chain_noalloc", rc) if check else rc


def wq4_chain_plan_destroy(table: wq4_layer_table) -> int:
    return load().wq4_chain_plan_destroy(ctypes.byref(table))


def wq4_chain_path(table: wq4_layer_table, decode_step: bool = False) -> int:
    """1: the table's cached plan runs the persistent chain kernel; 2: the
    tensor-core stage graph.  Raises if no plan exists yet."""
    rc = load().wq4_chain_path(ctypes.byref(table), 1 if decode_step else 0)
    if rc < 0:
        raise Wq4Error("wq4_chain_path", rc)
    return rc


def wq4_chain_trace_offsets(table: wq4_layer_table, layer: int) -> wq4_chain_trace:
    out = wq4_chain_trace()
    _check("wq4_chain_trace_offsets", load().wq4_chain_trace_offsets(ctypes.byref(table), layer, ctypes.byref(out)))
    return out


def wq4_decode_step_workspace_bytes(table: wq4_layer_table) -> int:
    return load().wq4_decode_step_workspace_bytes(ctypes.byref(table))


def wq4_decode_step(table: wq4_layer_table, attn: wq4_decode_attn, x, logits, stream=None, check: bool = True) -> int:
    rc = load().wq4_decode_step(ctypes.byref(table), ctypes.byref(attn), _ptr(x), _ptr(logits), _stream(stream))
    return _check("wq4_decode_step", rc) if check else rc


def wq4_decode_step_host(table: wq4_layer_table, attn: wq4_decode_attn, x_host, logits_host, stream=None,
                         check: bool = True) -> int:
    rc = load().wq4_decode_step_host(ctypes.byref(table), ctypes.byref(attn), _ptr(x_host), _ptr(logits_host),
                                     _stream(stream))
    return _check("wq4_decode_step_host", rc) if check else rc


def wq4_test_gemv_path(path: int) -> None:
    """Test hook: 0 size rule, 1 legacy-tensor-path kernel, 2 CUDA-core kernel (batch 1-2)."""
    _check("wq4_test_gemv_path", load().wq4_test_gemv_path(path))


def wq4_test_chain_waits(wait_limit_ns: int, stall_stage: int = -1) -> None:
    """Test hook: limit of the chain kernel's device waits and a stage whose
    input waits are made to run out (-1: none)."""
    _check("wq4_test_chain_waits", load().wq4_test_chain_waits(wait_limit_ns, stall_stage))


def wq4_synth_codes(W, word_start: int, nwords: int, seed: int, sid: int, symmetric: bool = False,
                    stream=None) -> None:
    rc = load().wq4_synth_codes(_ptr(W), word_start, nwords, seed, sid, int(bool(symmetric)), _stream(stream))
    if rc != 0:
        raise Wq4Error("wq4_synth_codes", rc)


def wq4_synth_scales(s, start: int, n: int, seed: int, sid: int, lo: float, hi: float, stream=None) -> None:
    rc = load().wq4_synth_scales(_ptr(s), start, n, seed, sid, lo, hi, _stream(stream))
    if rc != 0:
        raise Wq4Error("wq4_synth_scales", rc)


def wq4_synth_sum4(out, start: int, n: int, seed: int, sid: int, stream=None) -> None:
    rc = load().wq4_synth_sum4(_ptr(out), start, n, seed, sid, _stream(stream))
    if rc != 0:
        raise Wq4Error("wq4_synth_sum4", rc)


def kv_cache_desc(k, v, page_table, page_size: int) -> wq4_kv_cache:
    """wq4_kv_cache of device tensors k, v [num_pages][n_kv_heads][page_size][head_dim]
    and page_table int32 [batch][stride]."""
    num_pages, n_kv, ps, head_dim = k.shape
    if ps != page_size:
        raise ValueError("cache shape does not match page_size")
    return wq4_kv_cache(_ptr(k), _ptr(v), num_pages, n_kv, page_size, head_dim, _ptr(page_table),
                        page_table.shape[1])


def wq4_paged_attention_workspace_bytes(batch: int, n_q_heads: int, n_kv_heads: int, head_dim: int) -> int:
    return load().wq4_paged_attention_workspace_bytes(batch, n_q_heads, n_kv_heads, head_dim)


def wq4_paged_attention(cache: wq4_kv_cache, q, q_stride: int, seq_lens, out, out_stride: int, batch: int,
                        n_q_heads: int, scale: float, workspace, workspace_bytes: int, stream=None,
                        check: bool = True) -> int:
    rc = load().wq4_paged_attention(ctypes.byref(cache), _ptr(q), q_stride, _ptr(seq_lens), _ptr(out), out_stride,
                                    batch, n_q_heads, scale, _ptr(workspace), workspace_bytes, _stream(stream))
    return _check("wq4_paged_attention", rc) if check else rc


def wq4_kv_append(cache: wq4_kv_cache, new_k, new_v, new_stride: int, positions, batch: int, stream=None,
                  check: bool = True) -> int:
    rc = load().wq4_kv_append(ctypes.byref(cache), _ptr(new_k), _ptr(new_v), new_stride, _ptr(positions), batch,
                              _stream(stream))
    return _check("wq4_kv_append", rc) if check else rc
