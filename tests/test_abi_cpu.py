"""The C ABI without a GPU: the library loads, exports every entry point its
headers declare, and rejects bad arguments before touching the device."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

import oracle
from paper_2412_15803_gb300 import wq4

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in ("wq4.h", "wq4_synth.h", "wq4_attn.h"):
        text = open(os.path.join(ROOT, "include", h)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names |= set(re.findall(r"^[A-Za-z_][\w \*]*?\b(wq4_\w+)\s*\(", text, flags=re.M))
    return names


def test_exports_every_declared_symbol():
    lib = wq4.load()
    names = declared_functions()
    assert len(names) >= 12
    assert names == set(wq4.EXPORTED)
    dyn = subprocess.run(["nm", "-D", "--defined-only", wq4.lib_path()], capture_output=True, text=True).stdout
    for n in names:
        assert hasattr(lib, n), n
        assert re.search(rf"\bT {n}$", dyn, flags=re.M), n


def test_status_strings():
    assert wq4.wq4_status_string(0) == "ok"
    assert "alignment" in wq4.wq4_status_string(-2) or "misaligned" in wq4.wq4_status_string(-2)
    assert wq4.wq4_status_string(12345) == "unknown status"


def test_pack_host_matches_oracle_and_rejects_bad_codes():
    q = np.random.default_rng(0).integers(0, 16, size=(5, 64), dtype=np.uint8)
    assert np.array_equal(wq4.wq4_pack_host(q), oracle.pack(q))
    q[2, 3] = 16
    with pytest.raises(wq4.Wq4Error):
        wq4.wq4_pack_host(q)


A16 = 1 << 20  # fake, 16-byte aligned "device" addresses: never dereferenced


@pytest.mark.parametrize("args,expect", [
    (dict(W=0), wq4.WQ4_ERR_INVALID),
    (dict(x=0), wq4.WQ4_ERR_INVALID),
    (dict(N=0), wq4.WQ4_ERR_INVALID),
    (dict(K=48), wq4.WQ4_ERR_INVALID),
    (dict(K=16), wq4.WQ4_ERR_INVALID),
    (dict(batch=0), wq4.WQ4_ERR_INVALID),
    (dict(batch=33), wq4.WQ4_ERR_INVALID),
    (dict(W=A16 + 4), wq4.WQ4_ERR_ALIGN),
    (dict(x=8 * A16 + 8), wq4.WQ4_ERR_ALIGN),
    (dict(s=2 * A16 + 1), wq4.WQ4_ERR_ALIGN),
    (dict(y=A16 + 64), wq4.WQ4_ERR_INVALID),   # y overlaps W
])
def test_gemv_rejects_bad_arguments(args, expect):
    a = dict(W=A16, s=2 * A16, x=8 * A16, y=16 * A16, N=64, K=256, batch=1)
    a.update(args)
    rc = wq4.load().wq4_gemv(a["W"], a["s"], a["x"], a["y"], a["N"], a["K"], a["batch"], None)
    assert rc == expect


@pytest.mark.parametrize("args,expect", [
    (dict(W=0), wq4.WQ4_ERR_INVALID),
    (dict(M=0), wq4.WQ4_ERR_INVALID),
    (dict(N=0), wq4.WQ4_ERR_INVALID),
    (dict(K=48), wq4.WQ4_ERR_INVALID),
    (dict(K=288), wq4.WQ4_ERR_UNSUPPORTED),
    (dict(N=100), wq4.WQ4_ERR_UNSUPPORTED),
    (dict(s=2 * A16 + 8), wq4.WQ4_ERR_ALIGN),
    (dict(y=16 * A16 + 8), wq4.WQ4_ERR_ALIGN),
    (dict(y=A16 + 64), wq4.WQ4_ERR_INVALID),   # y overlaps W
])
def test_gemm_rejects_bad_arguments(args, expect):
    a = dict(W=A16, s=2 * A16, x=8 * A16, y=16 * A16, N=64, K=256, M=300)
    a.update(args)
    rc = wq4.load().wq4_gemm(a["W"], a["s"], a["x"], a["y"], a["N"], a["K"], a["M"], None)
    assert rc == expect


def test_unpack_debug_rejects_bad_arguments():
    L = wq4.load()
    assert L.wq4_unpack_debug(A16, 2 * A16, None, None, 4, 64, None) == wq4.WQ4_ERR_INVALID
    assert L.wq4_unpack_debug(A16, 2 * A16, 4 * A16 + 2, None, 4, 64, None) == wq4.WQ4_ERR_ALIGN
    assert L.wq4_unpack_debug(A16, 2 * A16, 4 * A16, None, 4, 40, None) == wq4.WQ4_ERR_INVALID


def _table(**kw):
    layers = (wq4.wq4_layer * 2)()
    t = wq4.wq4_layer_table()
    t.num_layers, t.hidden, t.ffn, t.n_q_heads, t.n_kv_heads, t.head_dim = 2, 256, 512, 2, 1, 128
    t.vocab, t.batch, t.rms_eps = 1000, 1, 1e-5
    t.layers = layers
    for k, v in kw.items():
        setattr(t, k, v)
    return t, layers


def test_chain_workspace_bytes_and_invalid_tables():
    t, _ = _table()
    n = wq4.wq4_chain_workspace_bytes(t)
    assert n > 0 and n % 256 == 0
    t4, _ = _table(batch=4)
    assert wq4.wq4_chain_workspace_bytes(t4) > n
    for bad in (dict(hidden=200), dict(ffn=100), dict(n_q_heads=3), dict(batch=0), dict(batch=33),
                dict(vocab=0), dict(rms_eps=0.0), dict(num_layers=0)):
        tb, _ = _table(**bad)
        assert wq4.wq4_chain_workspace_bytes(tb) == 0, bad
        assert wq4.load().wq4_decode_chain(ctypes.byref(tb), A16, 2 * A16, None) == wq4.WQ4_ERR_INVALID


def test_chain_trace_offsets_are_disjoint_and_inside_workspace():
    t, _ = _table(batch=2)
    total = wq4.wq4_chain_workspace_bytes(t)
    spans = []
    lens = dict(x_in=256, qkv=512, o=256, x_mid=256, gate_up=1024, act=512, down=256, x_out=256)
    for layer in range(2):
        off = wq4.wq4_chain_trace_offsets(t, layer)
        for name, n in lens.items():
            o = getattr(off, name)
            assert o % 2 == 0 and o + 2 * 2 * n <= total
            spans.append((o, o + 4 * n))
    spans.append((wq4.wq4_chain_trace_offsets(t, 2).x_in, wq4.wq4_chain_trace_offsets(t, 2).x_in + 4 * 256))
    spans.sort()
    for (a0, a1), (b0, b1) in zip(spans, spans[1:]):
        assert a1 <= b0
    with pytest.raises(wq4.Wq4Error):
        wq4.wq4_chain_trace_offsets(t, 3)


def test_chain_rejects_null_and_misaligned_io():
    t, _ = _table()
    L = wq4.load()
    assert L.wq4_decode_chain(ctypes.byref(t), None, A16, None) == wq4.WQ4_ERR_INVALID
    assert L.wq4_decode_chain(ctypes.byref(t), A16 + 8, 2 * A16, None) == wq4.WQ4_ERR_ALIGN
    assert L.wq4_chain_plan_destroy(ctypes.byref(t)) == wq4.WQ4_ERR_INVALID
    assert L.wq4_chain_path(ctypes.byref(t), 0) == wq4.WQ4_ERR_INVALID      # no plan was built


def test_synth_rejects_bad_arguments():
    L = wq4.load()
    assert L.wq4_synth_codes(A16, 1, 4, 0, 0, 0, None) == -1
    assert L.wq4_synth_codes(A16, 0, 3, 0, 0, 1, None) == -1
    assert L.wq4_synth_scales(None, 0, 4, 0, 0, 0.005, 0.02, None) == -1

    assert L.wq4_synth_sum4(None, 0, 4, 0, 0, None) == -1
    assert L.wq4_synth_sum4(A16, -1, 4, 0, 0, None) == -1


def _cache(**kw):
    c = wq4.wq4_kv_cache(A16, 64 * A16, 64, 2, 16, 128, 128 * A16, 8)
    for k, v in kw.items():
        setattr(c, k, v)
    return c


@pytest.mark.parametrize("cache_kw,call_kw,expect", [
    (dict(), dict(q=0), wq4.WQ4_ERR_INVALID),
    (dict(k=0), dict(), wq4.WQ4_ERR_INVALID),
    (dict(page_table=0), dict(), wq4.WQ4_ERR_INVALID),
    (dict(page_size=8), dict(), wq4.WQ4_ERR_INVALID),
    (dict(page_size=24), dict(), wq4.WQ4_ERR_INVALID),
    (dict(num_pages=0), dict(), wq4.WQ4_ERR_INVALID),
    (dict(), dict(batch=0), wq4.WQ4_ERR_INVALID),
    (dict(), dict(batch=1025), wq4.WQ4_ERR_INVALID),
    (dict(), dict(n_q_heads=5), wq4.WQ4_ERR_INVALID),
    (dict(), dict(n_q_heads=1), wq4.WQ4_ERR_INVALID),
    (dict(head_dim=64), dict(), wq4.WQ4_ERR_UNSUPPORTED),
    (dict(), dict(n_q_heads=18), wq4.WQ4_ERR_UNSUPPORTED),
    (dict(), dict(q_stride=1000), wq4.WQ4_ERR_INVALID),
    (dict(), dict(q=256 * A16 + 8), wq4.WQ4_ERR_ALIGN),
    (dict(), dict(q_stride=1028), wq4.WQ4_ERR_ALIGN),
    (dict(k=A16 + 2), dict(), wq4.WQ4_ERR_ALIGN),
    (dict(), dict(scale=float("nan")), wq4.WQ4_ERR_INVALID),
])
def test_paged_attention_rejects_bad_arguments(cache_kw, call_kw, expect):
    a = dict(q=256 * A16, q_stride=1024, lens=300 * A16, out=400 * A16, out_stride=1024, batch=2, n_q_heads=8,
             scale=0.088, ws=500 * A16, ws_bytes=1 << 30)
    a.update(call_kw)
    c = _cache(**cache_kw)
    rc = wq4.load().wq4_paged_attention(ctypes.byref(c), a["q"], a["q_stride"], a["lens"], a["out"],
                                        a["out_stride"], a["batch"], a["n_q_heads"], a["scale"], a["ws"],
                                        a["ws_bytes"], None)
    assert rc == expect


def test_paged_attention_workspace_bytes_rejects_bad_geometry():
    L = wq4.load()
    for args in ((0, 8, 2, 128), (2, 8, 2, 64), (2, 6, 4, 128), (2, 36, 4, 128), (2000, 8, 2, 128)):
        assert L.wq4_paged_attention_workspace_bytes(*args) == 0


def test_kv_append_rejects_bad_arguments():
    L = wq4.load()
    c = _cache()
    assert L.wq4_kv_append(ctypes.byref(c), None, A16 * 2, 256, A16 * 3, 1, None) == wq4.WQ4_ERR_INVALID
    assert L.wq4_kv_append(ctypes.byref(c), 200 * A16, 210 * A16, 100, 220 * A16, 1, None) == wq4.WQ4_ERR_INVALID
    assert L.wq4_kv_append(ctypes.byref(c), 200 * A16 + 8, 210 * A16, 256, 220 * A16, 1, None) == wq4.WQ4_ERR_ALIGN
    c64 = _cache(head_dim=64)
    assert L.wq4_kv_append(ctypes.byref(c64), 200 * A16, 210 * A16, 256, 220 * A16, 1, None) == wq4.WQ4_ERR_UNSUPPORTED


def test_chain_wait_hook_rejects_bad_values():
    lib = wq4.load()
    assert lib.wq4_test_chain_waits(0, -1) == wq4.WQ4_ERR_INVALID
    assert lib.wq4_test_chain_waits(500_000_001, -1) == wq4.WQ4_ERR_INVALID
    assert lib.wq4_test_chain_waits(1000, -2) == wq4.WQ4_ERR_INVALID
    assert lib.wq4_test_chain_waits(500_000_000, -1) == wq4.WQ4_OK


def test_gemv_path_hook_rejects_bad_values():
    lib = wq4.load()
    assert lib.wq4_test_gemv_path(-1) == wq4.WQ4_ERR_INVALID
    assert lib.wq4_test_gemv_path(3) == wq4.WQ4_ERR_INVALID
    assert lib.wq4_test_gemv_path(0) == wq4.WQ4_OK
