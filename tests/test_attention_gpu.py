"""GPU parity of paged decode attention and the cache append against the oracle.

The bar: every output element within
|o_gpu - o_ref| <= 2e-3 * sum_t p_t |V_t| + ulp16(|o_ref|)   (o_ref, p from the fp64 oracle);
the append and the device sum4 generator bit-exact.  All calls go through the C ABI.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2412_15803_gb300 import synth, wq4
from paper_2412_15803_gb300.attention import ATTN_WORKLOADS, PagedAttentionLayer
from paper_2412_15803_gb300.model import SHAPES

pytestmark = pytest.mark.gpu

NAN16 = np.uint16(0x7E00)


def dev(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a).view(dtype)).cuda()


def run_attention(q, k, v, table, lens, Hq, scale, q_stride=None, out_stride=None, ws=None, check_status=True):
    batch = len(lens)
    Hkv, P, D = k.shape[1], k.shape[2], k.shape[3]
    q_stride = q.shape[1] if q_stride is None else q_stride
    out_stride = Hq * D if out_stride is None else out_stride
    qd = torch.zeros((batch, q_stride), dtype=torch.int16, device="cuda")
    qd[:, :q.shape[1]] = dev(q, np.int16)
    kd, vd = dev(k, np.int16), dev(v, np.int16)
    td, ld = dev(table.astype(np.int32), np.int32), dev(np.asarray(lens, np.int32), np.int32)
    out = torch.full((batch, out_stride), -1, dtype=torch.int16, device="cuda")
    nbytes = wq4.wq4_paged_attention_workspace_bytes(batch, Hq, Hkv, D)
    assert nbytes > 0
    if ws is None:
        ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    cache = wq4.kv_cache_desc(kd, vd, td, P)
    wq4.wq4_paged_attention(cache, qd, q_stride, ld, out, out_stride, batch, Hq, scale, ws, ws.numel())
    torch.cuda.synchronize()
    if check_status:
        assert wq4.wq4_device_status() == 0
    o = out.cpu().numpy().view(np.uint16)
    return o[:, :Hq * D].reshape(batch, Hq, D), o, ws


def check(o16_gpu, q, k, v, table, lens, Hq, scale):
    o_ref, A, _ = oracle.paged_attention(q, k, v, table, lens, scale, Hq)
    og = oracle.half_to_double(o16_gpu)
    tol = oracle.attention_tolerance(o_ref, A)
    err = np.abs(og - o_ref)
    bad = np.argwhere(~(err <= tol))
    assert bad.size == 0, (f"{len(bad)} elements out of tolerance, first {bad[:3]}, "
                           f"err {err[tuple(bad[0])]} tol {tol[tuple(bad[0])]}")
    return float((err / tol).max())


def make_case(seed, lens, Hq, Hkv, P, spare=2, garbage=True):
    D = 128
    lens = np.asarray(lens, np.int32)
    num_pages = int(((lens.astype(np.int64) + P - 1) // P).sum()) + spare
    k, v = synth.kv_cache(seed, num_pages, Hkv, P, D)
    table = synth.page_table(seed, lens, P, num_pages)
    q = synth.queries(seed, len(lens), Hq, D)
    if garbage:
        # rows past each sequence's end and unreferenced pages hold NaN
        k, v = k.copy(), v.copy()
        for b, T in enumerate(lens):
            if T > 0 and T % P:
                last = table[b][(T - 1) // P]
                k[last, :, T % P:] = NAN16
                v[last, :, T % P:] = NAN16
        used = set(table[table >= 0].tolist())
        for p in range(num_pages):
            if p not in used:
                k[p] = NAN16
                v[p] = NAN16
    return q, k, v, table, lens


# ------------------------------------------------------------- generator --

def test_device_sum4_matches_host():
    n = 100_003
    out = torch.empty(n + 5, dtype=torch.int16, device="cuda")
    wq4.wq4_synth_sum4(out, 12345, n, 7, 99)
    torch.cuda.synchronize()
    assert np.array_equal(out[:n].cpu().numpy().view(np.uint16), synth.sum4_fp16(7, 99, 12345, n))


# ---------------------------------------------------------------- parity --

LEN_MIXES = {
    "ragged": [1, 15, 16, 17, 100, 333],
    "long": [1000, 2049],
    "one": [5],
    "with_empty": [0, 40, 0, 7],
}


@pytest.mark.parametrize("Hq,Hkv", [(32, 8), (24, 8), (8, 1), (4, 4)])
@pytest.mark.parametrize("mix", list(LEN_MIXES))
def test_parity_small(Hq, Hkv, mix):
    lens = LEN_MIXES[mix]
    q, k, v, table, lens = make_case(3, lens, Hq, Hkv, 16)
    scale = 1.0 / math.sqrt(128)
    o16, _, _ = run_attention(q, k, v, table, lens, Hq, scale)
    check(o16, q, k, v, table, lens, Hq, scale)
    for b, T in enumerate(lens):
        if T == 0:
            assert np.all(o16[b] == 0)


@pytest.mark.parametrize("P", [32, 64, 256])
def test_parity_page_sizes(P):
    q, k, v, table, lens = make_case(5, [3, 31, 64, 65, 700], 32, 8, P)
    scale = 1.0 / math.sqrt(128)
    o16, _, _ = run_attention(q, k, v, table, lens, 32, scale)
    check(o16, q, k, v, table, lens, 32, scale)


def test_parity_strided_rows_and_peaked_scores():
    """q read from QKV-shaped rows (stride > Hq * D), output into wider rows,
    scale 1 (softmax close to one-hot): strides honoured, tail untouched."""
    q, k, v, table, lens = make_case(6, [50, 129], 8, 2, 16)
    qs = 8 * 128 + 2 * 2 * 128
    o16, full, _ = run_attention(q, k, v, table, lens, 8, 1.0, q_stride=qs, out_stride=8 * 128 + 64)
    check(o16, q, k, v, table, lens, 8, 1.0)
    assert np.all(full[:, 8 * 128:] == 0xFFFF)


def test_deterministic_and_counters_left_zero():
    q, k, v, table, lens = make_case(8, [900, 17, 3000], 32, 8, 16)
    scale = 1.0 / math.sqrt(128)
    o1, _, ws = run_attention(q, k, v, table, lens, 32, scale)
    assert int(ws[: 4 * 3 * 8].count_nonzero()) == 0   # arrival counters
    o2, _, _ = run_attention(q, k, v, table, lens, 32, scale, ws=ws)
    assert np.array_equal(o1, o2)


def test_graph_replay():
    layer = PagedAttentionLayer(SHAPES["8b"], [300, 5000, 64], seed=11)
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        layer.run(stream=s)
        s.synchronize()
        ref = layer.out.clone()
        layer.out.fill_(0)
        with torch.cuda.graph(g, stream=s):
            layer.run(stream=s)
    for _ in range(3):
        layer.out.fill_(0)
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(layer.out, ref)
    assert wq4.wq4_device_status() == 0


# ------------------------------------------------------------ full sizes --

@pytest.mark.parametrize("name", ["attn-8b", "attn-3b"])
def test_full_size_sampled(name):
    """The benchmark's workload and launch: whole output computed, sampled
    sequences (shortest, longest, two others) checked against the oracle."""
    w = ATTN_WORKLOADS[name]
    layer = PagedAttentionLayer(w.shape, w.lens(0), page_size=w.page_size, seed=0)
    layer.run()
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    out = layer.out.cpu().numpy().view(np.uint16)
    Hq, D = w.shape.n_q_heads, w.shape.head_dim
    order = np.argsort(layer.lens)
    for b in sorted({int(order[0]), int(order[-1]), int(order[len(order) // 2]), 7}):
        q, k, v, table, lens = layer.host_sequence(b)
        check(out[b].reshape(1, Hq, D), q, k, v, table, lens, Hq, layer.scale)


def test_longest_sequence_sampled():
    """One sequence of 32768 tokens next to short ones (page table 2048 wide)."""
    layer = PagedAttentionLayer(SHAPES["8b"], [32768, 3, 700], seed=2)
    layer.run()
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    out = layer.out.cpu().numpy().view(np.uint16)
    for b in range(3):
        q, k, v, table, lens = layer.host_sequence(b)
        check(out[b].reshape(1, 32, 128), q, k, v, table, lens, 32, layer.scale)


# ----------------------------------------------------------- error paths --

def test_bad_page_id_and_length_are_flagged_not_faulted():
    q, k, v, table, lens = make_case(9, [40, 20], 8, 2, 16, garbage=False)
    bad = table.copy()
    bad[0, 1] = k.shape[0] + 1000
    run_attention(q, k, v, bad, lens, 8, 0.1, check_status=False)
    assert wq4.wq4_device_status() & 16
    long = np.array([40, 20 + 16 * table.shape[1]], np.int32)   # beyond the page table
    run_attention(q, k, v, table, long, 8, 0.1, check_status=False)
    assert wq4.wq4_device_status() & 8


def test_workspace_too_small_is_rejected():
    q, k, v, table, lens = make_case(9, [40], 8, 2, 16, garbage=False)
    nbytes = wq4.wq4_paged_attention_workspace_bytes(1, 8, 2, 128)
    ws = torch.zeros(nbytes - 16, dtype=torch.uint8, device="cuda")
    kd, vd = dev(k, np.int16), dev(v, np.int16)
    td, ld = dev(table, np.int32), dev(lens, np.int32)
    qd = dev(q, np.int16)
    out = torch.empty((1, 8 * 128), dtype=torch.int16, device="cuda")
    cache = wq4.kv_cache_desc(kd, vd, td, 16)
    rc = wq4.wq4_paged_attention(cache, qd, 8 * 128, ld, out, 8 * 128, 1, 8, 0.1, ws, ws.numel(), check=False)
    assert rc == wq4.WQ4_ERR_INVALID


# ---------------------------------------------------------------- append --

def test_kv_append_bit_exact_then_attend():
    Hq, Hkv, D, P = 32, 8, 128, 16
    lens = np.array([5, 16, 33, 0], np.int32)
    num_pages = 12
    k, v = synth.kv_cache(4, num_pages, Hkv, P, D)
    table = synth.page_table(4, lens + 1, P, num_pages)
    # new rows inside QKV-shaped rows: k at offset Hq*D, v at (Hq+Hkv)*D
    nq = (Hq + 2 * Hkv) * D
    qkv = synth.sum4_fp16(4, 200, 0, 4 * nq).reshape(4, nq)
    kd, vd = dev(k, np.int16), dev(v, np.int16)
    td, pd = dev(table, np.int32), dev(lens, np.int32)
    qkvd = dev(qkv, np.int16)
    cache = wq4.kv_cache_desc(kd, vd, td, P)
    wq4.wq4_kv_append(cache, qkvd[:, Hq * D:], qkvd[:, (Hq + Hkv) * D:], nq, pd, 4)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    k2, v2 = k.copy(), v.copy()
    oracle.kv_append(qkv[:, Hq * D:(Hq + Hkv) * D], qkv[:, (Hq + Hkv) * D:], k2, v2, table, lens)
    assert np.array_equal(kd.cpu().numpy().view(np.uint16), k2)
    assert np.array_equal(vd.cpu().numpy().view(np.uint16), v2)
    o16, _, _ = run_attention(qkv, k2, v2, table, lens + 1, Hq, 1 / math.sqrt(D), q_stride=nq)
    check(o16, qkv, k2, v2, table, lens + 1, Hq, 1 / math.sqrt(D))


def test_kv_append_bad_position_is_flagged():
    k, v = synth.kv_cache(4, 2, 1, 16, 128)
    kd, vd = dev(k, np.int16), dev(v, np.int16)
    td = dev(np.array([[0, 1]], np.int32), np.int32)
    pd = dev(np.array([32], np.int32), np.int32)   # beyond the 2-page table
    new = torch.zeros((1, 128), dtype=torch.int16, device="cuda")
    cache = wq4.kv_cache_desc(kd, vd, td, 16)
    wq4.wq4_kv_append(cache, new, new, 128, pd, 1)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() & 32
    assert np.array_equal(kd.cpu().numpy().view(np.uint16), k)
