"""Pins of the decode-attention oracle (oracle/attention_oracle.c).

Each test fixes the oracle to something other than itself: a library routine
(torch's scaled-dot-product attention in fp64 on the gathered cache), closed
forms (one token; equal scores; two tokens), invariances of the definition
(physical page order, data outside the sequence, the sign of the values) and
brute-force indexing of the append step.  A dropped term, a wrong page or
head index, a wrong scale or an off-by-one in the sequence length fails at
least one of them.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2412_15803_gb300 import synth


def _f16(a):
    return np.asarray(a, np.float16).view(np.uint16)


def _case(seed=1, lens=(1, 17, 100), Hq=8, Hkv=2, D=128, P=16, spare=3):
    lens = np.asarray(lens, np.int32)
    num_pages = int(((lens + P - 1) // P).sum()) + spare
    k, v = synth.kv_cache(seed, num_pages, Hkv, P, D)
    table = synth.page_table(seed, lens, P, num_pages)
    q = synth.queries(seed, len(lens), Hq, D)
    return q, k, v, table, lens


def _gather(cache, table, b, h, T, P):
    rows = [cache[table[b][t // P], h, t % P] for t in range(T)]
    return np.stack(rows) if rows else np.zeros((0, cache.shape[-1]), np.uint16)


def _sdpa_ref(q, k, v, table, lens, scale, Hq):
    """torch SDPA (fp64, CPU) on the gathered contiguous keys and values."""
    batch = len(lens)
    Hkv, P, D = k.shape[1], k.shape[2], k.shape[3]
    G = Hq // Hkv
    out = np.zeros((batch, Hq, D))
    for b in range(batch):
        T = int(lens[b])
        qb = torch.from_numpy(oracle.half_to_double(q[b].reshape(Hq, D)))[None, :, None, :]
        kb = np.stack([oracle.half_to_double(_gather(k, table, b, h, T, P)) for h in range(Hkv)])
        vb = np.stack([oracle.half_to_double(_gather(v, table, b, h, T, P)) for h in range(Hkv)])
        kt = torch.from_numpy(kb).repeat_interleave(G, dim=0)[None]
        vt = torch.from_numpy(vb).repeat_interleave(G, dim=0)[None]
        o = torch.nn.functional.scaled_dot_product_attention(qb, kt, vt, scale=scale)
        out[b] = o[0, :, 0, :].numpy()
    return out


@pytest.mark.parametrize("Hq,Hkv,D,P", [(8, 2, 128, 16), (6, 2, 64, 32), (4, 4, 128, 16)])
def test_matches_torch_sdpa(Hq, Hkv, D, P):
    q, k, v, table, lens = _case(Hq=Hq, Hkv=Hkv, D=D, P=P)
    scale = 1.0 / math.sqrt(D)
    o, A, o16 = oracle.paged_attention(q, k, v, table, lens, scale, Hq)
    ref = _sdpa_ref(q, k, v, table, lens, scale, Hq)
    assert np.max(np.abs(o - ref)) <= 1e-12
    assert np.all(A >= np.abs(o) - 1e-15)
    assert np.array_equal(o16, oracle.double_to_half(o))


def test_large_scores_do_not_overflow():
    """Scores of several thousand: exp without the max shift would overflow."""
    q, k, v, table, lens = _case(lens=(40, 9))
    o, _, _ = oracle.paged_attention(q, k, v, table, lens, 400.0, 8)
    assert np.all(np.isfinite(o))
    ref = _sdpa_ref(q, k, v, table, lens, 400.0, 8)
    assert np.max(np.abs(o - ref)) <= 1e-9


def test_single_token_returns_its_value():
    q, k, v, table, lens = _case(lens=(1, 1))
    o, A, _ = oracle.paged_attention(q, k, v, table, lens, 0.125, 8)
    for b in range(2):
        for j in range(8):
            vt = oracle.half_to_double(v[table[b][0], j // 4, 0])
            assert np.array_equal(o[b, j], vt)
            assert np.array_equal(A[b, j], np.abs(vt))


def test_equal_scores_give_the_mean():
    """q = 0: every weight is 1/T, so o is the exactly rounded mean (the fp64
    sum of these fp16 values is exact)."""
    q, k, v, table, lens = _case(lens=(37, 200))
    q = np.zeros_like(q)
    o, _, _ = oracle.paged_attention(q, k, v, table, lens, 0.3, 8)
    for b, T in enumerate(lens):
        for j in (0, 5):
            vals = oracle.half_to_double(_gather(v, table, b, j // 4, int(T), 16))
            mean = np.array([math.fsum(vals[:, d]) / int(T) for d in range(vals.shape[1])])
            assert np.array_equal(o[b, j], mean)


def test_fp16_output_is_one_rounding_of_the_fp64_value():
    """o16 = fp16_RNE(o) of the fp64 value, rounded once: four tokens with
    equal scores (q = 0) and values 4, 2^-9, 2^-22, 0 in dimension 0 give
    o = 1 + 2^-11 + 2^-24 exactly, just above the fp16 tie between 1 and
    1 + 2^-10, so 0x3C01; a rounding through fp32 first would land on the
    tie and round to even (0x3C00)."""
    D, P = 128, 16
    k = synth.sum4_fp16(5, 9, 0, P * D).reshape(1, 1, P, D)
    v = np.zeros((1, 1, P, D), np.uint16)
    v[0, 0, :4, 0] = _f16(np.array([4.0, 2.0 ** -9, 2.0 ** -22, 0.0]))
    q = np.zeros((1, D), np.uint16)
    o, _, o16 = oracle.paged_attention(q, k, v, np.array([[0]]), np.array([4]), 0.1, 1)
    assert o[0, 0, 0] == 1.0 + 2.0 ** -11 + 2.0 ** -24
    assert o16[0, 0, 0] == 0x3C01


def test_two_tokens_closed_form():
    """Scores a and 0: o = (e^a v0 + v1) / (e^a + 1)."""
    D, P = 128, 16
    k = np.zeros((1, 1, P, D), np.uint16)
    v = synth.sum4_fp16(3, 9, 0, P * D).reshape(1, 1, P, D)
    a = 1.75
    k[0, 0, 0, 0] = _f16(a)
    q = np.zeros((1, D), np.uint16)
    q[0, 0] = _f16(1.0)
    o, A, _ = oracle.paged_attention(q, k, v, np.array([[0]]), np.array([2]), 1.0, 1)
    v0 = oracle.half_to_double(v[0, 0, 0])
    v1 = oracle.half_to_double(v[0, 0, 1])
    ea = math.exp(a)
    want = (ea * v0 + v1) / (ea + 1.0)
    assert np.max(np.abs(o[0, 0] - want)) <= 1e-15
    assert np.max(np.abs(A[0, 0] - (ea * np.abs(v0) + np.abs(v1)) / (ea + 1.0))) <= 1e-15


def test_physical_page_order_does_not_matter():
    q, k, v, table, lens = _case(lens=(50, 33, 16))
    o1, A1, _ = oracle.paged_attention(q, k, v, table, lens, 0.1, 8)
    perm = np.random.default_rng(0).permutation(k.shape[0])
    inv = np.argsort(perm)
    k2, v2 = k[perm], v[perm]          # page p moves to slot inv[p]
    t2 = np.where(table >= 0, inv[np.maximum(table, 0)], -1).astype(np.int32)
    o2, A2, _ = oracle.paged_attention(q, k2, v2, t2, lens, 0.1, 8)
    assert np.array_equal(o1, o2) and np.array_equal(A1, A2)


def test_data_outside_the_sequence_is_ignored():
    """Rows past the length in the last page and unreferenced pages (filled
    with NaN here) change nothing; a length one larger does."""
    q, k, v, table, lens = _case(lens=(20, 5))
    o1, _, _ = oracle.paged_attention(q, k, v, table, lens, 0.1, 8)
    k2, v2 = k.copy(), v.copy()
    nan = _f16(np.nan)
    for b, T in enumerate(lens):
        last = table[b][(T - 1) // 16]
        k2[last, :, T % 16:] = nan
        v2[last, :, T % 16:] = nan
    used = set(table[table >= 0].tolist())
    for p in range(k.shape[0]):
        if p not in used:
            k2[p] = nan
            v2[p] = nan
    o2, _, _ = oracle.paged_attention(q, k2, v2, table, lens, 0.1, 8)
    assert np.array_equal(o1, o2)
    o3, _, _ = oracle.paged_attention(q, k, v, table, lens + 1, 0.1, 8)
    assert not np.array_equal(o1[0], o3[0])


def test_value_sign_and_magnitude():
    q, k, v, table, lens = _case(lens=(30, 7))
    o, A, _ = oracle.paged_attention(q, k, v, table, lens, 0.1, 8)
    vneg = v ^ np.uint16(0x8000)
    o2, A2, _ = oracle.paged_attention(q, k, vneg, table, lens, 0.1, 8)
    assert np.array_equal(o2, -o) and np.array_equal(A2, A)
    vabs = v & np.uint16(0x7FFF)
    o3, A3, _ = oracle.paged_attention(q, k, vabs, table, lens, 0.1, 8)
    assert np.array_equal(o3, A3) and np.array_equal(A3, A)


def test_query_heads_share_their_group():
    """Heads 0-3 read kv head 0, heads 4-7 kv head 1: changing kv head 1
    moves only the second group."""
    q, k, v, table, lens = _case(lens=(25,))
    o1, _, _ = oracle.paged_attention(q, k, v, table, lens, 0.1, 8)
    v2 = v.copy()
    v2[:, 1] = v2[:, 1] ^ np.uint16(0x8000)
    o2, _, _ = oracle.paged_attention(q, k, v2, table, lens, 0.1, 8)
    assert np.array_equal(o1[0, :4], o2[0, :4])
    assert np.array_equal(o1[0, 4:], -o2[0, 4:])


def test_empty_sequence_gives_zero():
    q, k, v, table, lens = _case(lens=(0, 3))
    o, A, o16 = oracle.paged_attention(q, k, v, table, lens, 0.1, 8)
    assert np.all(o[0] == 0) and np.all(A[0] == 0) and np.all(o16[0] == 0)
    assert np.any(o[1] != 0)


def test_bad_page_id_raises():
    q, k, v, table, lens = _case(lens=(20,))
    table = table.copy()
    table[0, 1] = k.shape[0]
    with pytest.raises(ValueError):
        oracle.paged_attention(q, k, v, table, lens, 0.1, 8)


def test_kv_append_brute_force():
    """The append writes exactly the rows [page(pos)][h][pos % P] and nothing else."""
    Hkv, D, P = 2, 128, 16
    lens = np.array([5, 16, 33], np.int32)
    num_pages = 9
    k, v = synth.kv_cache(4, num_pages, Hkv, P, D)
    table = synth.page_table(4, lens + 1, P, num_pages)
    newk = synth.sum4_fp16(4, 100, 0, 3 * Hkv * D).reshape(3, Hkv * D)
    newv = synth.sum4_fp16(4, 101, 0, 3 * Hkv * D).reshape(3, Hkv * D)
    k2, v2 = k.copy(), v.copy()
    oracle.kv_append(newk, newv, k2, v2, table, lens)
    changed = np.argwhere(np.any(k2 != k, axis=-1))
    want = set()
    for b, pos in enumerate(lens):
        for h in range(Hkv):
            page, row = table[b][pos // P], pos % P
            want.add((page, h, row))
            assert np.array_equal(k2[page, h, row], newk[b, h * D:(h + 1) * D])
            assert np.array_equal(v2[page, h, row], newv[b, h * D:(h + 1) * D])
    assert {tuple(c) for c in changed} <= want
    # the appended token is attended to at length pos + 1
    q = synth.queries(4, 3, 4, D)
    o, _, _ = oracle.paged_attention(q, k2, v2, table, lens + 1, 0.1, 4)
    ref = _sdpa_ref(q, k2, v2, table, lens + 1, 0.1, 4)
    assert np.max(np.abs(o - ref)) <= 1e-12


def test_kv_append_rejects_bad_position():
    k, v = synth.kv_cache(4, 2, 1, 16, 128)
    table = np.array([[0, 1]], np.int32)
    newk = np.zeros((1, 128), np.uint16)
    with pytest.raises(ValueError):
        oracle.kv_append(newk, newk, k, v, table, np.array([-1], np.int32))


def test_sum4_distribution():
    x = synth.sum4_fp16(0, 1, 0, 1 << 16).view(np.float16).astype(np.float64)
    assert abs(x.mean()) < 0.02
    assert abs(x.std() - 2 / math.sqrt(3)) < 0.02
    assert x.min() >= -4 and x.max() <= 4
    # the same elements at any offset
    assert np.array_equal(synth.sum4_fp16(0, 1, 1000, 10), synth.sum4_fp16(0, 1, 0, 1010)[1000:])
