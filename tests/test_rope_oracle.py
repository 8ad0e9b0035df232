"""Pins of the oracle's rotary embedding and of the attention step of its
decode chain (CPU only).

The paper names no positional encoding; the models it decodes rotate q and k
(rotary embedding).  The reading pinned here: adjacent pairs (2i, 2i+1) of a
head turn by pos * theta^(-2i / head_dim), on the fp16 values, rounded once.
The pins are closed forms (unit vectors through known angles), invariants of
a rotation (pair norms, dependence of q.k on the position difference only),
the complex-number form of the same map, and chain cases whose attention
result is fixed without the oracle (one token; two tokens).
"""
import math

import numpy as np

import oracle
from oracle import chain as ochain
from paper_2412_15803_gb300 import synth


def f16(v):
    return np.asarray(v, np.float64).astype(np.float16).view(np.uint16)


def h64(b):
    return np.asarray(b, np.uint16).view(np.float16).astype(np.float64)


def test_position_zero_is_the_identity():
    x = synth.sum4_fp16(1, 77, 0, 3 * 256).reshape(3, 256)
    _, out = oracle.rope(x, [0, 0, 0], 128, 500000.0)
    assert np.array_equal(out, x)


def test_unit_vectors_through_known_angles():
    """head_dim 4, theta 10000: w_0 = 1, w_1 = 10000^(-1/2) = 0.01."""
    c1, s1 = math.cos(1.0), math.sin(1.0)
    e = np.eye(4)
    y, _ = oracle.rope(f16(e[0][None]), [1], 4, 10000.0)        # pair 0 by 1 rad
    assert np.allclose(y[0], [c1, s1, 0, 0], rtol=0, atol=1e-15)
    y, _ = oracle.rope(f16(e[1][None]), [1], 4, 10000.0)        # the imaginary unit turns to (-sin, cos)
    assert np.allclose(y[0], [-s1, c1, 0, 0], rtol=0, atol=1e-15)
    y, _ = oracle.rope(f16(e[2][None]), [100], 4, 10000.0)      # pair 1 by 100 * 0.01 = 1 rad
    assert np.allclose(y[0], [0, 0, c1, s1], rtol=0, atol=1e-14)
    y, _ = oracle.rope(f16(e[0][None]), [3], 4, 10000.0)        # pair 0 by 3 rad
    assert np.allclose(y[0], [math.cos(3.0), math.sin(3.0), 0, 0], rtol=0, atol=1e-15)


def test_every_head_turns_alike():
    """The angle depends on the index within the head, not on the head."""
    x = synth.sum4_fp16(2, 5, 0, 128).reshape(1, 128)
    two = np.concatenate([x, x], axis=1)
    y1, _ = oracle.rope(x, [37], 64, 10000.0)
    y2, _ = oracle.rope(two, [37], 64, 10000.0)
    assert np.array_equal(y2[:, :128], y1) and np.array_equal(y2[:, 128:], y1)


def test_pair_norms_are_preserved():
    x = synth.sum4_fp16(3, 9, 0, 2 * 256).reshape(2, 256)
    y, _ = oracle.rope(x, [5, 4093], 128, 500000.0)
    a = h64(x).reshape(2, -1, 2)
    b = y.reshape(2, -1, 2)
    assert np.allclose((b * b).sum(-1), (a * a).sum(-1), rtol=1e-14, atol=0)


def test_scores_depend_on_the_position_difference_only():
    """rope(q, m) . rope(k, n) = q . rope(k, n - m) for every head."""
    D = 128
    q = synth.sum4_fp16(4, 1, 0, D).reshape(1, D)
    k = synth.sum4_fp16(4, 2, 0, D).reshape(1, D)
    dots = []
    for m, n in [(7, 3), (107, 103), (4011, 4007)]:
        qm, _ = oracle.rope(q, [m], D, 500000.0)
        kn, _ = oracle.rope(k, [n], D, 500000.0)
        dots.append(float(qm[0] @ kn[0]))
    k4, _ = oracle.rope(k, [-4], D, 500000.0)
    ref = float(h64(q)[0] @ k4[0])
    assert np.allclose(dots, ref, rtol=1e-11, atol=0)
    q0, _ = oracle.rope(q, [0], D, 500000.0)
    k0, _ = oracle.rope(k, [0], D, 500000.0)
    assert not np.isclose(float(q0[0] @ k0[0]), ref, rtol=1e-3)   # the difference matters


def test_complex_multiplication_form():
    D, theta = 96, 10000.0
    x = synth.sum4_fp16(5, 3, 0, 2 * 4 * D).reshape(2, 4 * D)
    pos = np.array([11, 2047])
    y, y16 = oracle.rope(x, pos, D, theta)
    z = h64(x).reshape(2, 4, D // 2, 2)
    zc = z[..., 0] + 1j * z[..., 1]
    freq = theta ** (-np.arange(0, D, 2) / D)
    zr = zc * np.exp(1j * pos[:, None, None] * freq[None, None, :])
    expect = np.stack([zr.real, zr.imag], axis=-1).reshape(2, 4 * D)
    assert np.allclose(y, expect, rtol=0, atol=1e-12)
    assert np.array_equal(y16, f16(expect))                  # one rounding of the exact value


def test_rows_use_their_own_positions():
    x = np.repeat(synth.sum4_fp16(6, 1, 0, 128).reshape(1, 128), 2, axis=0)
    y, _ = oracle.rope(x, [3, 9], 128, 10000.0)
    y3, _ = oracle.rope(x[:1], [3], 128, 10000.0)
    y9, _ = oracle.rope(x[:1], [9], 128, 10000.0)
    assert np.array_equal(y[0], y3[0]) and np.array_equal(y[1], y9[0])


# -------------------------------------------------- the chain's attention --

def _ident(N, K, code=8, scale=0x3C00, offset=0):
    """Row n copies input n - offset (code 8, w = +1), other weights 0."""
    q = np.full((N, K), 7, np.uint8)
    for n in range(N):
        k = n - offset
        if 0 <= k < K:
            q[n, k] = code
    return oracle.pack(q), np.full((N, K // 32), scale, np.uint16)


def _attn_desc(nq, nkv, D, batch, positions, pages_per_seq=2, P=16, seed=0):
    num_pages = batch * pages_per_seq
    k, v = synth.kv_cache(seed, num_pages, nkv, P, D)
    table = np.arange(num_pages, dtype=np.int32).reshape(batch, pages_per_seq)[:, ::-1].copy()
    return dict(n_q_heads=nq, n_kv_heads=nkv, head_dim=D, theta=10000.0, scale=1.0 / math.sqrt(D),
                positions=np.asarray(positions, np.int32), k_cache=k.copy(), v_cache=v.copy(), page_table=table)


def _qkv_layer(H, F, Nqkv):
    """QKV rows copy the layer input cyclically (q, k, v all see v = r(u) u),
    other projections identity-like."""
    q = np.full((Nqkv, H), 7, np.uint8)
    q[np.arange(Nqkv), np.arange(Nqkv) % H] = 8
    qkv = (oracle.pack(q), np.full((Nqkv, H // 32), 0x3C00, np.uint16))
    return dict(qkv=qkv, o=_ident(H, H), gate_up=_ident(2 * F, H), down=_ident(H, F))


def test_first_token_attends_to_itself_only():
    """At position 0 the rotation is the identity and the sequence holds the
    new token alone: each query head's output is its kv head's new value,
    and the cache's row 0 holds the new key and value."""
    H, F, D, nq, nkv, batch = 128, 64, 32, 4, 2, 2
    Nqkv = (nq + 2 * nkv) * D
    at = _attn_desc(nq, nkv, D, batch, [0, 0])
    x = synth.activations(3, batch, H)
    _, _, tr = ochain.token(x, [_qkv_layer(H, F, Nqkv)], _ident(H, H), H, F, 1e-5, [at])
    t = tr[0]
    qkv = t["qkv"]
    v_new = qkv[:, H + nkv * D:].reshape(batch, nkv, D)
    G = nq // nkv
    a = t["attn"].reshape(batch, nq, D)
    for j in range(nq):
        assert np.array_equal(a[:, j], v_new[:, j // G])
    assert np.array_equal(t["q_rot"], qkv[:, :H])
    for b in range(batch):
        page = at["page_table"][b, 0]
        assert np.array_equal(at["k_cache"][page, :, 0, :], qkv[b, H:H + nkv * D].reshape(nkv, D))
        assert np.array_equal(at["v_cache"][page, :, 0, :], v_new[b])


def test_two_tokens_closed_form():
    """Position 1: the cached token 0 (key k0, value v0) and the new token.
    QKV copies the normalised input v: q = v (two heads), k = v[:D] / 8,
    value = v[D:].  The cached key is k0 = v[:D] / 8 as well, so an
    unrotated query would score both keys alike; the rotation turns q by one
    position against k0 and by none against the new key (both turned by the
    same angle).  The output is the softmax mix of v0 and the new value."""
    H, F, D, nq, nkv, batch, eps = 64, 64, 32, 2, 1, 1, 1e-5
    Nqkv = (nq + 2 * nkv) * D
    q = np.full((Nqkv, H), 7, np.uint8)
    q[np.arange(Nqkv), np.arange(Nqkv) % H] = 8
    sc = np.full((Nqkv, H // 32), 0x3C00, np.uint16)
    sc[H:H + D] = 0x3000                                   # k rows: w = 1/8
    layer = dict(qkv=(oracle.pack(q), sc), o=_ident(H, H), gate_up=_ident(2 * F, H), down=_ident(H, F))
    at = _attn_desc(nq, nkv, D, batch, [1])
    x = synth.activations(8, batch, H)
    v_in = h64(oracle.rms_normalize(x, eps))[0]
    page = at["page_table"][0, 0]
    at["k_cache"][page, 0, 0] = f16(v_in[:D] / 8)
    _, _, tr = ochain.token(x, [layer], _ident(H, H), H, F, eps, [at])
    t = tr[0]
    qkv = h64(t["qkv"])[0]
    assert np.array_equal(qkv[:H], v_in) and np.array_equal(qkv[H:H + D], v_in[:D] / 8)
    k0 = h64(at["k_cache"][page, 0, 0])
    v0 = h64(at["v_cache"][page, 0, 0])
    v1 = qkv[H + D:H + 2 * D]
    kn = qkv[H:H + D]
    freq = 10000.0 ** (-np.arange(0, D, 2) / D)
    for j in range(nq):
        qj = qkv[j * D:(j + 1) * D]
        qc = (qj[0::2] + 1j * qj[1::2]) * np.exp(1j * freq)            # rope(q, 1) as complex pairs
        s0 = float(np.real(np.sum(qc * np.conj(k0[0::2] + 1j * k0[1::2])))) / math.sqrt(D)
        s1 = float(qj @ kn) / math.sqrt(D)                              # same angle on both sides
        e0, e1 = math.exp(s0), math.exp(s1)
        expect = (e0 * v0 + e1 * v1) / (e0 + e1)
        got = h64(t["attn"])[0, j * D:(j + 1) * D]
        assert np.allclose(got, expect, rtol=2e-3, atol=2e-3), j
        if j == 0:
            # unrotated, both keys score alike: the plain mean, which differs
            assert not np.allclose(got, (v0 + v1) / 2, rtol=2e-3, atol=2e-3)
    # the new token went to row 1 of the first page, rotated
    krot = h64(t["k_rot"])[0]
    assert np.array_equal(h64(at["k_cache"][page, 0, 1]), krot)
    assert not np.array_equal(krot, kn)


def test_attention_output_feeds_the_o_projection():
    """With O the identity, o = fp16(r(a) a) for the attention output a, not
    for the query block."""
    H, F, D, nq, nkv, batch = 64, 64, 32, 2, 1, 1
    Nqkv = (nq + 2 * nkv) * D
    at = _attn_desc(nq, nkv, D, batch, [5])
    x = synth.activations(9, batch, H)
    _, _, tr = ochain.token(x, [_qkv_layer(H, F, Nqkv)], _ident(H, H), H, F, 1e-5, [at])
    t = tr[0]
    a = h64(t["attn"])[0]
    r = 1.0 / math.sqrt(np.mean(a * a) + 1e-5)
    assert np.allclose(h64(t["o"])[0], a * r, rtol=2.0 ** -9, atol=2.0 ** -24)
    q = h64(t["qkv"])[0, :H]
    assert not np.allclose(h64(t["o"])[0], q / math.sqrt(np.mean(q * q) + 1e-5), rtol=1e-2)
