"""Pins of the oracle to things other than itself (CPU only).

Each test fixes a part of the oracle against the format's definition, a
closed form, an invariant, a brute-force computation by library routines, or
a library's own fp16 conversion, so that a dropped term, a wrong sign, a wrong
nibble or group index or a transposed operand fails at least one of them.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import chain as ochain
from paper_2412_15803_gb300 import synth

RNG = np.random.default_rng(12345)


# ----------------------------------------------------------------- fp16 ----

def test_half_decode_exhaustive_vs_numpy():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    ours = oracle.half_to_double(bits)
    ref = bits.view(np.float16).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])
    # signs of zeros too
    assert np.array_equal(np.signbit(ours[~nan]), np.signbit(ref[~nan]))


def test_half_encode_roundtrip_all_finite():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    vals = bits.view(np.float16).astype(np.float64)
    fin = np.isfinite(vals)
    assert np.array_equal(oracle.double_to_half(vals[fin]), bits[fin])


def test_half_encode_ties_to_even_and_vs_libraries():
    # all midpoints between consecutive positive finite fp16 values
    bits = np.arange(0, 0x7BFF, dtype=np.uint16)
    lo = bits.view(np.float16).astype(np.float64)
    hi = (bits + 1).view(np.float16).astype(np.float64)
    mid = (lo + hi) / 2  # exact in fp64
    ours = oracle.double_to_half(mid)
    even = np.where(bits % 2 == 0, bits, bits + 1).astype(np.uint16)
    assert np.array_equal(ours, even)
    assert np.array_equal(oracle.double_to_half(-mid), even | np.uint16(0x8000))
    # just above / below a midpoint goes to the nearer neighbour
    assert np.array_equal(oracle.double_to_half(np.nextafter(mid, np.inf)), (bits + 1).astype(np.uint16))
    assert np.array_equal(oracle.double_to_half(np.nextafter(mid, -np.inf)), bits)
    # random doubles over the whole range: numpy and torch conversions
    v = np.concatenate([RNG.standard_normal(200000) * 10.0 ** RNG.integers(-9, 5, 200000),
                        RNG.uniform(-70000, 70000, 20000)])
    v = v[np.abs(v) < 65000]
    ours = oracle.double_to_half(v)
    assert np.array_equal(ours, v.astype(np.float16).view(np.uint16))
    # torch converts double -> half through float32 (two roundings), so it is
    # a reference only for inputs that are exact in float32
    v32 = v.astype(np.float32).astype(np.float64)
    tv = torch.from_numpy(v32).to(torch.float16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.double_to_half(v32), tv)


def test_half_encode_overflow_and_subnormal_edges():
    enc = lambda t: int(oracle.double_to_half(np.array([t]))[0])
    assert enc(65504.0) == 0x7BFF
    assert enc(65519.99) == 0x7BFF
    assert enc(65520.0) == 0x7C00
    assert enc(-1e9) == 0xFC00
    assert enc(2.0 ** -24) == 0x0001
    assert enc(2.0 ** -25) == 0x0000          # tie to even (0)
    assert enc(3 * 2.0 ** -25) == 0x0002      # tie to even (2)
    assert enc(2.0 ** -14 - 2.0 ** -26) == 0x0400  # rounds up into the normals
    assert enc(-0.0) == 0x8000


def test_ulp16_closed_forms_and_vs_nextafter():
    assert oracle.ulp16(1.0) == 2.0 ** -10
    assert oracle.ulp16(1.999) == 2.0 ** -10
    assert oracle.ulp16(2.0) == 2.0 ** -9
    assert oracle.ulp16(-3.0) == 2.0 ** -9
    assert oracle.ulp16(0.0) == 2.0 ** -24
    assert oracle.ulp16(2.0 ** -15) == 2.0 ** -24
    assert oracle.ulp16(2.0 ** -14) == 2.0 ** -24
    assert oracle.ulp16(65504.0) == 32.0
    # library: spacing between a binary16 value and the next one up
    vals = np.abs(RNG.standard_normal(2000) * 100).astype(np.float16)
    vals = vals[(vals < 60000) & (vals > 0)]
    nxt = np.nextafter(vals, np.float16(np.inf))
    for v, n in zip(vals.astype(np.float64), nxt.astype(np.float64)):
        assert oracle.ulp16(v) == n - v


# --------------------------------------------------------------- format ----

def test_nibble_order_hand_written_word():
    # codes 0..7 at k = 0..7: lowest nibble first
    W = np.array([[0x76543210, 0xFEDCBA98, 0, 0]], dtype=np.uint32)
    q, _ = oracle.unpack(W, np.zeros((1, 1), np.uint16), 32)
    assert list(q[0, :16]) == list(range(16))
    assert oracle.pack(q).tolist() == W.tolist()


def test_pack_unpack_exhaustive_per_position():
    K = 32
    for i in range(K):
        for v in range(16):
            q = np.zeros((1, K), np.uint8)
            q[0, i] = v
            W = oracle.pack(q)
            expect = np.zeros((1, K // 8), np.uint32)
            expect[0, i // 8] = v << (4 * (i % 8))
            assert np.array_equal(W, expect)
            q2, _ = oracle.unpack(W, np.zeros((1, 1), np.uint16), K)
            assert np.array_equal(q2, q)


def test_pack_unpack_random_words():
    W = RNG.integers(0, 2 ** 32, size=(7, 64 // 8), dtype=np.uint64).astype(np.uint32)
    q, _ = oracle.unpack(W, np.zeros((7, 2), np.uint16), 64)
    assert np.array_equal(oracle.pack(q), W)
    # numpy bit slicing (independent of the oracle's loops)
    nib = np.stack([(W >> np.uint32(4 * i)) & np.uint32(0xF) for i in range(8)], axis=-1)
    assert np.array_equal(q, nib.reshape(7, 64).astype(np.uint8))


def test_dequant_exact_vs_numpy():
    N, K = 5, 96
    q = RNG.integers(0, 16, size=(N, K), dtype=np.uint8)
    s = synth.scales_fp16(3, 9, 0, N * K // 32).reshape(N, K // 32)
    W = oracle.pack(q)
    q2, w = oracle.unpack(W, s, K)
    assert np.array_equal(q2, q)
    s64 = s.view(np.float16).astype(np.float64)
    ref = (q.astype(np.float64) - 7.0) * np.repeat(s64, 32, axis=1)
    assert np.array_equal(w, ref)
    assert w.min() >= -7 * s64.max() and w.max() <= 8 * s64.max()


# ----------------------------------------------------------------- GEMV ----

def _random_case(N, K, batch, seed=1):
    W, s = synth.matrix(seed, N, K)
    x = synth.activations(seed, batch, K)
    return W, s, x


def test_all_codes_seven_give_exact_zero():
    N, K, batch = 9, 256, 3
    _, s, x = _random_case(N, K, batch)
    W = oracle.pack(np.full((N, K), 7, np.uint8))
    y, A, y16 = oracle.gemv(W, s, x)
    assert np.all(y == 0.0) and np.all(A == 0.0)
    assert np.all((y16 & 0x7FFF) == 0)


@pytest.mark.parametrize("q", range(16))
def test_one_nonzero_group_closed_form(q):
    N, K, n0, g0 = 4, 128, 2, 1
    codes = np.full((N, K), 7, np.uint8)
    codes[n0, 32 * g0:32 * (g0 + 1)] = q
    W = oracle.pack(codes)
    s = np.full((N, K // 32), 0x2400, np.uint16)      # 2^-6
    x = np.zeros((1, K), np.uint16)
    x[0, 32 * g0:32 * (g0 + 1)] = 0x3C00               # 1.0 in that group
    x[0, :32 * g0] = 0x4000                            # 2.0 elsewhere: must not matter
    y, A, _ = oracle.gemv(W, s, x)
    expect = np.zeros((1, N))
    expect[0, n0] = 32 * (q - 7) * 2.0 ** -6
    assert np.array_equal(y, expect)
    assert np.array_equal(A, np.abs(expect))


def test_group_scale_index():
    # each group gets its own power-of-two scale; x = 1: y = sum_g 32 (q_g - 7) s_g
    K = 256
    codes = np.repeat(np.arange(8, dtype=np.uint8) + 4, 32)[None, :]   # group g has q = g + 4
    W = oracle.pack(codes)
    s_vals = 2.0 ** -np.arange(3, 11)
    s = s_vals.astype(np.float16).view(np.uint16)[None, :]
    x = np.full((1, K), 0x3C00, np.uint16)
    y, _, _ = oracle.gemv(W, s, x)
    expect = sum(32 * (g + 4 - 7) * s_vals[g] for g in range(8))
    assert y[0, 0] == expect


def test_linearity_in_x_and_s():
    N, K = 6, 192
    W, s, _ = _random_case(N, K, 1, seed=4)
    # small integers so every product and sum is exact in fp64
    x1 = RNG.integers(-8, 9, size=(1, K)).astype(np.float16).view(np.uint16)
    x2 = RNG.integers(-8, 9, size=(1, K)).astype(np.float16).view(np.uint16)
    alpha, beta = 4.0, -0.5
    xs = (alpha * x1.view(np.float16).astype(np.float64)
          + beta * x2.view(np.float16).astype(np.float64)).astype(np.float16).view(np.uint16)
    y1, _, _ = oracle.gemv(W, s, x1)
    y2, _, _ = oracle.gemv(W, s, x2)
    ys, _, _ = oracle.gemv(W, s, xs)
    assert np.array_equal(ys, alpha * y1 + beta * y2)
    s2 = (s.view(np.float16).astype(np.float64) * 2).astype(np.float16).view(np.uint16)
    yd, _, _ = oracle.gemv(W, s2, x1)
    assert np.array_equal(yd, 2 * y1)
    y4, A4, _ = oracle.gemv(W, s, x1, r=np.array([4.0]))
    _, A1, _ = oracle.gemv(W, s, x1)
    assert np.array_equal(y4, 4 * y1) and np.array_equal(A4, 4 * A1)


def test_fp16_output_is_one_rounding_of_the_fp64_sum():
    """y16 = fp16_RNE(y) with y the exact fp64 sum, not a rounding through
    fp32: y = 1 + 2^-11 + 2^-24 (codes 8, scale 1, x = 1, 2^-11, 2^-24; exact
    in fp64) lies just above the fp16 tie between 1 and 1 + 2^-10, so it
    rounds up to 0x3C01; rounded to fp32 first it would become the tie itself
    (2^-24 is half an fp32 ulp at 1) and then round to even, 0x3C00."""
    K = 32
    q = np.full((1, K), 7, np.uint8)
    q[0, :3] = 8
    W = oracle.pack(q)
    s = np.full((1, 1), 0x3C00, np.uint16)
    x = np.zeros((1, K), np.uint16)
    x[0, :3] = np.array([1.0, 2.0 ** -11, 2.0 ** -24]).astype(np.float16).view(np.uint16)
    y, A, y16 = oracle.gemv(W, s, x)
    assert y[0, 0] == 1.0 + 2.0 ** -11 + 2.0 ** -24 and A[0, 0] == y[0, 0]
    assert y16[0, 0] == 0x3C01


def test_row_factors_scale_their_own_batch_row():
    """Each batch row b takes its own factor r_b: with powers of two the
    scaling is exact, so y(r)[b] = r_b y(1)[b] bit for bit."""
    N, K, batch = 5, 128, 3
    W, s, x = _random_case(N, K, batch, seed=9)
    r = np.array([0.5, 4.0, 2.0 ** -3])
    y, A, _ = oracle.gemv(W, s, x)
    yr, Ar, _ = oracle.gemv(W, s, x, r=r)
    assert np.array_equal(yr, r[:, None] * y) and np.array_equal(Ar, r[:, None] * A)


@pytest.mark.parametrize("N,K,batch", [(1, 32, 1), (3, 32, 2), (4, 64, 1), (2, 64, 2), (4, 96, 3)])
def test_brute_force_vs_dense_numpy(N, K, batch):
    W, s, x = _random_case(N, K, batch, seed=N * 100 + K + batch)
    y, A, y16 = oracle.gemv(W, s, x)
    # dense dequantization with numpy bit ops, then a float64 matmul
    nib = np.stack([(W >> np.uint32(4 * i)) & np.uint32(0xF) for i in range(8)], axis=-1)
    q = nib.reshape(N, K).astype(np.float64)
    wd = (q - 7.0) * np.repeat(s.view(np.float16).astype(np.float64), 32, axis=1)
    xd = x.view(np.float16).astype(np.float64)
    y_np = xd @ wd.T
    A_np = np.abs(xd[:, None, :] * wd[None, :, :]).sum(-1)
    assert np.allclose(y, y_np, rtol=1e-13, atol=1e-15)
    assert np.allclose(A, A_np, rtol=1e-13, atol=1e-15)
    assert np.array_equal(y16, y.astype(np.float16).view(np.uint16))
    assert np.all(A >= np.abs(y))


def test_tolerance_formula_values():
    tol = oracle.tolerance(np.array([0.0, 1.0, 3.0]), np.array([0.0, 10.0, 0.0]))
    assert np.array_equal(tol, np.array([2.0 ** -24, 1e-2 + 2.0 ** -10, 2.0 ** -9]))


# ----------------------------------------------------------------- glue ----

def test_rms_factor_closed_forms():
    eps = 1e-5
    ones = np.full(64, 0x3C00, np.uint16)
    assert oracle.rms_factor(ones, eps) == 1.0 / math.sqrt(1.0 + eps)
    v = np.array([3.0, 4.0]).astype(np.float16).view(np.uint16)
    assert oracle.rms_factor(v, 0.0) == 1.0 / math.sqrt(12.5)
    assert oracle.rms_factor(np.zeros(8, np.uint16), 0.25) == 2.0


def test_silu_mul_values():
    g = np.array([0.0, 1.0, -1.0, 10.0, -20.0]).astype(np.float16).view(np.uint16)
    u = np.array([5.0, 1.0, 2.0, 1.0, 1.0]).astype(np.float16).view(np.uint16)
    m, m16 = oracle.silu_mul(g, u)
    expect = [0.0, 1.0 / (1.0 + math.exp(-1.0)), -2.0 / (1.0 + math.e),
              10.0 / (1.0 + math.exp(-10.0)), -20.0 / (1.0 + math.exp(20.0))]
    assert np.allclose(m, expect, rtol=1e-15, atol=0)
    assert m[1] == pytest.approx(0.7310585786300049, rel=1e-15)
    assert np.array_equal(m16, np.array(expect).astype(np.float16).view(np.uint16))


def test_add_fp16_rounding():
    one = 0x3C00
    a = np.array([one, one, one], np.uint16)
    b = np.array([2.0 ** -11, 3 * 2.0 ** -11, 2.0 ** -10]).astype(np.float16).view(np.uint16)
    z = oracle.add_fp16(a, b).view(np.float16).astype(np.float64)
    assert list(z) == [1.0, 1.0 + 2.0 ** -9, 1.0 + 2.0 ** -10]


# ---------------------------------------------------------------- chain ----

def _identity_like(N, K, value_code=8, scale=0x3C00):
    """code 8 (w = +s) at k == n for n < min(N, K), code 7 (w = 0) elsewhere."""
    q = np.full((N, K), 7, np.uint8)
    d = np.arange(min(N, K))
    q[d, d] = value_code
    return oracle.pack(q), np.full((N, K // 32), scale, np.uint16)


def test_rms_normalize_closed_forms():
    eps = 1e-5
    c = np.full(64, 0x4200, np.uint16)                      # 3.0
    v = oracle.rms_normalize(c, eps).view(np.float16).astype(np.float64)
    assert np.all(v == np.float16(3.0 / math.sqrt(9.0 + eps)))
    u = np.array([3.0, 4.0]).astype(np.float16).view(np.uint16)
    v = oracle.rms_normalize(u, 0.0).view(np.float16).astype(np.float64)[0]
    assert list(v) == [np.float16(3 / math.sqrt(12.5)), np.float16(4 / math.sqrt(12.5))]
    assert np.all(oracle.rms_normalize(np.zeros(8, np.uint16), 1.0) == 0)
    # rows are normalised independently
    two = np.stack([c, np.full(64, 0x4400, np.uint16)])  # rows of 3.0 and 4.0
    out = oracle.rms_normalize(two, 0.0).view(np.float16).astype(np.float64)
    assert np.all(out == 1.0)


def test_chain_all_sevens_passes_the_normalised_input_through():
    H, F, V, Nqkv, L, batch, eps = 64, 96, 80, 128, 3, 2, 1e-5
    rnd = lambda N, K: (oracle.pack(np.full((N, K), 7, np.uint8)),
                        synth.scales_fp16(2, N * K, 0, N * K // 32).reshape(N, K // 32))
    layers = [dict(qkv=rnd(Nqkv, H), o=rnd(H, H), gate_up=rnd(2 * F, H), down=rnd(H, F))
              for _ in range(L)]
    x = synth.activations(7, batch, H)
    logits, y, tr = ochain.token(x, layers, rnd(V, H), H, F, eps)
    assert np.all(y == 0.0)
    assert np.array_equal(tr[0]["v"], oracle.rms_normalize(x, eps))
    for t in tr[:-1]:
        assert np.all(t["qkv"] & 0x7FFF == 0) and np.all(t["d"] & 0x7FFF == 0)
        assert np.array_equal(t["x2"], t["v"])          # o = d = 0: output = layer input


def test_chain_gate_and_up_halves():
    """SiLU acts on the gate half (rows [0, F)) and multiplies the up half
    (rows [F, 2F)): with up rows weighting the input twice as much as the
    gate rows (code 9, w = 2s, against code 8, w = s), m = silu(g) * 2g,
    which silu(2g) * g does not match."""
    H, F, batch, eps = 64, 64, 2, 1e-5
    qg = np.full((2 * F, H), 7, np.uint8)
    qg[np.arange(F), np.arange(F)] = 8          # gate row j: x1[j]
    qg[F + np.arange(F), np.arange(F)] = 9      # up row j: 2 x1[j]
    layers = [dict(qkv=_identity_like(2 * H, H), o=_identity_like(H, H),
                   gate_up=(oracle.pack(qg), np.full((2 * F, H // 32), 0x3C00, np.uint16)),
                   down=_identity_like(H, F))]
    x = synth.activations(13, batch, H)
    _, _, tr = ochain.token(x, layers, _identity_like(H, H), H, F, eps)
    t = tr[0]
    gu = t["gu"].view(np.float16).astype(np.float64)
    g, up = gu[:, :F], gu[:, F:]
    assert np.array_equal(up, 2 * g)            # exact: fp16 doubling
    m = t["m"].view(np.float16).astype(np.float64)
    expect = (g / (1.0 + np.exp(-g)) * up).astype(np.float16).astype(np.float64)
    swapped = (up / (1.0 + np.exp(-up)) * g).astype(np.float16).astype(np.float64)
    assert np.allclose(m, expect, rtol=2.0 ** -10, atol=2.0 ** -24)
    assert not np.allclose(m, swapped, rtol=2.0 ** -8, atol=2.0 ** -20)


def test_chain_wiring_with_identity_projections():
    """Identity-like projections make every stage observable: the expected
    values follow from the stage definitions with numpy fp16 rounding."""
    H, F, batch, eps = 64, 64, 1, 1e-5
    Nqkv = 2 * H
    qg = np.full((2 * F, H), 7, np.uint8)
    qg[np.arange(F), np.arange(F)] = 8        # gate rows copy the input
    qg[F + np.arange(F), np.arange(F)] = 8    # up rows copy it too
    layers = [dict(qkv=_identity_like(Nqkv, H), o=_identity_like(H, H),
                   gate_up=(oracle.pack(qg), np.full((2 * F, H // 32), 0x3C00, np.uint16)),
                   down=_identity_like(H, F))]
    lm = _identity_like(H, H)
    x = synth.activations(11, batch, H)
    logits, y, tr = ochain.token(x, layers, lm, H, F, eps)

    f16 = lambda v: np.asarray(v, np.float64).astype(np.float16).astype(np.float64)
    xv = x.view(np.float16).astype(np.float64)[0]
    r = lambda v: 1.0 / np.sqrt(np.mean(v * v) + eps)
    v = f16(r(xv) * xv)                         # layer input after normalisation
    qkv = v                                     # first H rows copy v
    o = f16(r(qkv) * qkv)
    x1 = f16(v + o)
    g = f16(r(x1) * x1)
    m = f16(g / (1.0 + np.exp(-g)) * g)
    x2 = f16(x1 + m)
    lg = f16(r(x2) * x2)
    t = tr[0]
    h64 = lambda b: b.view(np.float16).astype(np.float64)[0]
    assert np.allclose(h64(t["v"]), v, rtol=2.0 ** -10, atol=0)
    assert np.array_equal(h64(t["qkv"])[:H], h64(t["v"])) and np.all(h64(t["qkv"])[H:] == 0)
    assert np.allclose(h64(t["o"]), o, rtol=2.0 ** -9, atol=2.0 ** -24)
    assert np.array_equal(h64(t["x1"]), f16(h64(t["v"]) + h64(t["o"])))
    assert np.allclose(h64(t["gu"]), np.concatenate([g, g]), rtol=2.0 ** -9, atol=2.0 ** -24)
    assert np.allclose(h64(t["m"]), m, rtol=2.0 ** -8, atol=2.0 ** -24)
    assert np.array_equal(h64(t["d"]), h64(t["m"]))
    assert np.array_equal(h64(t["x2"]), f16(h64(t["x1"]) + h64(t["d"])))
    assert np.allclose(logits.view(np.float16).astype(np.float64)[0], lg, rtol=2.0 ** -8, atol=2.0 ** -24)
