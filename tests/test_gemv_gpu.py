"""GPU parity of the GEMV, the unpack and the device generator against the oracle.

The bar: unpack bit-exact; every y element within
|y_gpu - y_ref| <= 1e-3 * sum_k |w x| + ulp16(|y_ref|)  (y_ref, A from the fp64 oracle).
All calls go through the C ABI.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2412_15803_gb300 import synth, wq4

pytestmark = pytest.mark.gpu


def dev(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a).view(dtype)).cuda()


def run_gemv(W, s, x, N, K, batch, s_offset_elems=0):
    Wd = dev(W, np.int32)
    if s_offset_elems:
        sd_full = torch.zeros(s.size + s_offset_elems, dtype=torch.int16, device="cuda")
        sd_full[s_offset_elems:] = dev(s.ravel(), np.int16)
        sd = sd_full[s_offset_elems:]
    else:
        sd = dev(s, np.int16)
    xd = dev(x, np.int16)
    y = torch.full((batch, N), -1, dtype=torch.int16, device="cuda")
    wq4.wq4_gemv(Wd, sd, xd, y, N, K, batch)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    return y.cpu().numpy().view(np.uint16)


def check(y16_gpu, W, s, x, rows=None):
    y_ref, A, _ = oracle.gemv(W, s, x)
    g = y16_gpu if rows is None else y16_gpu[:, rows]
    yg = oracle.half_to_double(g)
    tol = oracle.tolerance(y_ref, A)
    err = np.abs(yg - y_ref)
    bad = np.argwhere(~(err <= tol))
    assert bad.size == 0, f"{len(bad)} elements out of tolerance, first {bad[:3]}, err {err[tuple(bad[0])]} tol {tol[tuple(bad[0])]}"
    return float((err / np.maximum(tol, 1e-30)).max())


# ------------------------------------------------------------------ unpack --

@pytest.mark.parametrize("N,K", [(3, 32), (17, 256), (64, 3072), (5, 14336)])
def test_unpack_bit_exact(N, K):
    W, s = synth.matrix(21, N, K)
    q_ref, w_ref = oracle.unpack(W, s, K)
    Wd, sd = dev(W, np.int32), dev(s, np.int16)
    q = torch.empty((N, K), dtype=torch.uint8, device="cuda")
    w = torch.empty((N, K), dtype=torch.float32, device="cuda")
    wq4.wq4_unpack_debug(Wd, sd, w, q, N, K)
    torch.cuda.synchronize()
    assert np.array_equal(q.cpu().numpy(), q_ref)
    wg = w.cpu().numpy().astype(np.float64)
    assert np.array_equal(wg, w_ref)   # (q - 7) * s is exact in fp32


def test_unpack_every_code_value():
    # every code 0..15 at every nibble position, and extreme scales
    K = 128
    q = np.tile(np.arange(16, dtype=np.uint8), (16, K // 16))
    for r in range(16):
        q[r] = np.roll(q[r], r)
    W = oracle.pack(q)
    s = np.array([[0x0001, 0x7BFF, 0x3C00, 0x8400]] * 16, np.uint16)  # min subnormal, max, 1, -min normal
    q_ref, w_ref = oracle.unpack(W, s, K)
    Wd, sd = dev(W, np.int32), dev(s, np.int16)
    qo = torch.empty((16, K), dtype=torch.uint8, device="cuda")
    wo = torch.empty((16, K), dtype=torch.float32, device="cuda")
    wq4.wq4_unpack_debug(Wd, sd, wo, qo, 16, K)
    torch.cuda.synchronize()
    assert np.array_equal(qo.cpu().numpy(), q_ref)
    assert np.array_equal(wo.cpu().numpy().astype(np.float64), w_ref)


# -------------------------------------------------------------------- GEMV --

def test_config1_full():
    """2048 x 2048, batch 1, seed 0: every element."""
    N = K = 2048
    W, s = synth.matrix(0, N, K)
    x = synth.activations(0, 1, K)
    check(run_gemv(W, s, x, N, K, 1), W, s, x)


@pytest.mark.parametrize("N,K", [(5120, 3072), (3072, 3072), (16384, 3072), (3072, 8192)])
def test_config2_layer_shapes_full_batch1(N, K):
    W, s = synth.matrix(2, N, K, layer=0, mat=N % 7)
    x = synth.activations(2, 1, K)
    check(run_gemv(W, s, x, N, K, 1), W, s, x)


@pytest.mark.parametrize("batch", [2, 3, 4, 8, 16, 32])
@pytest.mark.parametrize("N,K", [(5120, 3072), (3072, 8192)])
def test_config2_shapes_batches_sampled_rows(N, K, batch):
    W, s = synth.matrix(3, N, K)
    x = synth.activations(3 + batch, batch, K)
    y = run_gemv(W, s, x, N, K, batch)
    rng = np.random.default_rng(N + batch)
    rows = np.unique(np.concatenate([[0, 1, N - 1], rng.integers(0, N, 61)]))
    check(y, W[rows], s[rows], x, rows=rows)


@pytest.mark.parametrize("N,K,batch", [
    (1, 256, 1), (7, 256, 1), (1, 32, 1), (5, 32, 3), (33, 96, 2), (151, 288, 4),
    (153, 512, 1), (2, 14336, 4), (3, 14336, 1), (300, 2048, 5), (97, 4096, 32),
    (1000, 256, 17),
])
def test_edge_shapes_full(N, K, batch):
    W, s = synth.matrix(N * 3 + K, N, K)
    x = synth.activations(N + K + batch, batch, K)
    check(run_gemv(W, s, x, N, K, batch), W, s, x)


@pytest.mark.parametrize("N,K,batch", [
    (1, 256, 1), (2, 256, 2), (3, 512, 1), (151, 256, 2), (152, 768, 1), (153, 1024, 2), (303, 2048, 1),
    (304, 2048, 2), (305, 3072, 1), (999, 14336, 1), (2047, 8192, 2), (4097, 256, 1),
])
def test_mma_path_shapes_full(N, K, batch):
    """Batch 1-2 with K % 256 == 0 on the legacy-tensor-path kernel (forced
    by the test hook; the size rule would take it only from 12 Mi weights):
    odd row counts (a last word of one row), fewer words than SMs, CTA
    boundaries, one 256-code unit per row, the longest rows, every element."""
    W, s = synth.matrix(N + 7 * K, N, K)
    x = synth.activations(N + K + 3 * batch, batch, K)
    try:
        wq4.wq4_test_gemv_path(1)
        y = run_gemv(W, s, x, N, K, batch)
    finally:
        wq4.wq4_test_gemv_path(0)
    check(y, W, s, x)


@pytest.mark.parametrize("path", [1, 2])
def test_config1_both_batch1_kernels(path):
    """Config 1 on each batch 1 kernel; the two agree within the tolerance."""
    N = K = 2048
    W, s = synth.matrix(0, N, K)
    x = synth.activations(0, 1, K)
    try:
        wq4.wq4_test_gemv_path(path)
        y = run_gemv(W, s, x, N, K, 1)
    finally:
        wq4.wq4_test_gemv_path(0)
    check(y, W, s, x)


def test_unaligned_scales_take_generic_path():
    N, K = 64, 1024
    W, s = synth.matrix(8, N, K)
    x = synth.activations(8, 2, K)
    check(run_gemv(W, s, x, N, K, 2, s_offset_elems=1), W, s, x)


def test_degenerate_cases_exact():
    N, K = 40, 512
    # all codes 7: exactly zero whatever s and x
    W7 = oracle.pack(np.full((N, K), 7, np.uint8))
    _, s = synth.matrix(1, N, K)
    x = synth.activations(1, 1, K)
    y = run_gemv(W7, s, x, N, K, 1)
    assert np.all((y & 0x7FFF) == 0)
    # one nonzero group per row: closed form 32 * (q - 7) * 2^-6, exact in fp16
    codes = np.full((N, K), 7, np.uint8)
    for n in range(N):
        g = n % (K // 32)
        codes[n, 32 * g:32 * g + 32] = n % 16
    W1 = oracle.pack(codes)
    s1 = np.full((N, K // 32), 0x2400, np.uint16)
    x1 = np.full((1, K), 0x3C00, np.uint16)
    y = oracle.half_to_double(run_gemv(W1, s1, x1, N, K, 1))[0]
    assert np.array_equal(y, np.array([32 * ((n % 16) - 7) * 2.0 ** -6 for n in range(N)]))
    # x = 0 gives 0
    y = run_gemv(W1, s1, np.zeros((1, K), np.uint16), N, K, 1)
    assert np.all((y & 0x7FFF) == 0)


def test_deterministic_repeat():
    N, K = 4096, 4096
    W, s = synth.matrix(5, N, K)
    x = synth.activations(5, 1, K)
    a = run_gemv(W, s, x, N, K, 1)
    b = run_gemv(W, s, x, N, K, 1)
    assert np.array_equal(a, b)


def test_lm_head_full_size_sampled():
    """128256 x 3072 at batch 1 (the LM head of the 3B-shaped chain)."""
    from paper_2412_15803_gb300.model import fill_matrix
    N, K = 128256, 3072
    Wd = torch.empty((N, K // 8), dtype=torch.int32, device="cuda")
    sd = torch.empty((N, K // 32), dtype=torch.int16, device="cuda")
    fill_matrix(Wd, sd, N, K, 0, 28, synth.MAT_LM_HEAD)
    x = synth.activations(9, 1, K)
    y = torch.empty((1, N), dtype=torch.int16, device="cuda")
    wq4.wq4_gemv(Wd, sd, dev(x, np.int16), y, N, K, 1)
    torch.cuda.synchronize()
    yg = y.cpu().numpy().view(np.uint16)
    for start in (0, 60001, N - 64):
        W, s = synth.matrix(0, N, K, 28, synth.MAT_LM_HEAD, start, 64)
        check(yg[:, start:start + 64], W, s, x)


# ------------------------------------------------------- device generator --

def test_device_generator_matches_host_bit_exact():
    N, K = 1000, 3072
    Wd = torch.empty((N, K // 8), dtype=torch.int32, device="cuda")
    sd = torch.empty((N, K // 32), dtype=torch.int16, device="cuda")
    from paper_2412_15803_gb300.model import fill_matrix
    fill_matrix(Wd, sd, N, K, 77, 3, synth.MAT_DOWN)
    W, s = synth.matrix(77, N, K, 3, synth.MAT_DOWN)
    assert np.array_equal(Wd.cpu().numpy().view(np.uint32), W)
    assert np.array_equal(sd.cpu().numpy().view(np.uint16), s)
    # the symmetric draw of whole models, over an offset block of words
    Wsym = torch.empty(4096, dtype=torch.int32, device="cuda")
    wq4.wq4_synth_codes(Wsym, 2 * 777, 4096, 77, 9, symmetric=True)
    torch.cuda.synchronize()
    assert np.array_equal(Wsym.cpu().numpy().view(np.uint32), synth.codes_words(77, 9, 2 * 777, 4096, symmetric=True))
    # an offset block through the C ABI directly
    part = torch.empty(1000, dtype=torch.int16, device="cuda")
    wq4.wq4_synth_scales(part, 123457, 1000, 77, 5, 0.005, 0.02)
    torch.cuda.synchronize()
    assert np.array_equal(part.cpu().numpy().view(np.uint16), synth.scales_fp16(77, 5, 123457, 1000))
