"""The seeded generator against SplitMix64's published outputs, and the
oracle against its stored fixtures (CPU only)."""
import os

import numpy as np

import oracle
from paper_2412_15803_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "gemv_small.txt")


def test_splitmix64_reference_outputs():
    # SplitMix64 started from state 0: its first four outputs as published
    # with the reference implementation (Vigna, splitmix64.c).
    got = [int(v) for v in synth.u64(0, 0, 4)]
    assert got == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4,
                   0x06C45D188009454F, 0xF88BB8A8724C81EC]


def test_row_blocks_consistent_with_whole():
    W, s = synth.matrix(3, 40, 256)
    W2, s2 = synth.matrix(3, 40, 256, row_start=17, nrows=9)
    assert np.array_equal(W[17:26], W2) and np.array_equal(s[17:26], s2)


def test_draw_distributions():
    W, s = synth.matrix(0, 512, 2048)
    nib = np.stack([(W >> np.uint32(4 * i)) & np.uint32(0xF) for i in range(8)], -1).ravel()
    counts = np.bincount(nib, minlength=16) / nib.size
    assert np.all(np.abs(counts - 1 / 16) < 0.002)
    sv = s.view(np.float16).astype(np.float64)
    assert sv.min() >= 0.005 - 1e-5 and sv.max() <= 0.02 + 1e-5
    assert abs(sv.mean() - 0.0125) < 2e-4
    x = synth.activations(0, 4, 8192).view(np.float16).astype(np.float64)
    assert abs(x.mean()) < 0.03 and abs(x.std() - 1.0) < 0.02


def test_symmetric_code_draw():
    # fold15 on patterns with every field value: only fields equal to 15 change, to 7
    w = np.array([0xFFFFFFFF, 0xF0F0F0F0, 0xEDCBA987, 0x76543210, 0x8F7F0FEF], np.uint32)
    assert [int(v) for v in synth.fold15(w)] == [0x77777777, 0x70707070, 0xEDCBA987, 0x76543210, 0x877707E7]
    # the draw: the full-range words with fields 15 folded; codes 0..14 with
    # P(7) = 2/16, the others 1/16, so the mean of q - 7 is 0
    full = synth.codes_words(4, 11, 0, 1 << 18)
    sym = synth.codes_words(4, 11, 0, 1 << 18, symmetric=True)
    assert np.array_equal(sym, synth.fold15(full))
    nib = np.stack([(sym >> np.uint32(4 * i)) & np.uint32(0xF) for i in range(8)], -1).ravel().astype(np.int64)
    counts = np.bincount(nib, minlength=16) / nib.size
    assert counts[15] == 0
    assert abs(counts[7] - 2 / 16) < 0.002
    assert np.all(np.abs(np.delete(counts[:15], 7) - 1 / 16) < 0.002)
    assert abs((nib - 7).mean()) < 0.01


def test_oracle_matches_stored_fixtures():
    lines = [l.split() for l in open(GOLDEN) if l.strip() and not l.startswith("#")]
    i = 0
    ncase = 0
    while i < len(lines):
        assert lines[i][0] == "case"
        seed, N, K, batch = map(int, lines[i][1:])
        stored = np.array([[int(t, 16) for t in lines[i + 1 + b]] for b in range(batch)], np.uint16)
        W, s = synth.matrix(seed, N, K)
        x = synth.activations(seed, batch, K)
        _, _, y16 = oracle.gemv(W, s, x)
        assert np.array_equal(y16, stored)
        i += 1 + batch
        ncase += 1
    assert ncase >= 2
