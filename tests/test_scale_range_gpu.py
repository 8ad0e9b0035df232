"""Extreme fp16 scales through every GPU path, against the oracle.

The format admits any fp16 scale.  wq4_gemv and the batch 1-2 chain apply
the scale in fp32 (exact for every scale); wq4_gemm and the batch 3-32 chain
round the dequantized weight (q - 7) s to fp16, exact up to |s| = 8188
(8 * 8188 = 65504, the fp16 maximum): beyond it wq4_gemm flags bit 6 of the
device status word and the chain refuses the table at plan build.  Cases:
the largest finite scale 0x7BFF (65504), 0x7000 (8192, the first that
overflows), 0x6FFF (8188, the last that does not), the smallest subnormal
0x0001 and the largest subnormal 0x03FF, with code 15 (weight 8 s) and small
activations so that every output stays finite.
"""
import numpy as np
import pytest
import torch

import oracle
from oracle import chain as ochain
from paper_2412_15803_gb300 import synth, wq4
from paper_2412_15803_gb300.model import DecodeModel, ModelShape

pytestmark = pytest.mark.gpu

IN_RANGE = np.array([0x6FFF, 0x0001, 0x03FF, 0x3C00, 0x1A00], np.uint16)
ALL = np.array([0x7BFF, 0x7000, 0x6FFF, 0x0001, 0x03FF, 0xFBFF, 0xF000], np.uint16)
# for a chain's LM head (its input has unit RMS): large enough to test the
# exponent range, small enough that the logits stay finite
CHAIN = np.array([0x57FF, 0x5000, 0x0001, 0x03FF, 0x3C00, 0x2400, 0xD7FF], np.uint16)


def dev(a, dtype):
    return torch.from_numpy(np.ascontiguousarray(a).view(dtype)).cuda()


def extreme_matrix(seed, N, K, scales):
    """Codes uniform on 0..15 with code 15 at the first position of every
    group; scales drawn from `scales`."""
    rng = np.random.default_rng(seed)
    q = rng.integers(0, 16, size=(N, K), dtype=np.uint8)
    q[:, ::32] = 15
    W = wq4.wq4_pack_host(q)
    s = scales[rng.integers(0, len(scales), size=(N, K // 32))]
    return W, np.ascontiguousarray(s)


def small_x(seed, B, K, exp):
    """fp16 activations ~ N(0, 1) * 2^exp."""
    x = synth.activations(seed, B, K)
    xd = oracle.half_to_double(x) * 2.0 ** exp
    return oracle.double_to_half(xd)


def check(y16, W, s, x, what, r=None):
    y_ref, A, _ = oracle.gemv(W, s, x, r)
    assert np.all(np.isfinite(y_ref)), "test inputs overflow the fp64 reference"
    err = np.abs(oracle.half_to_double(y16) - y_ref)
    bad = np.argwhere(~(err <= oracle.tolerance(y_ref, A)))
    assert bad.size == 0, f"{what}: {len(bad)} out of tolerance, first {bad[:3]}"


@pytest.mark.parametrize("batch", [1, 2, 4, 8, 32])
def test_gemv_any_fp16_scale(batch):
    N, K = 256, 512
    W, s = extreme_matrix(1, N, K, ALL)
    x = small_x(2, batch, K, -14)
    y = torch.empty((batch, N), dtype=torch.int16, device="cuda")
    wq4.wq4_gemv(dev(W, np.int32), dev(s, np.int16), dev(x, np.int16), y, N, K, batch)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    check(y.cpu().numpy().view(np.uint16), W, s, x, f"gemv batch {batch}")


@pytest.mark.parametrize("M", [1, 130])
def test_gemm_scales_in_fp16_range(M):
    N, K = 256, 512
    W, s = extreme_matrix(3, N, K, IN_RANGE)
    x = small_x(4, M, K, -10)
    y = torch.empty((M, N), dtype=torch.int16, device="cuda")
    wq4.wq4_gemm(dev(W, np.int32), dev(s, np.int16), dev(x, np.int16), y, N, K, M)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    check(y.cpu().numpy().view(np.uint16), W, s, x, f"gemm M {M}")


@pytest.mark.parametrize("bad", [0x7000, 0x7BFF, 0xF000])
def test_gemm_scale_beyond_fp16_range_is_flagged(bad):
    N, K, M = 128, 256, 16
    W, s = extreme_matrix(5, N, K, IN_RANGE)
    s[7, 3] = bad
    x = small_x(6, M, K, -10)
    y = torch.empty((M, N), dtype=torch.int16, device="cuda")
    wq4.wq4_gemm(dev(W, np.int32), dev(s, np.int16), dev(x, np.int16), y, N, K, M)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 64
    assert wq4.wq4_device_status() == 0   # read and cleared


TINY = ModelShape("tiny", 2, 256, 512, 2, 1, 128, 1001)


def patch_lm_head(model, scales, seed):
    """Rewrites the LM head's scales (device and host copies) from `scales`."""
    sh = model.shape
    W, s = model.host_rows(sh.num_layers, "lm_head", 0, sh.vocab)
    rng = np.random.default_rng(seed)
    s = np.ascontiguousarray(scales[rng.integers(0, len(scales), size=s.shape)])
    model.lm_head[1].copy_(torch.from_numpy(s.view(np.int16)).reshape(model.lm_head[1].shape))
    torch.cuda.synchronize()
    return W, s


@pytest.mark.parametrize("batch", [1, 2, 3, 4, 8, 12])
def test_chain_lm_head_extreme_scales(batch):
    """The LM head with scales from the smallest subnormal to 128 and codes
    uniform on 0..15, on the persistent kernel (batch 1-2) and the stage
    graph (3-32); logits against the oracle on the GPU's own LM-head input."""
    model = DecodeModel(TINY, batch=batch, seed=60 + batch, symmetric=False)
    W, s = patch_lm_head(model, CHAIN, batch)
    x = synth.activations(61, batch, TINY.hidden)
    logits = torch.empty((batch, TINY.vocab), dtype=torch.int16, device="cuda")
    model.decode(torch.from_numpy(x.view(np.int16)).cuda(), logits)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    xL = model.trace(TINY.num_layers - 1)["x_out"]
    check(logits.cpu().numpy().view(np.uint16), W, s, xL, f"LM head batch {batch}",
          ochain.rms_factors(xL, model.eps))


@pytest.mark.parametrize("bad", [0x7000, 0xFBFF])
def test_chain_batched_refuses_scale_beyond_fp16_range(bad):
    model = DecodeModel(TINY, batch=12, seed=70)
    model.weights[1]["down"][1].view(-1)[5] = int(np.int16(np.uint16(bad).view(np.int16)))
    torch.cuda.synchronize()
    x = torch.from_numpy(synth.activations(71, 12, TINY.hidden).view(np.int16)).cuda()
    logits = torch.empty((12, TINY.vocab), dtype=torch.int16, device="cuda")
    with pytest.raises(wq4.Wq4Error) as e:
        model.decode(x, logits)
    assert e.value.status == -3   # WQ4_ERR_UNSUPPORTED
    # the same table at batch 1 runs (scales applied in fp32)
    m1 = DecodeModel(TINY, batch=1, seed=70)
    m1.weights[1]["down"][1].view(-1)[5] = int(np.int16(np.uint16(bad).view(np.int16)))
    torch.cuda.synchronize()
    l1 = torch.empty((1, TINY.vocab), dtype=torch.int16, device="cuda")
    m1.decode(x[:1].contiguous(), l1)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
