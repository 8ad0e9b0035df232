"""wq4_decode_chain_noalloc: the decode chain for callers that cannot call
cudaMalloc (a plug-in whose host framework owns all device memory, or a loop
that cannot afford cudaMalloc's implicit synchronization).  Its workspace is a
fixed device array inside the library.  Checked through the C ABI against
wq4_decode_chain, which uses a caller-allocated workspace, on two calls in a
row.  Collected last on purpose (file name), so a failure here comes after
every other test has run; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2412_15803_gb300 import synth, wq4
from paper_2412_15803_gb300.model import SHAPE_3B, DecodeModel, ModelShape

pytestmark = pytest.mark.gpu

TINY = ModelShape("tiny", 3, 256, 512, 2, 1, 128, 1001)
SMALL = ModelShape("small", 2, 1024, 2816, 8, 2, 128, 4000)


def _logits_pair(model, x):
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    ref = torch.empty((model.batch, model.shape.vocab), dtype=torch.int16, device="cuda")
    wq4.wq4_decode_chain(model.table, xd, ref)
    torch.cuda.synchronize()
    ref_np = ref.cpu().numpy().view(np.uint16)
    lm_in = model.trace(model.shape.num_layers - 1)["x_out"]   # from the allocated workspace
    outs = []
    for _ in range(2):                                       # two calls in a row
        out = torch.full((model.batch, model.shape.vocab), -1, dtype=torch.int16, device="cuda")
        wq4.wq4_decode_chain_noalloc(model.table, xd, out)
        torch.cuda.synchronize()
        outs.append(out.cpu().numpy().view(np.uint16))
    assert wq4.wq4_device_status() == 0
    return ref_np, lm_in, outs


def _within(got, ref16, model, lm_in):
    """|got - ref| within the GEMV tolerance 1e-3 * sum|w x| + ulp16(|ref|)."""
    sh = model.shape
    W, s = model.host_rows(sh.num_layers, "lm_head", 0, sh.vocab)
    from oracle import chain as ochain
    _, A, _ = oracle.gemv(W, s, lm_in, ochain.rms_factors(lm_in, model.eps))
    ref = oracle.half_to_double(ref16)
    err = np.abs(oracle.half_to_double(got) - ref)
    assert np.all(err <= oracle.tolerance(ref, A))


@pytest.mark.parametrize("shape,batch", [(TINY, 1), (TINY, 3), (TINY, 12), (SMALL, 2)])
def test_noalloc_matches_allocated_workspace(shape, batch):
    model = DecodeModel(shape, batch=batch, seed=batch + 20)
    x = synth.activations(50 + batch, batch, shape.hidden)
    ref, lm_in, outs = _logits_pair(model, x)
    for out in outs:
        _within(out, ref, model, lm_in)
        assert np.array_equal(out, ref)        # same kernel, deterministic


def test_noalloc_switching_models_and_oversize_rejection():
    a = DecodeModel(TINY, batch=1, seed=31)
    b = DecodeModel(SMALL, batch=1, seed=32)
    xa = synth.activations(61, 1, TINY.hidden)
    xb = synth.activations(62, 1, SMALL.hidden)
    ra, lma, oa = _logits_pair(a, xa)
    rb, lmb, ob = _logits_pair(b, xb)       # another table takes over the array
    ra2, _, oa2 = _logits_pair(a, xa)       # and back
    for o in oa + oa2:
        _within(o, ra, a, lma)
    for o in ob:
        _within(o, rb, b, lmb)
    # a table whose workspace would exceed the array is refused before any launch
    big = wq4.wq4_layer_table()
    layers = (wq4.wq4_layer * SHAPE_3B.num_layers)()
    for f, v in dict(num_layers=28, hidden=3072, ffn=8192, n_q_heads=24, n_kv_heads=8, head_dim=128,
                     vocab=128256, batch=4, rms_eps=1e-5).items():
        setattr(big, f, v)
    big.layers = layers
    assert wq4.wq4_chain_workspace_bytes(big) > 16 << 20
    x = torch.zeros((4, 3072), dtype=torch.int16, device="cuda")
    out = torch.zeros((4, 128256), dtype=torch.int16, device="cuda")
    rc = wq4.load().wq4_decode_chain_noalloc(ctypes.byref(big), x.data_ptr(), out.data_ptr(), None)
    assert rc == wq4.WQ4_ERR_UNSUPPORTED


def test_noalloc_3b_batch2_full_size_sampled():
    """The largest model shape the array holds at batch 2 (3B: 14.1 MiB):
    bit-identical to the allocated-workspace chain; LM head rows sampled at
    the start, middle and end of the vocabulary against the oracle."""
    sh = SHAPE_3B
    model = DecodeModel(sh, batch=2, seed=24)
    assert wq4.wq4_chain_workspace_bytes(model.table) <= 16 << 20
    x = synth.activations(52, 2, sh.hidden)
    ref, lm_in, outs = _logits_pair(model, x)
    for out in outs:
        assert np.array_equal(out, ref)
    from oracle import chain as ochain
    r = ochain.rms_factors(lm_in, model.eps)
    for r0 in (0, sh.vocab // 2 - 128, sh.vocab - 256):
        W, s = model.host_rows(sh.num_layers, "lm_head", r0, 256)
        y, A, _ = oracle.gemv(W, s, lm_in, r)
        err = np.abs(oracle.half_to_double(ref[:, r0:r0 + 256]) - y)
        assert np.all(err <= oracle.tolerance(y, A))
