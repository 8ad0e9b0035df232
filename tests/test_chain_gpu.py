"""GPU parity of the persistent decode chain, stage by stage.

Each projection is compared with the oracle on the GPU's own fp16 input to
that stage (read back from the workspace trace), with the GEMV tolerance;
residual adds must be bit-exact; silu(gate) * up within one fp16 ulp of the
fp64 value; the LM head like a projection.  End-to-end logits of the small
model are compared with the oracle chain by relative L2 (information only).
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
from oracle import chain as ochain
from paper_2412_15803_gb300 import synth, wq4
from paper_2412_15803_gb300.model import SHAPE_3B, SHAPE_8B, SHAPE_PHI, DecodeModel, ModelShape

pytestmark = pytest.mark.gpu

TINY = ModelShape("tiny", 3, 256, 512, 2, 1, 128, 1001)
SMALL = ModelShape("small", 2, 1024, 2816 - 2816 % 256, 8, 2, 128, 4000)


def within(gpu16, ref, A, what):
    err = np.abs(oracle.half_to_double(gpu16) - ref)
    tol = oracle.tolerance(ref, A)
    bad = np.argwhere(~(err <= tol))
    assert bad.size == 0, f"{what}: {len(bad)} out of tolerance, first {bad[:3]}"


def run(model, x):
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    logits = torch.empty((model.batch, model.shape.vocab), dtype=torch.int16, device="cuda")
    model.decode(xd, logits)
    torch.cuda.synchronize()
    from paper_2412_15803_gb300 import wq4
    assert wq4.wq4_device_status() == 0
    return logits.cpu().numpy().view(np.uint16)


def check_norm(v_gpu, u, eps, what):
    """The re-fed input: fp16(r(u) u) with r in fp32 on the GPU, within one
    fp16 ulp of the fp64 value."""
    r = ochain.rms_factors(u, eps)
    ref = r[:, None] * oracle.half_to_double(u)
    err = np.abs(oracle.half_to_double(v_gpu) - ref)
    assert np.all(err <= oracle.ulp16_array(np.abs(ref))), what


def check_stages(model, layer, rows=None, u=None, t=None):
    """Stage-wise parity of one layer; rows: None = all, else a dict name -> row
    index array; u: the layer's raw input (None: the previous layer's output);
    t: the layer's trace, if already read back."""
    sh, eps = model.shape, model.eps
    H, F = sh.hidden, sh.ffn
    if t is None:
        t = model.trace(layer)
    if u is None:
        u = model.trace(layer - 1)["x_out"]
    check_norm(t["x_in"], u, eps, f"layer {layer} input normalisation")

    def proj(name, inp, use_r, out, N):
        r = ochain.rms_factors(inp, eps) if use_r else None
        idx = np.arange(N) if rows is None else rows[name]
        W, s = model.host_rows(layer, name, 0, N) if rows is None else _rows(model, layer, name, idx)
        y, A, _ = oracle.gemv(W, s, inp, r)
        within(out[:, idx], y, A, f"layer {layer} {name}")

    proj("qkv", np.ascontiguousarray(u), True, t["qkv"], sh.n_qkv)
    a = np.ascontiguousarray(t["qkv"][:, :H])
    proj("o", a, True, t["o"], H)
    assert np.array_equal(t["x_mid"], oracle.add_fp16(t["x_in"], t["o"]))
    proj("gate_up", t["x_mid"], True, t["gate_up"], 2 * F)
    m64, _ = oracle.silu_mul(np.ascontiguousarray(t["gate_up"][:, :F]), np.ascontiguousarray(t["gate_up"][:, F:]))
    err = np.abs(oracle.half_to_double(t["act"]) - m64)
    assert np.all(err <= oracle.ulp16_array(np.abs(m64))), f"layer {layer} act"
    proj("down", t["act"], False, t["down"], H)
    assert np.array_equal(t["x_out"], oracle.add_fp16(t["x_mid"], t["down"]))


def _rows(model, layer, name, idx):
    Ws, ss = [], []
    for i in idx:
        W, s = model.host_rows(layer, name, int(i), 1)
        Ws.append(W)
        ss.append(s)
    return np.concatenate(Ws), np.concatenate(ss)


def check_logits(model, logits, rows=None):
    sh = model.shape
    xL = model.trace(sh.num_layers - 1)["x_out"]
    check_norm(model.trace(sh.num_layers)["x_in"], xL, model.eps, "LM head input normalisation")
    xin = xL
    r = ochain.rms_factors(xL, model.eps)
    if rows is None:
        W, s = model.host_rows(sh.num_layers, "lm_head", 0, sh.vocab)
        idx = np.arange(sh.vocab)
    else:
        idx = rows
        W, s = _rows(model, sh.num_layers, "lm_head", idx)
    y, A, _ = oracle.gemv(W, s, xin, r)
    within(logits[:, idx], y, A, "lm_head")


@pytest.mark.parametrize("batch", [1, 2, 3, 4, 5, 6, 7, 8, 9, 13, 17, 32])
def test_tiny_chain_every_stage_every_element(batch):
    """Batch 1-2: the persistent kernel; 3-32: the graph of tensor-core stage
    kernels (batch padded to 16 up to 16, else to 32; 13 and 17 leave a
    partly padded group of four batch rows)."""
    model = DecodeModel(TINY, batch=batch, seed=batch)
    x = synth.activations(100 + batch, batch, TINY.hidden)
    logits = run(model, x)
    assert wq4.wq4_chain_path(model.table) == (1 if batch <= 2 else 2)
    for l in range(TINY.num_layers):
        check_stages(model, l, u=x if l == 0 else None)
    check_logits(model, logits)
    # end to end against the oracle chain (information: fp16 stage roundings may differ)
    layers = [{n: model.host_rows(l, n, 0, N) for n, N, _, _ in TINY.mats(l)} for l in range(TINY.num_layers)]
    lm = model.host_rows(TINY.num_layers, "lm_head", 0, TINY.vocab)
    ref16, ref, _ = ochain.token(x, layers, lm, TINY.hidden, TINY.ffn, model.eps)
    g = oracle.half_to_double(logits)
    rel = np.linalg.norm(g - ref) / np.linalg.norm(ref)
    assert rel < 2e-2, rel


@pytest.mark.parametrize("shape,batch", [(TINY, 1), (TINY, 2), (TINY, 3), (TINY, 8), (TINY, 12), (TINY, 32), (SMALL, 1),
                                         (SMALL, 4), (SMALL, 6), (SMALL, 8), (SMALL, 10)])
def test_chain_full_range_codes_every_element(shape, batch):
    """Codes uniform on 0..15 (every code value, code 15 = weight 8 s, on
    every path: the persistent kernel's exact tensor-path dequantization at
    batch 1-2, the fp16 dequantized weights of the stage graph at 3-32);
    every stage, every element, and the logits."""
    model = DecodeModel(shape, batch=batch, seed=40 + batch, symmetric=False)
    x = synth.activations(140 + batch, batch, shape.hidden)
    logits = run(model, x)
    for l in range(shape.num_layers):
        check_stages(model, l, u=x if l == 0 else None)
    check_logits(model, logits)


def test_tiny_chain_repeat_and_host_variant():
    model = DecodeModel(TINY, batch=2, seed=9)
    x = synth.activations(7, 2, TINY.hidden)
    a = run(model, x)
    tr_a = model.trace(1)
    b = run(model, x)
    assert np.array_equal(a, b)
    tr_b = model.trace(1)
    for k in tr_a:
        assert np.array_equal(tr_a[k], tr_b[k])
    lh = np.zeros((2, TINY.vocab), np.uint16)
    model.decode_host(np.ascontiguousarray(x), lh)
    assert np.array_equal(lh, a)
    # a new input after the plan exists
    x2 = synth.activations(8, 2, TINY.hidden)
    c = run(model, x2)
    assert not np.array_equal(c, a)
    for l in range(TINY.num_layers):
        check_stages(model, l, u=x2 if l == 0 else None)


def test_small_chain_ragged_items():
    """Non-power-of-two FFN and a vocab that is not a multiple of the item size."""
    model = DecodeModel(SMALL, batch=1, seed=4)
    x = synth.activations(44, 1, SMALL.hidden)
    logits = run(model, x)
    for l in range(SMALL.num_layers):
        check_stages(model, l, u=x if l == 0 else None)
    check_logits(model, logits)


def test_plan_rebuilds_when_table_changes():
    model = DecodeModel(TINY, batch=1, seed=3)
    x = synth.activations(1, 1, TINY.hidden)
    a = run(model, x)
    other = DecodeModel(TINY, batch=1, seed=12)
    # point layer 1's down projection at another model's weights
    model._layers[1].down = other._layers[1].down
    model.weights[1]["down"] = other.weights[1]["down"]
    b = run(model, x)
    assert not np.array_equal(a, b)
    t = model.trace(1)
    W, s = other.host_rows(1, "down", 0, TINY.hidden)
    y, A, _ = oracle.gemv(W, s, t["act"])
    within(t["down"], y, A, "rebuilt plan down")
    model.destroy_plan()


@pytest.mark.parametrize("batch", [1, 3, 8])
def test_3b_chain_full_size_sampled(batch):
    """The 28-layer 3B-shaped chain at batch 1 (the persistent kernel, as the
    benchmark runs it) and at batch 3 and 8 (the tensor-core stage graph):
    sampled rows of every projection of three layers, and of the LM head."""
    model = DecodeModel(SHAPE_3B, batch=batch, seed=0)
    x = synth.activations(0, batch, SHAPE_3B.hidden)
    logits = run(model, x)
    assert wq4.wq4_chain_path(model.table) == (1 if batch == 1 else 2)
    rng = np.random.default_rng(0)
    sh = SHAPE_3B

    def pick(N):
        return np.unique(np.concatenate([[0, 1, N - 2, N - 1], rng.integers(0, N, 24)]))

    for l in (0, 13, 27):
        rows = dict(qkv=pick(sh.n_qkv), o=pick(sh.hidden), gate_up=pick(2 * sh.ffn), down=pick(sh.hidden))
        check_stages(model, l, rows, u=x if l == 0 else None)
    check_logits(model, logits, rows=pick(sh.vocab))
    # the whole output is finite and the chain is deterministic
    assert np.all(np.isfinite(oracle.half_to_double(logits)))
    assert np.array_equal(run(model, x), logits)


@pytest.mark.parametrize("shape,batch", [(SHAPE_3B, 1), (SHAPE_3B, 8), (SHAPE_8B, 1)], ids=["3b-b1", "3b-b8", "8b-b1"])
def test_full_size_every_layer_every_element(shape, batch):
    """Full-size chains checked whole: the 28-layer 3B shape at batch 1 (the
    benchmarked configuration, persistent kernel) and 8 (tensor-core stage
    graph), the 32-layer 8B shape at batch 1: every output element of every
    projection of every layer (stage by stage, each on the GPU's own input to
    that stage; residual adds bit-exact) and every logit, against the oracle.
    The host side (weights regenerated from the seeded generator, the fp64
    GEMVs) runs on a thread pool: numpy and the oracle's C calls release the
    interpreter lock."""
    sh = shape
    model = DecodeModel(sh, batch=batch, seed=11 + batch)
    x = synth.activations(13 + batch, batch, sh.hidden)
    logits = run(model, x)
    assert wq4.wq4_chain_path(model.table) == (1 if batch <= 2 else 2)
    traces = [model.trace(l) for l in range(sh.num_layers + 1)]   # every device read before the threads
    xL = traces[sh.num_layers - 1]["x_out"]
    check_norm(traces[sh.num_layers]["x_in"], xL, model.eps, "LM head input normalisation")
    r = ochain.rms_factors(xL, model.eps)
    oracle.lib()

    def layer(l):
        check_stages(model, l, u=x if l == 0 else traces[l - 1]["x_out"], t=traces[l])

    def lm_block(r0):
        n = min(8192, sh.vocab - r0)
        W, s = model.host_rows(sh.num_layers, "lm_head", r0, n)
        y, A, _ = oracle.gemv(W, s, xL, r)
        within(logits[:, r0:r0 + n], y, A, f"lm_head rows {r0}..{r0 + n - 1}")

    with ThreadPoolExecutor(max_workers=max(1, min(16, os.cpu_count() or 1))) as ex:
        jobs = [ex.submit(layer, l) for l in range(sh.num_layers)]
        jobs += [ex.submit(lm_block, r0) for r0 in range(0, sh.vocab, 8192)]
        for j in jobs:
            j.result()


@pytest.mark.parametrize("batch", [1, 2, 4, 5, 8, 16, 32])
def test_8b_chain_full_size_sampled(batch):
    """The 32-layer 8B-shaped chain over the batch sweep: batch 1-2 on the
    persistent kernel (the longest rows, K = 14336 in the down projection,
    one row pair per item), 4-32 on the tensor-core stage graph (batch 5: a
    partly padded group of four batch rows; batch 17-32: 32-column tiles and
    8-part K splits at K = 14336).  Sampled rows of three layers and of the
    LM head, and twenty tokens with identical bits."""
    sh = SHAPE_8B
    model = DecodeModel(sh, batch=batch, seed=3)
    x = synth.activations(5, batch, sh.hidden)
    logits = run(model, x)
    assert wq4.wq4_chain_path(model.table) == (1 if batch <= 2 else 2)
    rng = np.random.default_rng(1)

    def pick(N):
        return np.unique(np.concatenate([[0, 1, N - 2, N - 1], rng.integers(0, N, 16)]))

    for l in (0, 17, 31):
        rows = dict(qkv=pick(sh.n_qkv), o=pick(sh.hidden), gate_up=pick(2 * sh.ffn), down=pick(sh.hidden))
        check_stages(model, l, rows, u=x if l == 0 else None)
    check_logits(model, logits, rows=pick(sh.vocab))
    for _ in range(20):
        assert np.array_equal(run(model, x), logits)


@pytest.mark.parametrize("batch", [1, 8])
def test_phi_chain_full_size_sampled(batch):
    """The Phi-3.5-mini-shaped chain (32 layers, 32 + 32 heads of 96, QKV
    9216 x 3072, vocabulary 32064: the LM head's last 128-row tile is
    partial) on the persistent kernel (batch 1) and the tensor-core graph
    (batch 8): sampled rows of three layers and of the LM head."""
    sh = SHAPE_PHI
    model = DecodeModel(sh, batch=batch, seed=7)
    x = synth.activations(9, batch, sh.hidden)
    logits = run(model, x)
    rng = np.random.default_rng(2)

    def pick(N):
        return np.unique(np.concatenate([[0, 1, N - 2, N - 1], rng.integers(0, N, 16)]))

    for l in (0, 15, 31):
        rows = dict(qkv=pick(sh.n_qkv), o=pick(sh.hidden), gate_up=pick(2 * sh.ffn), down=pick(sh.hidden))
        check_stages(model, l, rows, u=x if l == 0 else None)
    check_logits(model, logits, rows=pick(sh.vocab))
    assert np.all(np.isfinite(oracle.half_to_double(logits)))
    assert np.array_equal(run(model, x), logits)


def test_two_models_with_different_rings_alternate():
    """Plans of different shapes (different shared-memory rings) stay valid
    whichever plan was built last."""
    a = DecodeModel(TINY, batch=1, seed=41)
    b = DecodeModel(SMALL, batch=1, seed=42)
    xa = synth.activations(71, 1, TINY.hidden)
    xb = synth.activations(72, 1, SMALL.hidden)
    la = run(a, xa)
    lb = run(b, xb)
    assert np.array_equal(run(a, xa), la)
    assert np.array_equal(run(b, xb), lb)
    check_logits(a, la)


@pytest.mark.parametrize("batch", [6, 12, 16])
def test_small_chain_repeat_and_rebuild(batch):
    """The stage graph: repeated tokens, the host-buffer call and a rebuilt
    plan (a new graph) give the same bits."""
    model = DecodeModel(SMALL, batch=batch, seed=60 + batch)
    x = synth.activations(61, batch, SMALL.hidden)
    a = run(model, x)
    assert np.array_equal(run(model, x), a)          # repeated tokens are deterministic
    for l in range(SMALL.num_layers):
        check_stages(model, l, u=x if l == 0 else None)
    check_logits(model, a)
    lh = np.zeros((batch, SMALL.vocab), np.uint16)
    model.decode_host(np.ascontiguousarray(x), lh)
    assert np.array_equal(lh, a)
    model.destroy_plan()
    assert np.array_equal(run(model, x), a)          # a new plan gives the same bits


@pytest.mark.parametrize("batch", [1, 2, 3, 5, 12])
def test_cached_plan_on_a_zeroed_workspace(batch):
    """A table whose workspace was freed and came back zero-filled at the same
    address (same table contents, so the cached plan is reused without
    re-initialisation) decodes the same token again: the batch 1-2 kernel
    takes its weight pointers from the launch, not from the workspace."""
    model = DecodeModel(TINY, batch=batch, seed=90 + batch)
    x = synth.activations(91, batch, TINY.hidden)
    first = run(model, x)
    model.workspace.zero_()
    torch.cuda.synchronize()
    assert np.array_equal(run(model, x), first)
