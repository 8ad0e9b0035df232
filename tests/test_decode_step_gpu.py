"""GPU parity of the decode step with attention (wq4_decode_step), stage by
stage, through the C ABI.

Each stage is checked against the oracle on the GPU's own input to that
stage (read back from the workspace traces and the caches):
  * the QKV projection with the GEMV tolerance;
  * the rotary embedding of q and k within one fp16 ulp of the exact rotation
    of the GPU's fp16 QKV output (oracle.rope);
  * the append: the new cache rows equal the rotated key and the value block
    bit for bit, every other row is unchanged;
  * the attention output with the attention tolerance (oracle.paged_attention
    over the cache as the step left it, positions + 1 tokens);
  * the O projection on the attention output, and the rest of the layer as in
    the chain tests; the logits against the oracle GEMV.
Batch 1-2 runs the attention inside the persistent kernel; 3-32 the graph
path (rotation/append kernel, wq4_paged_attention, the stage kernels).
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
from oracle import chain as ochain
from paper_2412_15803_gb300 import synth, wq4
from paper_2412_15803_gb300.model import SHAPE_3B, SHAPE_8B, DecodeModel, ModelShape, StepCaches

pytestmark = pytest.mark.gpu

TINY = ModelShape("tiny", 3, 256, 512, 2, 1, 128, 1001)          # two query heads on one kv head
TINY3 = ModelShape("tiny3", 2, 768, 512, 6, 2, 128, 777)          # groups of three (the 3B grouping)
SMALL = ModelShape("small", 2, 1024, 2560, 8, 2, 128, 4000)       # groups of four (the 8B grouping)


def within(gpu16, ref, A, what):
    err = np.abs(oracle.half_to_double(gpu16) - ref)
    tol = oracle.tolerance(ref, A)
    bad = np.argwhere(~(err <= tol))
    assert bad.size == 0, f"{what}: {len(bad)} out of tolerance, first {bad[:3]}"


def run_step(model, caches, x):
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    logits = torch.empty((model.batch, model.shape.vocab), dtype=torch.int16, device="cuda")
    model.decode_step(caches, xd, logits)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
    return logits.cpu().numpy().view(np.uint16)


def _rows(model, layer, name, idx):
    Ws, ss = [], []
    for i in idx:
        W, s = model.host_rows(layer, name, int(i), 1)
        Ws.append(W)
        ss.append(s)
    return np.concatenate(Ws), np.concatenate(ss)


def check_step_layer(model, caches, layer, before, rows=None, u=None, t=None, after=None):
    """Every stage of one layer of a step.  before: (k, v) host copies of the
    layer's cache pools taken before the step; t, after: the layer's trace and
    its (k, v) pools after the step, if already read back."""
    sh, eps = model.shape, model.eps
    H, F, D, Hkv = sh.hidden, sh.ffn, sh.head_dim, sh.n_kv_heads
    KD = Hkv * D
    if t is None:
        t = model.trace(layer)
    if u is None:
        u = model.trace(layer - 1)["x_out"]
    r = ochain.rms_factors(u, eps)
    ref = r[:, None] * oracle.half_to_double(u)
    assert np.all(np.abs(oracle.half_to_double(t["x_in"]) - ref) <= oracle.ulp16_array(np.abs(ref)))

    def proj(name, inp, use_r, out, N):
        rr = ochain.rms_factors(inp, eps) if use_r else None
        idx = np.arange(N) if rows is None else rows[name]
        W, s = model.host_rows(layer, name, 0, N) if rows is None else _rows(model, layer, name, idx)
        y, A, _ = oracle.gemv(W, s, inp, rr)
        within(out[:, idx], y, A, f"layer {layer} {name}")

    proj("qkv", np.ascontiguousarray(u), True, t["qkv"], sh.n_qkv)
    # rotary embedding of the GPU's own fp16 projection output
    pos = caches.positions
    for name, lo, hi in (("q_rot", 0, H), ("k_rot", H, H + KD)):
        r64, _ = oracle.rope(np.ascontiguousarray(t["qkv"][:, lo:hi]), pos, D, caches.rope_theta)
        err = np.abs(oracle.half_to_double(t[name]) - r64)
        assert np.all(err <= oracle.ulp16_array(np.abs(r64))), f"layer {layer} {name}"
    # the append: new rows bit-exact, the rest untouched
    k_after, v_after = caches.host_cache(layer) if after is None else after
    k_exp, v_exp = before[0].copy(), before[1].copy()
    P = caches.page_size
    for b in range(model.batch):
        page = caches.table_host[b, pos[b] // P]
        k_exp[page, :, pos[b] % P, :] = t["k_rot"][b].reshape(Hkv, D)
        v_exp[page, :, pos[b] % P, :] = t["qkv"][b, H + KD:H + 2 * KD].reshape(Hkv, D)
    assert np.array_equal(k_after, k_exp), f"layer {layer} key cache"
    assert np.array_equal(v_after, v_exp), f"layer {layer} value cache"
    # attention over positions + 1 tokens of the cache as the step left it
    o, A, _ = oracle.paged_attention(np.ascontiguousarray(t["q_rot"]), k_after, v_after, caches.table_host,
                                     pos + 1, caches.scale, sh.n_q_heads)
    o = o.reshape(model.batch, H)
    A = A.reshape(model.batch, H)
    err = np.abs(oracle.half_to_double(t["attn"]) - o)
    bad = np.argwhere(~(err <= oracle.attention_tolerance(o, A)))
    assert bad.size == 0, f"layer {layer} attention: {len(bad)} out of tolerance, first {bad[:3]}"
    # the rest of the layer on the attention output
    proj("o", np.ascontiguousarray(t["attn"]), True, t["o"], H)
    assert np.array_equal(t["x_mid"], oracle.add_fp16(t["x_in"], t["o"]))
    proj("gate_up", t["x_mid"], True, t["gate_up"], 2 * F)
    m64, _ = oracle.silu_mul(np.ascontiguousarray(t["gate_up"][:, :F]), np.ascontiguousarray(t["gate_up"][:, F:]))
    assert np.all(np.abs(oracle.half_to_double(t["act"]) - m64) <= oracle.ulp16_array(np.abs(m64)))
    proj("down", t["act"], False, t["down"], H)
    assert np.array_equal(t["x_out"], oracle.add_fp16(t["x_mid"], t["down"]))


def check_logits(model, logits, rows=None):
    sh = model.shape
    xL = model.trace(sh.num_layers - 1)["x_out"]
    r = ochain.rms_factors(xL, model.eps)
    idx = np.arange(sh.vocab) if rows is None else rows
    W, s = model.host_rows(sh.num_layers, "lm_head", 0, sh.vocab) if rows is None else \
        _rows(model, sh.num_layers, "lm_head", idx)
    y, A, _ = oracle.gemv(W, s, xL, r)
    within(logits[:, idx], y, A, "lm_head")


def step_and_check(shape, positions, seed, theta=10000.0, page_size=16, rows=None, layers=None):
    batch = len(positions)
    model = DecodeModel(shape, batch=batch, seed=seed, step=True)
    caches = StepCaches(shape, positions, page_size=page_size, seed=seed + 1, spare_pages=3, rope_theta=theta)
    layers = list(range(shape.num_layers)) if layers is None else list(layers)
    before = {l: caches.host_cache(l) for l in layers}
    x = synth.activations(seed + 2, batch, shape.hidden)
    logits = run_step(model, caches, x)
    for l in layers:
        check_step_layer(model, caches, l, before[l], rows=None if rows is None else rows(l),
                         u=x if l == 0 else None)
    return model, caches, x, logits


@pytest.mark.parametrize("positions", [[0], [5], [15], [16], [1000], [3, 700], [0, 0]])
def test_tiny_step_every_stage(positions):
    """Batch 1-2 (the persistent kernel): the first token (only itself to
    attend to), positions inside, at the end of and just past a page, a long
    sequence, two rows at different lengths."""
    model, caches, x, logits = step_and_check(TINY, positions, seed=10 + sum(positions))
    check_logits(model, logits)


@pytest.mark.parametrize("positions", [[0, 17, 300], [31, 32, 33, 64, 5, 1, 250, 999]])
def test_tiny_step_graph_path(positions):
    """Batch 3 and 8: the graph path's rotation/append kernel and
    wq4_paged_attention between the tensor-core stages."""
    model, caches, x, logits = step_and_check(TINY, positions, seed=20 + len(positions))
    check_logits(model, logits)


@pytest.mark.parametrize("positions", [[77], [4, 2047], [9, 400, 1500]])
def test_grouped_heads_step(positions):
    """Groups of three query heads per kv head (the 3B grouping), batch 1, 2
    and 3."""
    model, caches, x, logits = step_and_check(TINY3, positions, seed=30 + len(positions), theta=500000.0)
    check_logits(model, logits)


@pytest.mark.parametrize("positions", [[2047], [100, 900, 3000, 17]])
def test_small_step(positions):
    """Groups of four (the 8B grouping), wider layers."""
    model, caches, x, logits = step_and_check(SMALL, positions, seed=40 + len(positions), theta=500000.0)
    check_logits(model, logits)


def test_step_repeat_is_deterministic_and_host_variant_agrees():
    model = DecodeModel(TINY, batch=2, seed=50, step=True)
    caches = StepCaches(TINY, [40, 41], seed=51)
    x = synth.activations(52, 2, TINY.hidden)
    first = run_step(model, caches, x)
    again = run_step(model, caches, x)        # the same position again: the same rows rewritten
    assert np.array_equal(first, again)
    host = np.empty_like(first)
    model.decode_step_host(caches, x, host)
    assert np.array_equal(host, first)


def test_chain_and_step_on_one_table():
    """The stand-in chain and the decode step keep separate plans on the same
    table and workspace; alternating them changes neither's result."""
    model = DecodeModel(TINY, batch=1, seed=60, step=True)
    caches = StepCaches(TINY, [12], seed=61)
    x = synth.activations(62, 1, TINY.hidden)
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    lc = torch.empty((1, TINY.vocab), dtype=torch.int16, device="cuda")
    model.decode(xd, lc)
    s1 = run_step(model, caches, x)
    model.decode(xd, lc)
    c1 = lc.cpu().numpy().copy()
    s2 = run_step(model, caches, x)
    model.decode(xd, lc)
    torch.cuda.synchronize()
    assert np.array_equal(s1, s2) and np.array_equal(lc.cpu().numpy(), c1)
    assert not np.array_equal(s1, c1.view(np.uint16))


@pytest.mark.parametrize("batch", [1, 2, 4])
def test_3b_step_full_size_sampled(batch):
    """The 28-layer 3B-shaped decode step at a context of about 4096 tokens:
    sampled projection rows and the whole attention output of three layers,
    sampled logits."""
    sh = SHAPE_3B
    rng = np.random.default_rng(batch)
    positions = [4095] + list(rng.integers(1000, 4096, batch - 1))

    def pick(N):
        return np.unique(np.concatenate([[0, 1, N - 2, N - 1], rng.integers(0, N, 16)]))

    def rows(l):
        return dict(qkv=pick(sh.n_qkv), o=pick(sh.hidden), gate_up=pick(2 * sh.ffn), down=pick(sh.hidden))

    model, caches, x, logits = step_and_check(sh, positions, seed=70 + batch, theta=500000.0, rows=rows,
                                              layers=(0, 13, 27))
    check_logits(model, logits, rows=pick(sh.vocab))
    assert np.all(np.isfinite(oracle.half_to_double(logits)))


def test_3b_step_batch1_every_layer_every_element():
    """The decode step of the 3B shape at batch 1 with 4096 tokens in context
    (the token at position 4095) checked whole: every stage of every one of
    the 28 layers -- all projection outputs, the rotated q and k, the cache
    append, the whole attention output -- and every logit.  The host side
    runs on a thread pool after every device read."""
    sh = SHAPE_3B
    model = DecodeModel(sh, batch=1, seed=91, step=True)
    caches = StepCaches(sh, [4095], page_size=16, seed=92, spare_pages=3, rope_theta=500000.0)
    L = sh.num_layers
    before = [caches.host_cache(l) for l in range(L)]
    x = synth.activations(93, 1, sh.hidden)
    logits = run_step(model, caches, x)
    assert wq4.wq4_chain_path(model.table, decode_step=True) == 1
    traces = [model.trace(l) for l in range(L + 1)]
    after = [caches.host_cache(l) for l in range(L)]
    xL = traces[L - 1]["x_out"]
    r = ochain.rms_factors(xL, model.eps)
    oracle.lib()

    def layer(l):
        check_step_layer(model, caches, l, before[l], u=x if l == 0 else traces[l - 1]["x_out"], t=traces[l],
                         after=after[l])

    def lm_block(r0):
        n = min(8192, sh.vocab - r0)
        W, s = model.host_rows(L, "lm_head", r0, n)
        y, A, _ = oracle.gemv(W, s, xL, r)
        within(logits[:, r0:r0 + n], y, A, f"lm_head rows {r0}..{r0 + n - 1}")

    with ThreadPoolExecutor(max_workers=max(1, min(16, os.cpu_count() or 1))) as ex:
        jobs = [ex.submit(layer, l) for l in range(L)]
        jobs += [ex.submit(lm_block, r0) for r0 in range(0, sh.vocab, 8192)]
        for j in jobs:
            j.result()


def test_8b_step_full_size_sampled():
    sh = SHAPE_8B
    rng = np.random.default_rng(8)

    def pick(N):
        return np.unique(np.concatenate([[0, N - 1], rng.integers(0, N, 12)]))

    def rows(l):
        return dict(qkv=pick(sh.n_qkv), o=pick(sh.hidden), gate_up=pick(2 * sh.ffn), down=pick(sh.hidden))

    model, caches, x, logits = step_and_check(sh, [2999], seed=80, theta=500000.0, rows=rows, layers=(0, 31))
    check_logits(model, logits, rows=pick(sh.vocab))


@pytest.mark.parametrize("batch", [1, 3])
def test_bad_positions_are_flagged_not_written(batch):
    """A negative position (row 0) and one past the page table (row 1): no
    append for those rows (flag bit 5), the second sequence clamped to its
    page table (bit 3); a valid row still appends; the call completes and
    the next valid step is clean."""
    model = DecodeModel(TINY, batch=batch, seed=90, step=True)
    good = np.full(batch, 5, np.int32)
    caches = StepCaches(TINY, good, seed=91)
    before = [caches.host_cache(l) for l in range(TINY.num_layers)]
    P, stride = caches.page_size, caches.table_host.shape[1]
    bad = good.copy()
    bad[0] = -1
    if batch > 1:
        bad[1] = stride * P
    caches.pos_dev.copy_(torch.from_numpy(bad))
    x = synth.activations(92, batch, TINY.hidden)
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    logits = torch.empty((batch, TINY.vocab), dtype=torch.int16, device="cuda")
    model.decode_step(caches, xd, logits)
    torch.cuda.synchronize()
    flags = wq4.wq4_device_status()
    assert flags & 32
    if batch > 1:
        assert flags & 8
    allowed = {(int(caches.table_host[b, bad[b] // P]), int(bad[b] % P)) for b in range(2, batch)}
    for l in range(TINY.num_layers):
        for new, old in zip(caches.host_cache(l), before[l]):
            pages, _, rows, _ = np.nonzero(new != old)
            assert set(zip(pages.tolist(), rows.tolist())) <= allowed, l
    assert np.all(np.isfinite(oracle.half_to_double(logits.cpu().numpy().view(np.uint16))))
    caches.pos_dev.copy_(torch.from_numpy(good))
    model.decode_step(caches, xd, logits)
    torch.cuda.synchronize()
    assert wq4.wq4_device_status() == 0
