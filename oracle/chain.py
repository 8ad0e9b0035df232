"""Oracle of one decoded token through the projection chain.

TEST INFRASTRUCTURE ONLY (see the package docstring).

The paper's workload is token decoding of 4-bit quantized transformer models
(Section 3, Table 1); the weight stream of every projection of every layer is
read once per token.  Without an attention description (``attn=None``) the
query block of the fused QKV output stands in for the attention output;
with one, each layer runs the decode step's attention (PagedAttention /
FlashAttention, Section 2.3) on rotary-embedded queries and keys:

    q, k = rope(qkv[:, :H]), rope(qkv[:, H:H + Hkv D])    fp16, see oracle.rope
    v    = qkv[:, H + Hkv D:]
    the cache of the layer gets k, v at positions[b]     (oracle.kv_append)
    a    = fp16( attention(q, cache, positions + 1) )    (oracle.paged_attention)

Layer l takes u (fp16 [batch][H]: the token input for l = 0, else the previous
layer's output) and re-feeds it after RMS normalisation; every stage output
is rounded to fp16:

    v   = fp16( r(u) * u )                       the normalised layer input
    qkv = fp16( r(u)   * W_qkv  . u  )          [batch][Nqkv]
    a   = qkv[:, :H]                             (stands in for attention)
    o   = fp16( r(a)   * W_o    . a  )          [batch][H]
    x1  = fp16( v + o )
    gu  = fp16( r(x1)  * W_gu   . x1 )          [batch][2F]  (gate | up)
    m   = fp16( silu(gu[:, :F]) * gu[:, F:] )   [batch][F]
    d   = fp16(          W_down . m  )          [batch][H]
    x2  = fp16( x1 + d )                         layer output

and after the last layer: logits = fp16( r(xL) * W_lm . xL ).

r(v) = 1 / sqrt(mean(v^2) + eps) is RMS normalisation without a learned gain.
Before every projection it is applied as a per-row factor of the projection
(r(v) W.v = W.(r(v) v) in real arithmetic), so the projection's input is the
fp16 vector itself; the normalised vector v is rounded to fp16 only where it
is kept, in the residual stream (x1 = v + o).

Each step calls the primitives of ``oracle`` and nothing else.
"""
from __future__ import annotations

import numpy as np

from . import add_fp16, gemv, kv_append, paged_attention, rms_factor, rms_normalize, rope, silu_mul


def rms_factors(v, eps):
    v = np.atleast_2d(v)
    return np.array([rms_factor(row, eps) for row in v])


def attention_step(qkv, H: int, attn: dict, t: dict):
    """The decode step's attention of one layer (see the module docstring).

    attn: n_q_heads, n_kv_heads, head_dim, theta, scale, positions (int32
    [batch]), and this layer's k_cache, v_cache (modified in place) and
    page_table.  Returns a (fp16 bits [batch][H]) and records the steps in t."""
    D, Hkv, nq = attn["head_dim"], attn["n_kv_heads"], attn["n_q_heads"]
    pos = np.asarray(attn["positions"], np.int32)
    q64, q = rope(np.ascontiguousarray(qkv[:, :H]), pos, D, attn["theta"])
    k64, k = rope(np.ascontiguousarray(qkv[:, H:H + Hkv * D]), pos, D, attn["theta"])
    v = np.ascontiguousarray(qkv[:, H + Hkv * D:H + 2 * Hkv * D])
    kv_append(k, v, attn["k_cache"], attn["v_cache"], attn["page_table"], pos)
    o, A, o16 = paged_attention(q, attn["k_cache"], attn["v_cache"], attn["page_table"], pos + 1,
                                attn["scale"], nq)
    a = o16.reshape(qkv.shape[0], H)
    t.update(q_rot=q, q_rot_ref=q64, k_rot=k, k_rot_ref=k64, v_new=v, attn=a, attn_ref=o.reshape(a.shape),
             attn_A=A.reshape(a.shape))
    return a


def layer(u, w, H: int, F: int, eps: float, attn: dict | None = None):
    """One layer.  w = dict(qkv=(W, s), o=..., gate_up=..., down=...); attn as
    attention_step's, or None for the stand-in.

    Returns (x2, trace) where trace holds every stage's fp16 output and the
    fp64 values with their magnitudes A for the projections."""
    t = {"u": u}
    r1 = rms_factors(u, eps)
    v = rms_normalize(u, eps)
    t["v"] = v
    y, A, qkv = gemv(*w["qkv"], u, r1)
    t.update(r_u=r1, qkv=qkv, qkv_ref=y, qkv_A=A)
    if attn is None:
        a = np.ascontiguousarray(qkv[:, :H])
    else:
        a = attention_step(qkv, H, attn, t)
    r2 = rms_factors(a, eps)
    y, A, o = gemv(*w["o"], a, r2)
    t.update(r_a=r2, o=o, o_ref=y, o_A=A)
    x1 = add_fp16(v, o)
    t["x1"] = x1
    r3 = rms_factors(x1, eps)
    y, A, gu = gemv(*w["gate_up"], x1, r3)
    t.update(r_x1=r3, gu=gu, gu_ref=y, gu_A=A)
    m64, m = silu_mul(np.ascontiguousarray(gu[:, :F]), np.ascontiguousarray(gu[:, F:]))
    t.update(m=m, m_ref=m64)
    y, A, d = gemv(*w["down"], m)
    t.update(d=d, d_ref=y, d_A=A)
    x2 = add_fp16(x1, d)
    t["x2"] = x2
    return x2, t


def token(x, layers, lm_head, H: int, F: int, eps: float, attn: list | None = None):
    """Whole token: all layers, final RMS normalisation and LM head; attn:
    one attention_step description per layer, or None for the stand-in.

    Returns (logits fp16 bits, logits fp64, traces)."""
    traces = []
    for l, w in enumerate(layers):
        x, t = layer(x, w, H, F, eps, None if attn is None else attn[l])
        traces.append(t)
    rf = rms_factors(x, eps)
    y, A, logits = gemv(*lm_head, x, rf)
    traces.append({"u": x, "v": rms_normalize(x, eps), "logits_ref": y, "logits_A": A})
    return logits, y, traces
