"""Reference Llama-style decoder layer (CPU, fp64).

TEST INFRASTRUCTURE ONLY: the tests use it to check the library's composed
decoder-layer op; the product never imports it.

The paper's end-to-end evaluation tunes the kernels of a Llama-3-8B model
(Sec. 4, Table 2). The layer composed here is the standard pre-norm decoder
block of that model family, written from its definition:

  a   = RMSNorm(x) * g1                      RMSNorm(v) = v / sqrt(mean(v^2) + eps)
  q, k, v = split(a Wqkv^T)                  Wqkv = [Wq; Wk; Wv], heads of D = 128
  q, k = RoPE(q, p), RoPE(k, p)              p = token position (0 .. T-1)
  o   = causal GQA attention(q, k, v)        query head h reads KV head h / (Hq/Hkv)
  h1  = x + o Wo^T
  y   = h1 + W2 (silu(b Wg^T) * (b Wu^T)),   b = RMSNorm(h1) * g2

RoPE rotates the pair (j, j + D/2) of every head by the angle p * theta^(-2j/D)
(the rotate-half pairing). Tensors the kernels store in bf16 (a, q, k, v, o,
h1, b) are rounded to bf16 (round to nearest even) here at the same points,
with this module's own rounding; everything else is fp64.
"""
from __future__ import annotations

import numpy as np

import oracle


def bf16_round(x):
    """Round fp64 values to the nearest bf16 (ties to even); returns fp64."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def bf16_bits(x):
    """bf16 bit patterns (uint16) of fp64 values, rounded to nearest even."""
    r = bf16_round(x).astype(np.float32)
    return (r.view(np.uint32) >> 16).astype(np.uint16)


def widen(bits):
    """fp64 values of bf16 bit patterns."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def rmsnorm(x, g, eps):
    """x[..., H] / sqrt(mean(x^2) + eps) * g[H]."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def rope(x, pos, theta):
    """Rotary embedding of x[T, heads, D] at positions pos[T] (rotate-half pairing)."""
    x = np.asarray(x, dtype=np.float64)
    D = x.shape[-1]
    j = np.arange(D // 2, dtype=np.float64)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * theta ** (-2.0 * j / D)  # [T, D/2]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    lo, hi = x[..., : D // 2], x[..., D // 2:]
    return np.concatenate([lo * c - hi * s, hi * c + lo * s], axis=-1)


def decoder_layer_bf16(x, g1, Wqkv, Wo, g2, W1, W2, heads_q, heads_kv, theta=500000.0, eps=1e-5, rows=None):
    """The layer above on bf16 bit-pattern inputs; returns y[rows] (fp64), all rows by default.

    x[T, H], g1[H], Wqkv[(Hq + 2 Hkv) D, H], Wo[H, Hq D], g2[H], W1[2I, H], W2[H, I]."""
    X = widen(x)
    T, H = X.shape
    D = 128
    a = bf16_round(rmsnorm(X, widen(g1), eps))
    qkv = a @ widen(Wqkv).T
    q = qkv[:, : heads_q * D].reshape(T, heads_q, D)
    k = qkv[:, heads_q * D:(heads_q + heads_kv) * D].reshape(T, heads_kv, D)
    v = qkv[:, (heads_q + heads_kv) * D:].reshape(T, heads_kv, D)
    pos = np.arange(T)
    q = bf16_bits(rope(q, pos, theta))[None]
    k = bf16_bits(rope(k, pos, theta))[None]
    v = bf16_bits(v)[None]
    sel = np.arange(T) if rows is None else np.asarray(rows, dtype=np.int64)
    o, _ = oracle.attention_bf16(q, k, v, causal=True, qpos=sel)  # [1, n, Hq, D]
    o = bf16_round(o[0].reshape(len(sel), heads_q * D))
    h1 = bf16_round(X[sel] + o @ widen(Wo).T)
    b = bf16_bits(rmsnorm(h1, widen(g2), eps))
    return h1 + oracle.mlp_bf16(b, W1, W2)
