"""Pins for the CPU oracle (no GPU).

Each oracle function is checked against something other than itself: brute
force in pure Python, a library routine (numpy matmul, scipy softmax /
logsumexp / expit), a closed form, or an invariant of the operator. The cases
are chosen so that a dropped term, a wrong sign or index, or a transposed
operand in the oracle fails at least one of them.
"""
import math

import numpy as np
import pytest
from scipy.special import expit, logsumexp, softmax

import oracle
from paper_2506_01374_gb300 import inputs

bf = inputs.to_bf16_bits
wid = inputs.bf16_bits_to_f64


def rnd_bf16(rng, shape, std=1.0):
    return bf(rng.standard_normal(shape) * std)


# ----------------------------------------------------------------- generator

def test_splitmix64_published_sequence():
    # splitmix64 from state 0 (Steele et al. 2014): first three outputs.
    d = inputs._draws(0, 0, 3)
    assert [int(x) for x in d] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_bf16_fast_path_matches_numpy_definition():
    a = inputs._bf16_normal(3, 2, (300, 700), 0.02)
    b = inputs.to_bf16_bits(inputs.normal(inputs.key(3, 2), 300 * 700, 0.0, 0.02)).reshape(300, 700)
    np.testing.assert_array_equal(a, b)


def test_bf16_rne():
    x = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 0.0])
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: even mantissa wins (1.0)
    assert list(wid(bf(x))) == [1.0, 1.0, 1.0 + 2 ** -6, -2.5, 0.0]


# ------------------------------------------------------------------------ K0

def test_k0_brute_force_tiny():
    rng = np.random.default_rng(0)
    M, N, K = 3, 5, 4
    A = rng.uniform(-1, 1, (M, K)).astype(np.float32)
    B = rng.uniform(-1, 1, (K, N)).astype(np.float32)
    bias = rng.standard_normal(N).astype(np.float32)
    C = oracle.gemm_bias_relu_f32(A, B, bias)
    for i in range(M):
        for j in range(N):
            s = float(bias[j])
            for k in range(K):
                s += float(A[i, k]) * float(B[k, j])
            assert C[i, j] == pytest.approx(max(0.0, s), abs=1e-12)


def test_k0_numpy_nonsquare():
    A, B, bias = inputs.gemm_f32(37, 29, 41, seed=3)
    C = oracle.gemm_bias_relu_f32(A, B, bias)
    ref = np.maximum(A.astype(np.float64) @ B.astype(np.float64) + bias.astype(np.float64), 0.0)
    np.testing.assert_allclose(C, ref, rtol=1e-12, atol=1e-12)
    C2 = oracle.gemm_bias_relu_f32(A, B, None, relu=False)
    np.testing.assert_allclose(C2, A.astype(np.float64) @ B.astype(np.float64), rtol=1e-12, atol=1e-12)
    assert (C2 < 0).any() and (C == 0).any()


def test_k0_identity():
    _, B, bias = inputs.gemm_f32(16, 16, 16, seed=1)
    C = oracle.gemm_bias_relu_f32(np.eye(16, dtype=np.float32), B, bias)
    np.testing.assert_array_equal(C, np.maximum(B.astype(np.float64) + bias, 0.0))


def test_k0_appendix_a_moe_matmul():
    # App. A: C[b,t,j] = sum_k A[b,t,k] B[k,j], A(1,16,7168), B(7168,2048), C init 0.
    rng = np.random.default_rng(7)
    A = rng.uniform(-1, 1, (16, 7168)).astype(np.float32)
    B = rng.uniform(-1, 1, (7168, 2048)).astype(np.float32)
    C = oracle.gemm_bias_relu_f32(A, B, None, relu=False)
    np.testing.assert_allclose(C, A.astype(np.float64) @ B.astype(np.float64), rtol=1e-10, atol=1e-9)


# -------------------------------------------------------------------- linear

def test_linear_numpy_and_rows():
    X, W = inputs.linear_bf16(19, 23, 33, seed=2)
    Y = oracle.linear_bf16(X, W)
    np.testing.assert_allclose(Y, wid(X) @ wid(W).T, rtol=1e-12, atol=1e-12)
    rows = np.array([18, 0, 7])
    np.testing.assert_array_equal(oracle.linear_bf16(X, W, rows), Y[rows])


# -------------------------------------------------------------------- SwiGLU

def test_swiglu_closed_form_probes():
    # X = e_0, gate column 0 = a, up column 0 = c  =>  h = silu(a) * c.
    a = np.array([0.0, 1.0, -1.0, 2.0, -2.0])
    c = np.array([1.0, 1.0, 1.0, 3.0, 0.5])
    I, K = len(a), 8
    X = np.zeros((1, K))
    X[0, 0] = 1.0
    W1 = np.zeros((2 * I, K))
    W1[:I, 0] = a
    W1[I:, 0] = c
    h = oracle.swiglu_bf16(bf(X), bf(W1))[0]
    silu_known = [0.0, 0.7310585786300049, -0.2689414213699951, 1.7615941559557646, -0.2384058440442351]
    np.testing.assert_allclose(h, np.array(silu_known) * c, rtol=1e-14, atol=1e-15)


def test_swiglu_numpy_and_permutation():
    rng = np.random.default_rng(1)
    X = rnd_bf16(rng, (13, 24))
    W1 = rnd_bf16(rng, (2 * 10, 24), 0.3)
    h = oracle.swiglu_bf16(X, W1)
    g = wid(X) @ wid(W1[:10]).T
    u = wid(X) @ wid(W1[10:]).T
    np.testing.assert_allclose(h, g * expit(g) * u, rtol=1e-12, atol=1e-14)
    p = rng.permutation(13)
    np.testing.assert_array_equal(oracle.swiglu_bf16(X[p], W1), h[p])


def test_mlp_numpy_zero_gate_and_rounding():
    X, W1, W2 = inputs.mlp(11, 32, 20, seed=9)
    Y = oracle.mlp_bf16(X, W1, W2)
    g = wid(X) @ wid(W1[:20]).T
    u = wid(X) @ wid(W1[20:]).T
    ref = (g * expit(g) * u) @ wid(W2).T
    np.testing.assert_allclose(Y, ref, rtol=1e-12, atol=1e-15)
    Yr = oracle.mlp_bf16(X, W1, W2, round_h=True)
    hr = wid(bf(g * expit(g) * u))
    np.testing.assert_allclose(Yr, hr @ wid(W2).T, rtol=1e-12, atol=1e-15)
    W1z = W1.copy()
    W1z[:20] = 0
    assert not oracle.mlp_bf16(X, W1z, W2).any()
    rows = np.array([10, 3])
    np.testing.assert_array_equal(oracle.mlp_bf16(X, W1, W2, rows), Y[rows])


# ----------------------------------------------------------------- attention

def _np_attention(Q, K, V, causal, scale):
    Qd, Kd, Vd = wid(Q), wid(K), wid(V)
    B, S, Hq, D = Qd.shape
    Hkv = Kd.shape[2]
    O = np.zeros_like(Qd)
    L = np.zeros((B, Hq, S))
    for b in range(B):
        for h in range(Hq):
            g = h // (Hq // Hkv)
            s = Qd[b, :, h] @ Kd[b, :, g].T * scale
            if causal:
                s = np.where(np.tril(np.ones((S, S), bool)), s, -np.inf)
            O[b, :, h] = softmax(s, axis=1) @ Vd[b, :, g]
            L[b, h] = logsumexp(s, axis=1)
    return O, L


@pytest.mark.parametrize("causal", [True, False])
def test_attention_matches_matrix_softmax(causal):
    rng = np.random.default_rng(3)
    Q = rnd_bf16(rng, (2, 7, 4, 8))
    K = rnd_bf16(rng, (2, 7, 2, 8))
    V = rnd_bf16(rng, (2, 7, 2, 8))
    O, L = oracle.attention_bf16(Q, K, V, causal=causal, scale=0.37)
    Or, Lr = _np_attention(Q, K, V, causal, 0.37)
    np.testing.assert_allclose(O, Or, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(L, Lr, rtol=1e-12, atol=1e-13)
    qpos = np.array([6, 2])
    O2, L2 = oracle.attention_bf16(Q, K, V, causal=causal, scale=0.37, qpos=qpos)
    np.testing.assert_array_equal(O2, O[:, qpos])
    np.testing.assert_array_equal(L2, L[:, :, qpos])


def test_attention_single_key_returns_v():
    rng = np.random.default_rng(4)
    Q = rnd_bf16(rng, (1, 1, 4, 16))
    K = rnd_bf16(rng, (1, 1, 2, 16))
    V = rnd_bf16(rng, (1, 1, 2, 16))
    O, L = oracle.attention_bf16(Q, K, V)
    for h in range(4):
        np.testing.assert_array_equal(O[0, 0, h], wid(V)[0, 0, h // 2])
    # LSE of a single score is the score itself
    s = (wid(Q)[0, 0, 0] @ wid(K)[0, 0, 0]) / 4.0
    assert L[0, 0, 0] == pytest.approx(s, rel=1e-14)


def test_attention_equal_keys_give_prefix_mean():
    rng = np.random.default_rng(5)
    S = 9
    Q = rnd_bf16(rng, (1, S, 2, 8))
    K = np.repeat(rnd_bf16(rng, (1, 1, 1, 8)), S, axis=1)
    V = rnd_bf16(rng, (1, S, 1, 8))
    O, _ = oracle.attention_bf16(Q, K, V, causal=True)
    Vd = wid(V)[0, :, 0]
    prefix_mean = np.cumsum(Vd, axis=0) / np.arange(1, S + 1)[:, None]
    for h in range(2):
        np.testing.assert_allclose(O[0, :, h], prefix_mean, rtol=1e-12, atol=1e-13)


def test_attention_gqa_map_is_contiguous_groups():
    # Hq=4, Hkv=2: heads 0,1 read KV head 0; heads 2,3 read KV head 1.
    rng = np.random.default_rng(6)
    Q = rnd_bf16(rng, (1, 5, 4, 8))
    K = rnd_bf16(rng, (1, 5, 2, 8))
    V = np.zeros((1, 5, 2, 8))
    V[:, :, 1] = 1.0
    O, _ = oracle.attention_bf16(Q, K, bf(V))
    np.testing.assert_allclose(O[0, :, :2], 0.0, atol=0)
    np.testing.assert_allclose(O[0, :, 2:], 1.0, rtol=1e-14)


def test_attention_head_permutation_invariance():
    rng = np.random.default_rng(8)
    Q = rnd_bf16(rng, (1, 6, 4, 8))
    K = rnd_bf16(rng, (1, 6, 2, 8))
    V = rnd_bf16(rng, (1, 6, 2, 8))
    O, _ = oracle.attention_bf16(Q, K, V)
    # swap the two KV heads and the two query-head groups together
    qp = [2, 3, 0, 1]
    O2, _ = oracle.attention_bf16(Q[:, :, qp], K[:, :, ::-1], V[:, :, ::-1])
    np.testing.assert_array_equal(O2, O[:, :, qp])


def test_attention_one_hot_v_gives_probabilities():
    rng = np.random.default_rng(10)
    S = 6
    Q = rnd_bf16(rng, (1, S, 1, S))
    K = rnd_bf16(rng, (1, S, 1, S))
    V = bf(np.eye(S)[None, :, None, :])  # D = S, V_j = e_j
    O, _ = oracle.attention_bf16(Q, K, V, causal=True, scale=0.5)
    P = O[0, :, 0]
    np.testing.assert_allclose(P.sum(axis=1), 1.0, rtol=1e-14)
    assert np.all(np.triu(P, 1) == 0)


# ---------------------------------------------------------------------- conv

def _im2col_conv(x, w, b, stride, pad, act):
    xd, wd = wid(x), wid(w)
    N, H, W, C = xd.shape
    Co, R, S, _ = wd.shape
    xp = np.pad(xd, ((0, 0), (pad, pad), (pad, pad), (0, 0)))
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    cols = np.stack([xp[:, r:r + stride * P:stride, s:s + stride * Q:stride, :]
                     for r in range(R) for s in range(S)], axis=3)  # N,P,Q,RS,C
    y = cols.reshape(N * P * Q, R * S * C) @ wd.reshape(Co, R * S * C).T
    if b is not None:
        y = y + wid(b)
    return y * expit(y) if act else y


@pytest.mark.parametrize("stride,pad", [(1, 1), (2, 1), (1, 0)])
def test_conv_matches_im2col(stride, pad):
    x, w, b = inputs.conv2d(2, 7, 9, 5, 6, seed=11)
    y = oracle.conv2d_nhwc_bf16(x, w, b, stride=stride, pad=pad, silu=True)
    np.testing.assert_allclose(y, _im2col_conv(x, w, b, stride, pad, True), rtol=1e-12, atol=1e-14)
    y0 = oracle.conv2d_nhwc_bf16(x, w, None, stride=stride, pad=pad, silu=False)
    np.testing.assert_allclose(y0, _im2col_conv(x, w, None, stride, pad, False), rtol=1e-12, atol=1e-14)


def test_conv_delta_kernel_and_1x1():
    rng = np.random.default_rng(12)
    C = 6
    x = rnd_bf16(rng, (1, 5, 4, C))
    b = rnd_bf16(rng, (C,))
    w = np.zeros((C, 3, 3, C))
    w[np.arange(C), 1, 1, np.arange(C)] = 1.0
    y = oracle.conv2d_nhwc_bf16(x, bf(w), b)
    z = wid(x).reshape(-1, C) + wid(b)
    np.testing.assert_allclose(y, z * expit(z), rtol=1e-14, atol=1e-15)
    w1 = rnd_bf16(rng, (4, 1, 1, C))
    y1 = oracle.conv2d_nhwc_bf16(x, w1, None, pad=0, silu=False)
    np.testing.assert_allclose(y1, wid(x).reshape(-1, C) @ wid(w1).reshape(4, C).T, rtol=1e-13)
    pix = np.array([19, 0, 7])
    np.testing.assert_array_equal(oracle.conv2d_nhwc_bf16(x, bf(w), b, pix=pix), y[pix])


# --------------------------------------------------------------- MoE routing

@pytest.mark.parametrize("fp32", [False, True])
def test_route_brute_force_sort(fp32):
    T, E, k = 50, 16, 4
    logits, _, _, _ = inputs.moe(T, 8, E, 4, seed=13, logits_fp32=fp32)
    ids, w, offsets, perm = oracle.moe_route(logits, k)
    L = logits.astype(np.float64) if fp32 else wid(logits)
    for t in range(T):
        order = sorted(range(E), key=lambda e: (-L[t, e], e))[:k]
        assert list(ids[t]) == order
        np.testing.assert_allclose(w[t], softmax(L[t, order]), rtol=1e-13)
    _, w_raw, _, _ = oracle.moe_route(logits, k, renorm=False)
    np.testing.assert_allclose(w_raw, np.take_along_axis(softmax(L, axis=1), ids, 1), rtol=1e-13)
    counts = np.bincount(ids.ravel(), minlength=E)
    np.testing.assert_array_equal(offsets, np.concatenate([[0], np.cumsum(counts)]))
    np.testing.assert_array_equal(perm, np.argsort(ids.ravel(), kind="stable"))


def test_route_ties_prefer_lower_id():
    T, E, k = 3, 64, 8
    L = np.zeros((T, E))
    L[1, [5, 9, 40]] = 1.0  # three equal winners, the rest tie at 0
    L[2, :] = -1.0
    L[2, [63, 2]] = 0.5
    ids, w, _, _ = oracle.moe_route(bf(L), k)
    assert list(ids[0]) == list(range(8))
    np.testing.assert_allclose(w[0], 1 / 8, rtol=1e-15)
    assert list(ids[1]) == [5, 9, 40, 0, 1, 2, 3, 4]
    assert list(ids[2]) == [2, 63, 0, 1, 3, 4, 5, 6]


@pytest.mark.parametrize("fp32", [False, True])
def test_route_nan_logits_rank_last(fp32):
    # NaN has no order; the routing reads it as -inf: below every number, ties by lower id, weight 0
    E, k = 8, 4
    L = np.full((3, E), np.nan)
    L[0, [1, 3]] = [1.0, 0.5]  # two numbers, six NaNs: the numbers first, then the lowest NaN ids
    L[1, :] = np.arange(E)[::-1]  # no NaN: plain order
    L[1, 0] = np.nan  # the largest value replaced by NaN drops to the end
    L[2, [6]] = -30.0  # one number, far below zero, still ranks above every NaN
    logits = L.astype(np.float32) if fp32 else bf(L)
    ids, w, offsets, perm = oracle.moe_route(logits, k)
    assert list(ids[0]) == [1, 3, 0, 2]
    e5 = np.exp(-0.5)
    np.testing.assert_allclose(w[0], [1 / (1 + e5), e5 / (1 + e5), 0, 0], rtol=1e-15, atol=0)
    assert list(ids[1]) == [1, 2, 3, 4]
    assert list(ids[2]) == [6, 0, 1, 2]
    np.testing.assert_allclose(w[2], [1, 0, 0, 0], rtol=1e-15, atol=0)
    counts = np.bincount(ids.ravel(), minlength=E)
    np.testing.assert_array_equal(offsets, np.concatenate([[0], np.cumsum(counts)]))
    np.testing.assert_array_equal(perm, np.argsort(ids.ravel(), kind="stable"))


# ------------------------------------------------------------------- MoE FFN

def _np_expert(x, W1e, W2e):
    I = W1e.shape[0] // 2
    g = x @ W1e[:I].T
    u = x @ W1e[I:].T
    return (g * expit(g) * u) @ W2e.T


def test_moe_ffn_all_experts_dense_mixture():
    T, H, E, I = 6, 16, 4, 8
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=14)
    ids, w, _, _ = oracle.moe_route(logits, E)  # top-k = E: every expert
    out = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    P = softmax(wid(logits), axis=1)
    ref = sum(P[:, e:e + 1] * _np_expert(wid(X), wid(W1[e]), wid(W2[e])) for e in range(E))
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-14)


def test_moe_ffn_identical_experts_equal_dense_mlp():
    T, H, E, I, k = 9, 16, 5, 8, 2
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=15)
    W1s = np.repeat(W1[:1], E, axis=0)
    W2s = np.repeat(W2[:1], E, axis=0)
    ids, w, _, _ = oracle.moe_route(logits, k)
    out = oracle.moe_ffn_bf16(X, W1s, W2s, ids, w)
    np.testing.assert_allclose(out, _np_expert(wid(X), wid(W1[0]), wid(W2[0])), rtol=1e-11, atol=1e-14)


def test_moe_ffn_expert_relabel_invariance_and_tokens():
    T, H, E, I, k = 8, 16, 6, 8, 3
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=16)
    ids, w, _, _ = oracle.moe_route(logits, k)
    out = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    p = np.array([3, 0, 5, 1, 4, 2])
    # relabel: new expert j is old expert p[j]; logits columns move with them.
    # Distinct logits per row keep the selected set unchanged.
    ids2, w2, _, _ = oracle.moe_route(logits[:, p], k)
    out2 = oracle.moe_ffn_bf16(X, W1[p], W2[p], ids2, w2)
    np.testing.assert_allclose(out2, out, rtol=1e-13, atol=1e-15)
    # direct per-slot sum in k order
    ref = np.zeros((T, H))
    for t in range(T):
        for j in range(k):
            e = ids[t, j]
            ref[t] += w[t, j] * _np_expert(wid(X[t:t + 1]), wid(W1[e]), wid(W2[e]))[0]
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-15)
    tok = np.array([7, 1])
    np.testing.assert_array_equal(oracle.moe_ffn_bf16(X, W1, W2, ids, w, tok=tok), out[tok])
