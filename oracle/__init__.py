"""CPU fp64 oracle (ctypes wrapper around ``oracle.c``).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this package; the product path (the
CUDA library and its binding) never imports it and shares no code with it.

Each wrapper cites the passage of the paper or workload definition it
follows; the arithmetic lives in ``oracle.c`` as plain loop nests.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

_P = ctypes.c_void_p
_I = ctypes.c_int64


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so (gcc, -O2, OpenMP when available)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-fvisibility=hidden", _SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = ctypes.CDLL(build())
            for name, nargs in [
                ("oracle_gemm_bias_relu_f32", 8),
                ("oracle_linear_bf16", 8),
                ("oracle_swiglu_bf16", 9),
                ("oracle_mlp_bf16", 10),
                ("oracle_attention_bf16", 14),
                ("oracle_conv2d_nhwc_bf16", 16),
                ("oracle_moe_route", 10),
                ("oracle_moe_ffn_bf16", 14),
            ]:
                getattr(_lib, name).restype = None
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(_P)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def _rows(rows):
    return None if rows is None else _c(rows, np.int64)


def threads(n=0):
    """Thread count of the oracle's OpenMP loops; n > 0 sets it. Results do not depend on it."""
    lib = _load()
    lib.oracle_threads.restype = ctypes.c_int
    return int(lib.oracle_threads(ctypes.c_int(int(n))))


def gemm_bias_relu_f32(A, B, bias=None, relu=True):
    """K0: C = max(0, A B + bias) in fp64 (App. A loop nest plus bias/ReLU). A[M,K], B[K,N]."""
    A = _c(A, np.float32)
    B = _c(B, np.float32)
    M, K = A.shape
    N = B.shape[1]
    bias = None if bias is None else _c(bias, np.float32)
    C = np.empty((M, N), np.float64)
    _load().oracle_gemm_bias_relu_f32(_I(M), _I(N), _I(K), _ptr(A), _ptr(B), _ptr(bias),
                                      ctypes.c_int(int(relu)), _ptr(C))
    return C


def linear_bf16(X, W, rows=None):
    """Y = X W^T (bf16 inputs as uint16 bits, fp64 result). X[M,K], W[N,K]."""
    X = _c(X, np.uint16)
    W = _c(W, np.uint16)
    M, K = X.shape
    N = W.shape[0]
    r = _rows(rows)
    nr = M if r is None else len(r)
    Y = np.empty((nr, N), np.float64)
    _load().oracle_linear_bf16(_I(M), _I(N), _I(K), _ptr(X), _ptr(W), _ptr(r), _I(nr), _ptr(Y))
    return Y


def swiglu_bf16(X, W1, rows=None, round_h=False):
    """h = silu(X W1[:I]^T) * (X W1[I:]^T). X[M,K], W1[2I,K]."""
    X = _c(X, np.uint16)
    W1 = _c(W1, np.uint16)
    M, K = X.shape
    I = W1.shape[0] // 2
    r = _rows(rows)
    nr = M if r is None else len(r)
    h = np.empty((nr, I), np.float64)
    _load().oracle_swiglu_bf16(_I(M), _I(I), _I(K), _ptr(X), _ptr(W1), _ptr(r), _I(nr),
                               ctypes.c_int(int(round_h)), _ptr(h))
    return h


def mlp_bf16(X, W1, W2, rows=None, round_h=False):
    """SwiGLU MLP block Y = (silu(X Wg^T) * (X Wu^T)) W2^T. X[T,H], W1[2I,H], W2[H,I]."""
    X = _c(X, np.uint16)
    W1 = _c(W1, np.uint16)
    W2 = _c(W2, np.uint16)
    T, H = X.shape
    I = W1.shape[0] // 2
    r = _rows(rows)
    nr = T if r is None else len(r)
    Y = np.empty((nr, H), np.float64)
    _load().oracle_mlp_bf16(_I(T), _I(H), _I(I), _ptr(X), _ptr(W1), _ptr(W2), _ptr(r), _I(nr),
                            ctypes.c_int(int(round_h)), _ptr(Y))
    return Y


def attention_bf16(Q, K, V, causal=True, scale=None, qpos=None):
    """GQA attention. Q[B,S,Hq,D], K/V[B,S,Hkv,D] -> O[B,nq,Hq,D], LSE[B,Hq,nq] (fp64)."""
    Q = _c(Q, np.uint16)
    K = _c(K, np.uint16)
    V = _c(V, np.uint16)
    B, S, Hq, D = Q.shape
    Hkv = K.shape[2]
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    r = _rows(qpos)
    nq = S if r is None else len(r)
    O = np.empty((B, nq, Hq, D), np.float64)
    lse = np.empty((B, Hq, nq), np.float64)
    _load().oracle_attention_bf16(_I(B), _I(S), _I(Hq), _I(Hkv), _I(D), _ptr(Q), _ptr(K), _ptr(V),
                                  ctypes.c_int(int(causal)), ctypes.c_double(scale), _ptr(r), _I(nq),
                                  _ptr(O), _ptr(lse))
    return O, lse


def conv2d_nhwc_bf16(x, w, bias=None, stride=1, pad=1, silu=True, pix=None):
    """Conv2d NHWC/KRSC with zero padding, bias and SiLU. Returns y[npix, Cout] (fp64)."""
    x = _c(x, np.uint16)
    w = _c(w, np.uint16)
    N, H, W, Cin = x.shape
    Cout, R, S, _ = w.shape
    bias = None if bias is None else _c(bias, np.uint16)
    P = (H + 2 * pad - R) // stride + 1
    Qo = (W + 2 * pad - S) // stride + 1
    r = _rows(pix)
    npix = N * P * Qo if r is None else len(r)
    y = np.empty((npix, Cout), np.float64)
    _load().oracle_conv2d_nhwc_bf16(_I(N), _I(H), _I(W), _I(Cin), _I(Cout), _I(R), _I(S), _I(stride),
                                    _I(pad), _ptr(x), _ptr(w), _ptr(bias), ctypes.c_int(int(silu)),
                                    _ptr(r), _I(npix), _ptr(y))
    return y


def moe_route(logits, topk, renorm=True):
    """Top-k softmax routing (ids, weights, offsets, perm); logits uint16 (bf16) or float32."""
    fp32 = logits.dtype == np.float32
    lg = _c(logits, np.float32 if fp32 else np.uint16)
    T, E = lg.shape
    ids = np.empty((T, topk), np.int32)
    w = np.empty((T, topk), np.float64)
    offsets = np.empty(E + 1, np.int32)
    perm = np.empty(T * topk, np.int32)
    _load().oracle_moe_route(_I(T), _I(E), _I(topk), _ptr(lg), ctypes.c_int(int(fp32)),
                             ctypes.c_int(int(renorm)), _ptr(ids), _ptr(w), _ptr(offsets), _ptr(perm))
    return ids, w, offsets, perm


def moe_ffn_bf16(X, W1, W2, ids, w, tok=None, round_h=False):
    """Routed SwiGLU experts with weighted combine. X[T,H], W1[E,2I,H], W2[E,H,I]."""
    X = _c(X, np.uint16)
    W1 = _c(W1, np.uint16)
    W2 = _c(W2, np.uint16)
    ids = _c(ids, np.int32)
    w = _c(w, np.float64)
    T, H = X.shape
    E = W1.shape[0]
    I = W1.shape[1] // 2
    topk = ids.shape[1]
    r = _rows(tok)
    nt = T if r is None else len(r)
    out = np.empty((nt, H), np.float64)
    _load().oracle_moe_ffn_bf16(_I(T), _I(H), _I(E), _I(I), _I(topk), _ptr(X), _ptr(W1), _ptr(W2),
                                _ptr(ids), _ptr(w), _ptr(r), _I(nt), ctypes.c_int(int(round_h)),
                                _ptr(out))
    return out
