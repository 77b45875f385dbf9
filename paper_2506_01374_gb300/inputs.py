"""Seeded synthetic inputs shared by the tests, the oracle runs and bench.py.

This module holds only random-number generation and storage conversion. It
contains none of the operators' arithmetic, so both the CUDA path and the CPU
oracle can consume its arrays without sharing any computation.

Generator (counter based, so any element can be drawn independently):

* ``key(seed, tensor_id)`` = splitmix64 finaliser of ``seed * 0x100000001B3 + tensor_id``.
* The n-th 64-bit draw of a stream is ``mix(key + (n + 1) * 0x9E3779B97F4A7C15)``,
  where ``mix`` is the splitmix64 output function (Steele, Lea, Flood,
  "Fast splittable pseudorandom number generators", OOPSLA 2014).
* A uniform double in [0, 1) is ``(draw >> 11) * 2**-53``.
* A normal is Box-Muller on draws ``2i`` and ``2i + 1``:
  ``sqrt(-2 ln(1 - u1)) * cos(2 pi u2)`` (cosine branch only).
* bf16 storage: float64 -> float32 (round to nearest even), then float32 ->
  bf16 by round-to-nearest-even on the bit pattern. bf16 tensors are carried
  as ``numpy.uint16`` bit patterns.

Shapes and distributions follow the five workloads: fp32 GEMM with bias and
ReLU (A, B ~ U(-1, 1), bias ~ N(0, 1)); a SwiGLU MLP block (weights
N(0, 0.02), activations N(0, 1)); causal GQA attention (Q, K, V ~ N(0, 1));
a 3x3 NHWC conv2d (weights N(0, 0.02), inputs and bias N(0, 1)); and an MoE
layer (router logits N(0, 1), activations N(0, 1), weights N(0, 0.02)).
"""
from __future__ import annotations

import concurrent.futures as _cf
import ctypes
import os
import subprocess
import threading

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 22


def _mix(z: np.ndarray) -> np.ndarray:
    z = z ^ (z >> np.uint64(30))
    z = z * _M1
    z = z ^ (z >> np.uint64(27))
    z = z * _M2
    return z ^ (z >> np.uint64(31))


def key(seed: int, tensor_id: int) -> int:
    """Stream key of tensor ``tensor_id`` under ``seed``."""
    with np.errstate(over="ignore"):
        z = np.uint64((seed * 0x100000001B3 + tensor_id) & 0xFFFFFFFFFFFFFFFF)
        return int(_mix(np.array([z], dtype=np.uint64))[0])


def _draws(k: int, start: int, n: int) -> np.ndarray:
    ctr = np.arange(start + 1, start + 1 + n, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix(np.uint64(k) + ctr * _GOLDEN)


def _unit(d: np.ndarray) -> np.ndarray:
    return (d >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def _parallel(n: int, fn) -> np.ndarray:
    """Fill an n-vector chunk by chunk; numpy releases the GIL inside each chunk."""
    out = np.empty(n, dtype=np.float64)
    starts = list(range(0, n, _CHUNK))
    if len(starts) <= 1:
        out[:] = fn(0, n)
        return out
    workers = min(len(starts), os.cpu_count() or 1)

    def job(s):
        e = min(n, s + _CHUNK)
        out[s:e] = fn(s, e - s)

    with _cf.ThreadPoolExecutor(workers) as ex:
        list(ex.map(job, starts))
    return out


def uniform(k: int, n: int, lo: float = 0.0, hi: float = 1.0) -> np.ndarray:
    """n doubles ~ U(lo, hi) from stream k (element i uses draw i)."""
    return _parallel(n, lambda s, m: lo + (hi - lo) * _unit(_draws(k, s, m)))


def normal(k: int, n: int, mean: float = 0.0, std: float = 1.0) -> np.ndarray:
    """n doubles ~ N(mean, std^2) from stream k (element i uses draws 2i, 2i+1)."""

    return _parallel(n, lambda s, m: _normal_chunk(k, s, m, mean, std))


def to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float64/float32 -> bf16 bit patterns (uint16), round to nearest even."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))) >> np.uint64(16)
    out = u.astype(np.uint16)
    nan = np.isnan(f)
    if nan.any():
        out[nan] = 0x7FC0
    return out.reshape(np.shape(x))


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    u = np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def _normal_chunk(k: int, s: int, m: int, mean: float, std: float) -> np.ndarray:
    d = _draws(k, 2 * s, 2 * m)
    u1 = _unit(d[0::2])
    u2 = _unit(d[1::2])
    return mean + std * np.sqrt(-2.0 * np.log1p(-u1)) * np.cos(2.0 * np.pi * u2)


_HERE = os.path.dirname(os.path.abspath(__file__))
_SYNTH_SRC = os.path.join(_HERE, "synth.c")
_SYNTH_LIB = os.path.join(_HERE, "libsynth.so")
_synth = None
_synth_lock = threading.Lock()


def build_synth(force: bool = False) -> str:
    """Compile synth.c (the generator's C fast path) into libsynth.so."""
    if not force and os.path.exists(_SYNTH_LIB) and os.path.getmtime(_SYNTH_LIB) >= os.path.getmtime(_SYNTH_SRC):
        return _SYNTH_LIB
    tmp = _SYNTH_LIB + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", _SYNTH_SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _SYNTH_LIB)
    return _SYNTH_LIB


def _synth_lib():
    global _synth
    with _synth_lock:
        if _synth is None:
            L = ctypes.CDLL(build_synth())
            L.synth_bf16_normal.restype = None
            L.synth_bf16_normal.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int64, ctypes.c_double,
                                            ctypes.c_double, ctypes.c_void_p]
            _synth = L
    return _synth


def _bf16_normal(seed, tid, shape, std):
    """N(0, std^2) bf16 bits of stream (seed, tid), drawn by the C fast path
    (the same definition as to_bf16_bits(normal(...)), without a float64 copy)."""
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.uint16)
    if n:
        _synth_lib().synth_bf16_normal(key(seed, tid), 0, n, 0.0, float(std), out.ctypes.data)
    return out.reshape(shape)


# ---------------------------------------------------------------- workloads --

def gemm_f32(M: int, N: int, K: int, seed: int = 0):
    """fp32 GEMM+bias+ReLU inputs: A[M,K], B[K,N] ~ U(-1,1), bias[N] ~ N(0,1)."""
    A = uniform(key(seed, 1), M * K, -1.0, 1.0).astype(np.float32).reshape(M, K)
    B = uniform(key(seed, 2), K * N, -1.0, 1.0).astype(np.float32).reshape(K, N)
    bias = normal(key(seed, 3), N).astype(np.float32)
    return A, B, bias


def linear_bf16(M: int, N: int, K: int, seed: int = 3, x_std=1.0, w_std=0.02):
    """bf16 linear inputs: X[M,K] ~ N(0,x_std), W[N,K] ~ N(0,w_std) (nn.Linear layout)."""
    X = _bf16_normal(seed, 1, (M, K), x_std)
    W = _bf16_normal(seed, 2, (N, K), w_std)
    return X, W


def mlp(T: int, H: int, I: int, seed: int = 1):
    """SwiGLU MLP inputs.

    X[T,H] ~ N(0,1); W1[2I,H] ~ N(0,0.02) holds the gate projection in rows
    0..I-1 and the up projection in rows I..2I-1; W2[H,I] ~ N(0,0.02).
    """
    X = _bf16_normal(seed, 1, (T, H), 1.0)
    W1 = _bf16_normal(seed, 2, (2 * I, H), 0.02)
    W2 = _bf16_normal(seed, 3, (H, I), 0.02)
    return X, W1, W2


def attention(B: int, S: int, Hq: int, Hkv: int, D: int, seed: int = 4):
    """Q[B,S,Hq,D], K,V[B,S,Hkv,D] ~ N(0,1) in BSHD layout, bf16 bits."""
    Q = _bf16_normal(seed, 1, (B, S, Hq, D), 1.0)
    Kt = _bf16_normal(seed, 2, (B, S, Hkv, D), 1.0)
    V = _bf16_normal(seed, 3, (B, S, Hkv, D), 1.0)
    return Q, Kt, V


def decoder_layer(T: int, H: int, Hq: int, Hkv: int, I: int, seed: int = 8, D: int = 128, x_std: float = 1.0,
                  wqkv_std: float = 0.02):
    """Llama-style decoder layer inputs, bf16 bits.

    x[T,H] ~ N(0, x_std^2); norm weights g1, g2[H] = 1 + 0.1 N(0,1);
    Wqkv[(Hq + 2 Hkv) D, H] (query, key, value rows) ~ N(0, wqkv_std^2);
    Wo[H, Hq D], W1[2I, H] (gate rows, then up rows), W2[H, I] ~ N(0, 0.02).
    """
    x = _bf16_normal(seed, 1, (T, H), x_std)
    g1 = to_bf16_bits(1.0 + 0.1 * normal(key(seed, 2), H))
    Wqkv = _bf16_normal(seed, 3, ((Hq + 2 * Hkv) * D, H), wqkv_std)
    Wo = _bf16_normal(seed, 4, (H, Hq * D), 0.02)
    g2 = to_bf16_bits(1.0 + 0.1 * normal(key(seed, 5), H))
    W1 = _bf16_normal(seed, 6, (2 * I, H), 0.02)
    W2 = _bf16_normal(seed, 7, (H, I), 0.02)
    return x, g1, Wqkv, Wo, g2, W1, W2


def conv2d(N: int, H: int, W: int, Cin: int, Cout: int, R: int = 3, S: int = 3, seed: int = 5):
    """x[N,H,W,Cin] ~ N(0,1) (NHWC), w[Cout,R,S,Cin] ~ N(0,0.02) (KRSC), bias[Cout] ~ N(0,1)."""
    x = _bf16_normal(seed, 1, (N, H, W, Cin), 1.0)
    w = _bf16_normal(seed, 2, (Cout, R, S, Cin), 0.02)
    b = _bf16_normal(seed, 3, (Cout,), 1.0)
    return x, w, b


def moe(T: int, H: int, E: int, I: int, seed: int = 6, logits_fp32: bool = False):
    """MoE layer inputs.

    logits[T,E] ~ N(0,1) (bf16 bits, or float32 when ``logits_fp32``);
    X[T,H] ~ N(0,1); W1[E,2I,H] ~ N(0,0.02) with gate rows 0..I-1 and up rows
    I..2I-1 per expert; W2[E,H,I] ~ N(0,0.02).
    """
    lg = normal(key(seed, 1), T * E).reshape(T, E)
    logits = lg.astype(np.float32) if logits_fp32 else to_bf16_bits(lg)
    X = _bf16_normal(seed, 2, (T, H), 1.0)
    W1 = _bf16_normal(seed, 3, (E, 2 * I, H), 0.02)
    W2 = _bf16_normal(seed, 4, (E, H, I), 0.02)
    return logits, X, W1, W2
