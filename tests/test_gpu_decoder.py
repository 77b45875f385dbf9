"""The composed Llama-style decoder layer (RMSNorm, QKV GEMM, RoPE, causal GQA
attention, O GEMM + residual, RMSNorm, SwiGLU MLP + residual) on the GPU
against the fp64 oracle (oracle/decoder.py), to 2e-2 normwise (bf16).

The small cases scale x by 0.05 and the QKV weights up to N(0, 0.1^2): the
layer's increment (attention and MLP), not the residual copy of x, then
dominates y, and the attention weights are peaked, so a wrong RoPE angle,
head mapping or residual moves the error far above the bound (changing theta
from 10^4 to 5 10^5 alone moves y by about 12%). The full
Llama-3-8B layer is checked on sampled rows, on its increment y - x."""
import numpy as np
import pytest

from oracle import decoder
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import empty_bf16, from_dev_bf16, rel_err, to_dev

pytestmark = pytest.mark.gpu
TOL = 2e-2


def layer_op(T, H, Hq, Hkv, I):
    return rc.Op(rc.OP_DECODER_LAYER, tokens=T, hidden=H, inter=I, heads_q=Hq, heads_kv=Hkv, head_dim=128)


def run_layer(op, sched, args, T, H):
    y = empty_bf16(T, H)
    op.run(sched, [to_dev(a) for a in args] + [y])
    op.check()
    return from_dev_bf16(y)


def schedules(op):
    T = rc.T
    yield "P0", op.schedule()
    # fused SwiGLU, 4 tokens per RoPE CTA, 128-key blocks with V untransposed, deeper GEMM rings
    yield "fused", op.schedule(T(rc.T_TILE_SIZE, 128, axis=1, stage=0), T(rc.T_PIPELINE_STAGES, 4, stage=0),
                               T(rc.T_TILE_SIZE, 4, axis=0, stage=1),
                               T(rc.T_TILE_SIZE, 128, axis=1, stage=2), T(rc.T_LAYOUT, 0, stage=2),
                               T(rc.T_FUSE, 1, stage=4), T(rc.T_TILE_SIZE, 128, axis=1, stage=4),
                               T(rc.T_TILE_SIZE, 128, axis=2, stage=5), T(rc.T_PIPELINE_STAGES, 3, stage=5))
    # CTA pairs for every GEMM, persistent O projection, the one-tile split-issue attention kernel
    yield "pairs", op.schedule(T(rc.T_TILE_SIZE, 256, axis=0, stage=0), T(rc.T_PIPELINE_STAGES, 3, stage=0),
                               T(rc.T_TILE_SIZE, 8, axis=0, stage=1),
                               T(rc.T_TILE_SIZE, 64, axis=1, stage=2), T(rc.T_PIPELINE_STAGES, 2, stage=2),
                               T(rc.T_LOOP_ORDER, 1, group=1, stage=2), T(rc.T_COMPUTE_LOCATION, 1, stage=2),
                               T(rc.T_PARALLEL, 1, stage=2), T(rc.T_LAYOUT, 0, stage=2),
                               T(rc.T_TILE_SIZE, 256, axis=0, stage=3), T(rc.T_PARALLEL, 1, stage=3),
                               T(rc.T_TILE_SIZE, 256, axis=0, stage=4), T(rc.T_FUSE, 1, stage=4),
                               T(rc.T_TILE_SIZE, 256, axis=0, stage=5), T(rc.T_TILE_SIZE, 224, axis=1, stage=5))


@pytest.mark.parametrize("T,H,Hq,Hkv,I", [(200, 256, 4, 2, 384), (384, 512, 8, 2, 640), (24, 256, 2, 1, 256)])
def test_decoder_layer_parity(T, H, Hq, Hkv, I):
    args = inputs.decoder_layer(T, H, Hq, Hkv, I, seed=21, x_std=0.05, wqkv_std=0.1)
    ref = decoder.decoder_layer_bf16(*args, Hq, Hkv)
    op = layer_op(T, H, Hq, Hkv, I)
    for name, s in schedules(op):
        err = rel_err(run_layer(op, s, args, T, H), ref)
        assert err <= TOL, f"{name}: rel err {err:.3e}"


def test_decoder_layer_rope_theta_and_eps_are_used():
    T, H, Hq, Hkv, I = 128, 256, 4, 2, 256
    args = inputs.decoder_layer(T, H, Hq, Hkv, I, seed=22, x_std=0.05, wqkv_std=0.1)
    op = rc.Op(rc.OP_DECODER_LAYER, tokens=T, hidden=H, inter=I, heads_q=Hq, heads_kv=Hkv, head_dim=128,
               rope_theta=10000.0, norm_eps=1e-2)
    got = run_layer(op, op.schedule(), args, T, H)
    ref = decoder.decoder_layer_bf16(*args, Hq, Hkv, theta=10000.0, eps=1e-2)
    assert rel_err(got, ref) <= TOL
    # the default theta (500000) gives a clearly different layer at these positions
    other = decoder.decoder_layer_bf16(*args, Hq, Hkv, eps=1e-2)
    assert rel_err(other, ref) > 4 * TOL


def test_decoder_layer_profiled_stages():
    T, H, Hq, Hkv, I = 256, 512, 4, 2, 512
    args = inputs.decoder_layer(T, H, Hq, Hkv, I, seed=23)
    op = layer_op(T, H, Hq, Hkv, I)
    y = empty_bf16(T, H)
    ms = op.run_profiled(op.schedule(), [to_dev(a) for a in args] + [y])
    op.check()
    assert len(ms) == 6 and all(m > 0 for m in ms)
    np.testing.assert_array_equal(from_dev_bf16(y), run_layer(op, op.schedule(), args, T, H))


def test_decoder_layer_host_buffers():
    T, H, Hq, Hkv, I = 128, 256, 4, 2, 384
    args = inputs.decoder_layer(T, H, Hq, Hkv, I, seed=24, x_std=0.05, wqkv_std=0.1)
    op = layer_op(T, H, Hq, Hkv, I)
    y = np.empty((T, H), np.uint16)
    op.run_host(op.schedule(), list(args) + [y])
    widened = inputs.bf16_bits_to_f64(y)
    np.testing.assert_array_equal(widened, run_layer(op, op.schedule(), args, T, H))
    assert rel_err(widened, decoder.decoder_layer_bf16(*args, Hq, Hkv)) <= TOL


def test_llama3_8b_decoder_layer_sampled_rows():
    T, H, Hq, Hkv, I = 2048, 4096, 32, 8, 14336
    args = inputs.decoder_layer(T, H, Hq, Hkv, I, seed=8)
    op = layer_op(T, H, Hq, Hkv, I)
    rows = np.array([0, 1, 127, 128, 1000, 1535, 2046, 2047])
    ref = decoder.decoder_layer_bf16(*args, Hq, Hkv, rows=rows)
    x = decoder.widen(args[0][rows])
    for name, s in schedules(op):
        y = run_layer(op, s, args, T, H)[rows]
        err = rel_err(y - x, ref - x)
        assert err <= TOL, f"{name}: rel err of the increment {err:.3e}"
