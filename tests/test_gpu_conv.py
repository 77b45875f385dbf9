"""Implicit-GEMM NHWC conv2d (+ bias + SiLU) on the GPU against the fp64 oracle.

The A operand is a 4-D TMA view of the input whose out-of-range coordinates
read as zero (the padding); every schedule in the sweep must match the oracle
(Sec. 2: transformations preserve semantics). Tolerance 2e-2 normwise
(bf16 storage, fp32 accumulation).
"""
import itertools

import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import empty_bf16, from_dev_bf16, rel_err, to_dev, torch

pytestmark = pytest.mark.gpu
TOL = 2e-2


def conv_op(N, H, W, Cin, Cout, flags=rc.EPI_BIAS | rc.EPI_SILU):
    return rc.Op(rc.OP_CONV2D, img_n=N, img_h=H, img_w=W, c_in=Cin, c_out=Cout, kr=3, ks=3, stride=1, pad=1,
                 flags=flags)


def sched(op, tile_n, stages, split_k=1, fuse=1, persistent=0, layout=0, tile_k=64, tile_m=128):
    return op.schedule(rc.T(rc.T_TILE_SIZE, tile_n, axis=1), rc.T(rc.T_PIPELINE_STAGES, stages),
                       rc.T(rc.T_SPLIT_K, split_k), rc.T(rc.T_FUSE, fuse), rc.T(rc.T_PARALLEL, persistent),
                       rc.T(rc.T_LAYOUT, layout), rc.T(rc.T_TILE_SIZE, tile_k, axis=2),
                       rc.T(rc.T_TILE_SIZE, tile_m, axis=0))


@pytest.mark.parametrize("N,H,W,Cin", [(2, 16, 16, 128), (1, 16, 8, 64), (1, 4, 32, 64), (1, 2, 64, 192),
                                       (1, 1, 128, 64)])
def test_conv_geometries(N, H, W, Cin):
    Cout = 320
    x, w, b = inputs.conv2d(N, H, W, Cin, Cout, seed=31)
    ref = oracle.conv2d_nhwc_bf16(x, w, b)
    op = conv_op(N, H, W, Cin, Cout)
    dx, dw, db = to_dev(x), to_dev(w), to_dev(b)
    for tn, st, lay, tk, tm in itertools.product((64, 80, 160), (1, 2, 4), (0, 1, 2), (64, 128), (128, 256)):
        try:
            s = sched(op, tn, st, layout=lay, tile_k=tk, tile_m=tm)
        except rc.RcError:
            continue  # shared memory (K = 128, 4 stages, N = 160); CTA pairs read A as one 4-D box only
        dy = empty_bf16(N, H, W, Cout).fill_(0x7FC0)
        op.run(s, [dx, dw, db, dy])
        op.check()
        err = rel_err(from_dev_bf16(dy).reshape(-1, Cout), ref)
        assert err <= TOL, (tn, st, lay, tk, tm, err)


def test_conv_split_k_and_unfused_epilogue():
    N, H, W, Cin, Cout = 1, 8, 16, 320, 320
    x, w, b = inputs.conv2d(N, H, W, Cin, Cout, seed=32)
    ref = oracle.conv2d_nhwc_bf16(x, w, b)
    op = conv_op(N, H, W, Cin, Cout)
    dx, dw, db = to_dev(x), to_dev(w), to_dev(b)
    for sk, fuse, tn, pe, tk, tm in itertools.product((1, 3, 5), (0, 1), (80, 160), (0, 1), (64, 128), (128, 256)):
        try:
            s = sched(op, tn, 3 if tk == 64 else 2, sk, fuse, pe, tile_k=tk, tile_m=tm)
        except rc.RcError:
            continue  # illegal here (shared memory of the ring)
        dy = empty_bf16(N, H, W, Cout).fill_(0x7FC0)
        op.run(s, [dx, dw, db, dy])
        op.check()
        err = rel_err(from_dev_bf16(dy).reshape(-1, Cout), ref)
        assert err <= TOL, (sk, fuse, tn, pe, tk, tm, err)


def test_conv_without_bias_or_silu():
    N, H, W, Cin, Cout = 1, 8, 16, 64, 64
    x, w, _ = inputs.conv2d(N, H, W, Cin, Cout, seed=33)
    for flags, silu in [(0, False), (rc.EPI_SILU, True)]:
        op = conv_op(N, H, W, Cin, Cout, flags=flags)
        ref = oracle.conv2d_nhwc_bf16(x, w, None, silu=silu)
        for fuse in (0, 1):
            dy = empty_bf16(N, H, W, Cout).fill_(0x7FC0)
            op.run(sched(op, 64, 2, 1, fuse), [to_dev(x), to_dev(w), None, dy])
            op.check()
            assert rel_err(from_dev_bf16(dy).reshape(-1, Cout), ref) <= TOL, (flags, fuse)


def test_conv_full_size_sampled_pixels():
    # Diffusion-UNet-shaped conv: N=2, 64x64, Cin=Cout=320, 3x3, pad 1, bias + SiLU.
    N, H, W, C = 2, 64, 64, 320
    x, w, b = inputs.conv2d(N, H, W, C, C, seed=5)
    op = conv_op(N, H, W, C, C)
    dy = empty_bf16(N, H, W, C)
    dx, dw, db = to_dev(x), to_dev(w), to_dev(b)
    rng = np.random.default_rng(0)
    corners = [0, W - 1, (H - 1) * W, H * W - 1, H * W, 2 * H * W - 1, 63 * 64 + 5, 64 * 5]
    pix = np.unique(np.concatenate([corners, rng.integers(0, N * H * W, 120)])).astype(np.int64)
    ref = oracle.conv2d_nhwc_bf16(x, w, b, pix=pix)
    for s in [op.schedule(), sched(op, 160, 4), sched(op, 80, 3, 5, 1), sched(op, 64, 6, 3, 0),
              sched(op, 160, 3, 1, 1, 1), sched(op, 80, 4, 3, 1, 1), sched(op, 80, 3, 1, 1, 0, 1),
              sched(op, 160, 4, 3, 0, 1, 1), sched(op, 80, 4, 1, 1, 1, 2), sched(op, 160, 3, 3, 0, 0, 2),
              sched(op, 160, 3, 1, 1, 0, 0, 128, 256), sched(op, 80, 4, 3, 1, 1, 1, 64, 256)]:
        op.run(s, [dx, dw, db, dy])
        op.check()
        got = from_dev_bf16(dy).reshape(-1, C)[pix]
        assert rel_err(got, ref) <= TOL, str(s)


def test_conv_b_multicast_clusters():
    # TileSize M = 512: four CTAs along M share each B (weight) tile through TMA multicast
    N, H, W, Cin, Cout = 2, 16, 32, 128, 320
    x, w, b = inputs.conv2d(N, H, W, Cin, Cout, seed=32)
    ref = oracle.conv2d_nhwc_bf16(x, w, b)
    op = conv_op(N, H, W, Cin, Cout)
    n = 0
    for tn, st, tk, split, fuse, lay in itertools.product((64, 160), (1, 3, 4), (64, 128), (1, 3), (0, 1), (0, 1)):
        try:
            s = sched(op, tn, st, split, fuse, 0, lay, tk, 512)
        except rc.RcError:
            continue  # shared memory
        dy = empty_bf16(N, H, W, Cout).fill_(0x7FC0)
        op.run(s, [to_dev(x), to_dev(w), to_dev(b), dy])
        op.check()
        assert rel_err(from_dev_bf16(dy).reshape(-1, Cout), ref) <= TOL, str(s)
        n += 1
    assert n >= 30
    with pytest.raises(rc.RcError):  # B slices of 80 / 4 rows are not whole swizzle atoms
        sched(op, 80, 2, 1, 1, 0, 0, 64, 512)

