"""Tensor-core (tcgen05) GEMM family on the GPU against the fp64 oracle.

Every legal schedule of a sweep must match the oracle (semantics preservation,
Sec. 2). Shapes span several 128-row tiles with ragged M, N and K tails.
Tolerance: bf16 storage with fp32 accumulation, normwise max-relative error
<= 2e-2.
"""
import itertools

import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import empty_bf16, from_dev_bf16, rel_err, to_dev, torch

pytestmark = pytest.mark.gpu
TOL = 2e-2


def sched(op, stage=0, base=None, **kv):
    ts = []
    names = {"tile_m": (rc.T_TILE_SIZE, 0), "tile_n": (rc.T_TILE_SIZE, 1), "tile_k": (rc.T_TILE_SIZE, 2),
             "stages": (rc.T_PIPELINE_STAGES, 0),
             "split_k": (rc.T_SPLIT_K, 0),
             "fuse": (rc.T_FUSE, 0), "persistent": (rc.T_PARALLEL, 0)}
    for k, v in kv.items():
        if k == "raster":
            ts.append(rc.T(rc.T_LOOP_ORDER, v[0], stage=stage, group=v[1]))
        else:
            kind, axis = names[k]
            ts.append(rc.T(kind, v, axis=axis, stage=stage))
    return op.schedule(*ts, base=base)


@pytest.mark.parametrize("M,N,K", [(300, 384, 520), (128, 256, 64), (1, 64, 8), (513, 200, 1000)])
def test_linear_schedule_sweep(M, N, K):
    X, W = inputs.linear_bf16(M, N, K, seed=21)
    ref = oracle.linear_bf16(X, W)
    op = rc.Op(rc.OP_LINEAR, m=M, n=N, k=K)
    dX, dW = to_dev(X), to_dev(W)
    n = 0
    for tn, tk, st, sk, pe in itertools.product((64, 128, 224, 256), (64, 128), (1, 2, 4), (1, 2, 4), (0, 1)):
        try:  # K = 128 per stage with deep rings exceeds shared memory at the wide N tiles
            s = sched(op, tile_n=tn, tile_k=tk, stages=st, split_k=sk, persistent=pe)
        except rc.RcError:
            continue
        dY = empty_bf16(M, N).fill_(0x7FC0)  # NaN canary
        op.run(s, [dX, dW, dY])
        op.check()
        err = rel_err(from_dev_bf16(dY), ref)
        assert err <= TOL, (tn, tk, st, sk, pe, err)
        n += 1
    assert n >= 120


@pytest.mark.parametrize("M,N,K", [(300, 384, 520), (256, 256, 64), (1, 64, 8), (513, 224, 1000)])
def test_linear_cta_pairs(M, N, K):
    # TileSize M = 256: two CTAs share each UMMA (cta_group::2), each holding
    # 128 rows of A and half of the B tile; ragged M leaves the second CTA of
    # the last pair partly or wholly past the end.
    X, W = inputs.linear_bf16(M, N, K, seed=25)
    ref = oracle.linear_bf16(X, W)
    op = rc.Op(rc.OP_LINEAR, m=M, n=N, k=K)
    dX, dW = to_dev(X), to_dev(W)
    n = 0
    for tn, tk, st, sk, pe in itertools.product((64, 128, 224, 256), (64, 128), (1, 2, 4), (1, 2), (0, 1)):
        try:
            s = sched(op, tile_m=256, tile_n=tn, tile_k=tk, stages=st, split_k=sk, persistent=pe)
        except rc.RcError:
            continue
        dY = empty_bf16(M, N).fill_(0x7FC0)
        op.run(s, [dX, dW, dY])
        op.check()
        err = rel_err(from_dev_bf16(dY), ref)
        assert err <= TOL, (tn, tk, st, sk, pe, err)
        n += 1
    assert n >= 40


def test_linear_raster_orders():
    M, N, K = 640, 1024, 256
    X, W = inputs.linear_bf16(M, N, K, seed=22)
    ref = oracle.linear_bf16(X, W)
    op = rc.Op(rc.OP_LINEAR, m=M, n=N, k=K)
    dX, dW = to_dev(X), to_dev(W)
    for raster, pe in itertools.product([(0, 1), (1, 1), (0, 8), (1, 8)], (0, 1)):
        dY = empty_bf16(M, N).fill_(0x7FC0)
        op.run(sched(op, tile_n=128, stages=3, raster=raster, persistent=pe), [dX, dW, dY])
        op.check()
        assert rel_err(from_dev_bf16(dY), ref) <= TOL, raster


@pytest.mark.parametrize("M,I,K", [(200, 200, 256), (130, 64, 136)])
def test_swiglu_fused_and_unfused(M, I, K):
    X, W1, _ = inputs.mlp(M, K, I, seed=23)
    ref = oracle.swiglu_bf16(X, W1)
    op = rc.Op(rc.OP_SWIGLU, m=M, n=I, k=K)
    dX, dW = to_dev(X), to_dev(W1)
    for tn, st, fuse, pe, tm in itertools.product((32, 64, 128), (1, 3), (0, 1), (0, 1), (128, 256)):
        try:  # a CTA pair fuses SwiGLU with the gate rows in one CTA and the up rows in the other
            s = sched(op, tile_m=tm, tile_n=tn, stages=st, fuse=fuse, persistent=pe)
        except rc.RcError:
            continue
        dh = empty_bf16(M, I).fill_(0x7FC0)
        op.run(s, [dX, dW, dh])
        op.check()
        err = rel_err(from_dev_bf16(dh), ref)
        assert err <= TOL, (tn, st, fuse, pe, tm, err)


def test_mlp_block_small():
    T, H, I = 150, 256, 384
    X, W1, W2 = inputs.mlp(T, H, I, seed=24)
    ref = oracle.mlp_bf16(X, W1, W2)
    op = rc.Op(rc.OP_MLP, m=T, n=I, k=H)
    dX, d1, d2 = to_dev(X), to_dev(W1), to_dev(W2)
    cases = [dict(), dict(s0=dict(tile_n=128, stages=4, fuse=1), s1=dict(tile_n=256, stages=3, split_k=2)),
             dict(s0=dict(tile_n=64, stages=2, fuse=0), s1=dict(tile_n=64, stages=6, split_k=4)),
             dict(s0=dict(tile_n=128, stages=4, fuse=1, persistent=1),
                  s1=dict(tile_n=256, stages=4, split_k=2, persistent=1)),
             dict(s0=dict(tile_m=256, tile_n=128, stages=3, fuse=1, tile_k=128),
                  s1=dict(tile_m=256, tile_n=224, stages=4, persistent=0)),
             dict(s0=dict(tile_m=256, tile_n=64, stages=4, fuse=1, persistent=1),
                  s1=dict(tile_m=256, tile_n=128, stages=4, split_k=2, persistent=1))]
    for c in cases:
        s = op.schedule()
        if c:
            s = sched(op, stage=0, base=s, **c["s0"])
            s = sched(op, stage=1, base=s, **c["s1"])
        dY = empty_bf16(T, H).fill_(0x7FC0)
        op.run(s, [dX, d1, d2, dY])
        op.check()
        err = rel_err(from_dev_bf16(dY), ref)
        assert err <= TOL, (c, err)


def test_mlp_host_path_matches_device_path():
    T, H, I = 64, 128, 128
    X, W1, W2 = inputs.mlp(T, H, I, seed=25)
    op = rc.Op(rc.OP_MLP, m=T, n=I, k=H)
    s = op.schedule(rc.T(rc.T_FUSE, 1, stage=0))
    Yh = np.zeros((T, H), np.uint16)
    op.run_host(s, [X, W1, W2, Yh])
    dY = empty_bf16(T, H)
    op.run(s, [to_dev(X), to_dev(W1), to_dev(W2), dY])
    op.check()
    np.testing.assert_array_equal(Yh, dY.cpu().numpy().view(np.uint16))
    assert rel_err(inputs.bf16_bits_to_f64(Yh), oracle.mlp_bf16(X, W1, W2)) <= TOL


@pytest.mark.parametrize("M,N,K", [(1000, 512, 520), (2048, 256, 1024), (130, 128, 64)])
def test_linear_b_multicast_clusters(M, N, K):
    # TileSize M = 512: four CTAs along M share each B tile through TMA multicast; a ragged last
    # cluster reads zero rows past M and stores nothing there
    X, W = inputs.linear_bf16(M, N, K, seed=26)
    ref = oracle.linear_bf16(X, W)
    op = rc.Op(rc.OP_LINEAR, m=M, n=N, k=K)
    dX, dW = to_dev(X), to_dev(W)
    n = 0
    for tn, st, tk, split in itertools.product((64, 128, 256), (1, 2, 4), (64, 128), (1, 2)):
        try:
            s = sched(op, tile_m=512, tile_n=tn, stages=st, tile_k=tk, split_k=split)
        except rc.RcError:
            continue
        dY = empty_bf16(M, N).fill_(0x7FC0)
        op.run(s, [dX, dW, dY])
        op.check()
        assert rel_err(from_dev_bf16(dY), ref) <= TOL, str(s)
        n += 1
    assert n >= 20

