"""The schedules the benchmark reports, run at the benchmark's full sizes and
checked against the fp64 oracle on sampled rows.

The paper makes every transformation semantics preserving (Sec. 2, Eq. 1), so
a schedule's speed is worth reporting only once its output matches the
oracle at the very shapes it was timed on: the Llama-3-8B-shaped MLP block on
CTA pairs, the UNet-shaped conv2d with 128-deep K stages on persistent CTAs,
and the 64-expert MoE layer with a CTA-pair gate/up GEMM and a persistent
down GEMM at different ring depths. Tolerance 2e-2 normwise (bf16 storage,
fp32 accumulation); MoE routing bit-exact.
"""
import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import empty_bf16, from_dev_bf16, rel_err, to_dev, torch

pytestmark = pytest.mark.gpu
TOL = 2e-2

_KNOB = {"tile_m": (rc.T_TILE_SIZE, 0), "tile_n": (rc.T_TILE_SIZE, 1), "tile_k": (rc.T_TILE_SIZE, 2),
         "stages": (rc.T_PIPELINE_STAGES, 0), "split_k": (rc.T_SPLIT_K, 0), "fuse": (rc.T_FUSE, 0),
         "persistent": (rc.T_PARALLEL, 0), "layout": (rc.T_LAYOUT, 0), "location": (rc.T_COMPUTE_LOCATION, 0)}


def schedule(op, **stages):
    """schedule(op, s0=dict(tile_m=256, raster=(1, 8)), s1=dict(...)) -> the transformed program."""
    ts = []
    for name, kv in stages.items():
        g = int(name[1:])
        for k, v in kv.items():
            if k == "raster":
                ts.append(rc.T(rc.T_LOOP_ORDER, v[0], stage=g, group=v[1]))
            else:
                kind, axis = _KNOB[k]
                ts.append(rc.T(kind, v, axis=axis, stage=g))
    return op.schedule(*ts)


def test_mlp_block_full_size_reported_schedules():
    # T = 2048 tokens, hidden 4096, intermediate 14336 (Llama-3-8B), SwiGLU
    T, H, I = 2048, 4096, 14336
    X, W1, W2 = inputs.mlp(T, H, I, seed=1)
    rows = np.array([0, 1, 127, 128, 255, 256, 1000, 1023, 1024, 1500, 1791, 1792, 2000, 2046, 2047, 77],
                    dtype=np.int64)
    ref = oracle.mlp_bf16(X, W1, W2, rows=rows)
    op = rc.Op(rc.OP_MLP, m=T, n=I, k=H)
    dX, d1, d2 = to_dev(X), to_dev(W1), to_dev(W2)
    del W1, W2
    cases = [
        # gate/up: CTA pair, 256 x 128 outputs (a 256 x 256 UMMA over gate and up rows), 3 stages, fused,
        # raster bands of 8; down: CTA pair 256 x 224, 3 stages
        dict(s0=dict(tile_m=256, tile_n=128, tile_k=64, stages=3, fuse=1, raster=(1, 8)),
             s1=dict(tile_m=256, tile_n=224, stages=3, raster=(1, 1))),
        dict(s0=dict(tile_m=256, tile_n=128, tile_k=64, stages=3, fuse=1, raster=(0, 1)),
             s1=dict(tile_m=256, tile_n=224, stages=3, raster=(0, 1))),
        dict(s0=dict(tile_m=128, tile_n=128, stages=2, fuse=1),
             s1=dict(tile_m=256, tile_n=224, stages=3)),
        # gate/up on persistent CTA pairs (two 256-column accumulators: all 512 TMEM columns), K 128 per stage
        dict(s0=dict(tile_m=256, tile_n=128, tile_k=128, stages=3, fuse=1, persistent=1, raster=(0, 1)),
             s1=dict(tile_m=256, tile_n=224, stages=3, raster=(0, 1))),
        # and both GEMMs persistent
        dict(s0=dict(tile_m=256, tile_n=128, tile_k=64, stages=6, fuse=1, persistent=1, raster=(0, 8)),
             s1=dict(tile_m=256, tile_n=256, tile_k=128, stages=3, persistent=1, raster=(1, 8))),
    ]
    for c in cases:
        s = schedule(op, **c)
        dY = empty_bf16(T, H).fill_(0x7FC0)
        op.run(s, [dX, d1, d2, dY])
        op.check()
        err = rel_err(from_dev_bf16(dY)[rows], ref)
        assert err <= TOL, (str(s), err)


def test_conv2d_full_size_reported_schedules():
    # N = 2, 64 x 64, Cin = Cout = 320, 3 x 3, pad 1, bias + SiLU (diffusion UNet)
    N, Hh, W, C = 2, 64, 64, 320
    x, w, b = inputs.conv2d(N, Hh, W, C, C, seed=5)
    op = rc.Op(rc.OP_CONV2D, img_n=N, img_h=Hh, img_w=W, c_in=C, c_out=C, kr=3, ks=3, stride=1, pad=1,
               flags=rc.EPI_BIAS | rc.EPI_SILU)
    rng = np.random.default_rng(1)
    corners = [0, W - 1, (Hh - 1) * W, Hh * W - 1, Hh * W, 2 * Hh * W - 1]
    pix = np.unique(np.concatenate([corners, rng.integers(0, N * Hh * W, 200)])).astype(np.int64)
    ref = oracle.conv2d_nhwc_bf16(x, w, b, pix=pix)
    dx, dw, db = to_dev(x), to_dev(w), to_dev(b)
    for c in [dict(s0=dict(tile_n=160, tile_k=128, stages=3, fuse=1, persistent=1)),
              dict(s0=dict(tile_m=512, tile_n=160, tile_k=64, stages=4, fuse=1)),
              dict(s0=dict(tile_m=512, tile_n=160, tile_k=128, stages=3, fuse=1)),
              dict(s0=dict(tile_n=160, tile_k=128, stages=3, fuse=1, persistent=0)),
              dict(s0=dict(tile_n=160, tile_k=64, stages=6, fuse=1, persistent=1))]:
        s = schedule(op, **c)
        dy = empty_bf16(N, Hh, W, C).fill_(0x7FC0)
        op.run(s, [dx, dw, db, dy])
        op.check()
        err = rel_err(from_dev_bf16(dy).reshape(-1, C)[pix], ref)
        assert err <= TOL, (str(s), err)


def test_moe_full_size_reported_schedules():
    # T = 4096 tokens, hidden 7168, 64 experts of intermediate 2048, top-8
    T, H, E, I, K = 4096, 7168, 64, 2048, 8
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=6)
    ids, w, off, perm = oracle.moe_route(logits, K)
    tok = np.unique(np.concatenate([[0, 1, 2047, 2048, 4095],
                                    np.random.default_rng(2).integers(0, T, 64)])).astype(np.int64)
    assert len(tok) >= 64
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w, tok=tok)
    op = rc.Op(rc.OP_MOE, tokens=T, hidden=H, experts=E, inter=I, top_k=K)
    dl, dX, d1, d2 = to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2)
    del W1, W2
    cases = [
        # gate/up on CTA pairs (256 x 128 outputs, 3 stages); down on persistent single CTAs 128 x 256, 4 stages
        dict(s0=dict(tile_m=8), s1=dict(tile_m=256, tile_n=128, stages=3),
             s2=dict(tile_m=128, tile_n=256, stages=4, persistent=1, raster=(0, 8))),
        dict(s0=dict(tile_m=8), s1=dict(tile_m=256, tile_n=128, stages=3),
             s2=dict(tile_m=256, tile_n=224, stages=3)),
        dict(s0=dict(tile_m=4), s1=dict(tile_m=256, tile_n=128, stages=3, raster=(1, 1)),
             s2=dict(tile_m=128, tile_n=256, stages=4, persistent=1, fuse=1)),
    ]
    for c in cases:
        s = schedule(op, **c)
        out = empty_bf16(T, H).fill_(0x7FC0)
        gi = torch.empty(T, K, dtype=torch.int32, device="cuda")
        go = torch.empty(E + 1, dtype=torch.int32, device="cuda")
        gp = torch.empty(T * K, dtype=torch.int32, device="cuda")
        op.run(s, [dl, dX, d1, d2, out, gi, None, go, gp])
        op.check()
        np.testing.assert_array_equal(gi.cpu().numpy(), ids)
        np.testing.assert_array_equal(go.cpu().numpy(), off)
        np.testing.assert_array_equal(gp.cpu().numpy(), perm)
        err = rel_err(from_dev_bf16(out)[tok], ref)
        assert err <= TOL, (str(s), err)
