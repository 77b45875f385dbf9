"""The Vectorize transformation: 4-, 8- and 16-byte accesses in the memory-bound passes
(SwiGLU pass, bias/SiLU pass, split-K reduce, MoE row gather, combine and the fp32 -> bf16
pass of the atomic combine). Every width must give the oracle's result (Sec. 2: transformations
preserve semantics); the passes round exactly as before, so the three widths agree bit for bit.
"""
import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import empty_bf16, from_dev_bf16, rel_err, to_dev, torch

pytestmark = pytest.mark.gpu
TOL = 2e-2
VECS = (4, 8, 16)


def test_linear_split_k_reduce_widths():
    M, N, K = 300, 384, 1040
    X, W = inputs.linear_bf16(M, N, K, seed=71)
    ref = oracle.linear_bf16(X, W)
    op = rc.Op(rc.OP_LINEAR, m=M, n=N, k=K)
    outs = []
    for vec in VECS:
        s = op.schedule(rc.T(rc.T_SPLIT_K, 4), rc.T(rc.T_VECTORIZE, vec))
        assert s.knobs(0)["vec"] == vec
        Y = empty_bf16(M, N).fill_(0x7FC0)
        op.run(s, [to_dev(X), to_dev(W), Y])
        op.check()
        outs.append(Y.cpu().numpy())
        assert rel_err(from_dev_bf16(Y), ref) <= TOL, vec
    assert all(np.array_equal(o, outs[0]) for o in outs)


def test_mlp_swiglu_pass_widths():
    T, H, I = 150, 256, 384
    X, W1, W2 = inputs.mlp(T, H, I, seed=72)
    ref = oracle.mlp_bf16(X, W1, W2)
    op = rc.Op(rc.OP_MLP, m=T, n=I, k=H)
    outs = []
    for vec in VECS:
        s = op.schedule(rc.T(rc.T_FUSE, 0, stage=0), rc.T(rc.T_VECTORIZE, vec, stage=0),
                        rc.T(rc.T_SPLIT_K, 2, stage=1), rc.T(rc.T_VECTORIZE, vec, stage=1))
        Y = empty_bf16(T, H).fill_(0x7FC0)
        op.run(s, [to_dev(X), to_dev(W1), to_dev(W2), Y])
        op.check()
        outs.append(Y.cpu().numpy())
        assert rel_err(from_dev_bf16(Y), ref) <= TOL, vec
    assert all(np.array_equal(o, outs[0]) for o in outs)


def test_conv_bias_silu_pass_widths():
    N, H, W, C, Cout = 1, 8, 16, 64, 160
    x, w, b = inputs.conv2d(N, H, W, C, Cout, seed=73)
    ref = oracle.conv2d_nhwc_bf16(x, w, b)
    op = rc.Op(rc.OP_CONV2D, img_n=N, img_h=H, img_w=W, c_in=C, c_out=Cout, kr=3, ks=3, stride=1, pad=1,
               flags=rc.EPI_BIAS | rc.EPI_SILU)
    outs = []
    for split, fuse in ((1, 0), (3, 1)):
        for vec in VECS:
            s = op.schedule(rc.T(rc.T_TILE_SIZE, 80, axis=1), rc.T(rc.T_SPLIT_K, split), rc.T(rc.T_FUSE, fuse),
                            rc.T(rc.T_VECTORIZE, vec))
            y = empty_bf16(N, H, W, Cout).fill_(0x7FC0)
            op.run(s, [to_dev(x), to_dev(w), to_dev(b), y])
            op.check()
            outs.append(y.cpu().numpy())
            assert rel_err(from_dev_bf16(y).reshape(-1, Cout), ref) <= TOL, (split, fuse, vec)
    assert all(np.array_equal(o, outs[0]) for o in outs[:3]) and all(np.array_equal(o, outs[3]) for o in outs[3:])


@pytest.mark.parametrize("fuse", [0, 1])
def test_moe_gather_and_combine_widths(fuse):
    T, H, E, I, K = 200, 256, 8, 128, 2
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=74)
    ids, w, _, _ = oracle.moe_route(logits, K)
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    op = rc.Op(rc.OP_MOE, tokens=T, hidden=H, experts=E, inter=I, top_k=K)
    outs = []
    for vec in VECS:
        s = op.schedule(rc.T(rc.T_VECTORIZE, vec, stage=0), rc.T(rc.T_VECTORIZE, vec, stage=2),
                        rc.T(rc.T_FUSE, fuse, stage=2), rc.T(rc.T_TILE_SIZE, 64, axis=1, stage=1),
                        rc.T(rc.T_TILE_SIZE, 128, axis=1, stage=2))
        assert s.knobs(0)["vec"] == vec and s.knobs(2)["vec"] == vec
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(s, [to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2), out])
        op.check()
        outs.append(out.cpu().numpy())
        assert rel_err(from_dev_bf16(out), ref) <= TOL, vec
    if not fuse:  # the gather-reduce combine is deterministic; the atomic one sums in arrival order
        assert all(np.array_equal(o, outs[0]) for o in outs)
