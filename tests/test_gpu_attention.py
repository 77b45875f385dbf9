"""Fused causal GQA attention on the GPU against the fp64 oracle.

Every legal schedule (key block, ring depth, query-block order, V layout) must
match the oracle (Sec. 2: transformations preserve semantics). O is bf16
(2e-2 normwise); LSE is fp32 (1e-3 normwise).
"""
import itertools

import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import empty_bf16, from_dev_bf16, rel_err, to_dev, torch

pytestmark = pytest.mark.gpu
TOL = 2e-2
TOL_LSE = 1e-3


def att_op(B, S, Hq, Hkv, causal=True):
    return rc.Op(rc.OP_ATTENTION, batch=B, seq=S, heads_q=Hq, heads_kv=Hkv, head_dim=128, causal=int(causal))


def sched(op, bn, stages, raster, layout, loc=0, unroll=1, par=0, tm=128):
    """loc: P in shared (0) or tensor memory (1), or row sums on the tensor core (2); unroll: S buffers;
    par: one issuing warp (0), issue split over warps (1), and two softmax threads per row (2);
    tm: query rows per CTA (256: two query tiles sharing each K and V block)."""
    return op.schedule(rc.T(rc.T_TILE_SIZE, bn, axis=1), rc.T(rc.T_PIPELINE_STAGES, stages),
                       rc.T(rc.T_LOOP_ORDER, raster, group=1), rc.T(rc.T_LAYOUT, layout),
                       rc.T(rc.T_COMPUTE_LOCATION, loc), rc.T(rc.T_UNROLL, unroll), rc.T(rc.T_PARALLEL, par),
                       rc.T(rc.T_TILE_SIZE, tm, axis=0))


def sched2q(op, stages, raster, layout):
    """The two-query-tile kernel (TileSize M = 256); its other knobs are fixed by its canonical form."""
    return sched(op, 128, stages, raster, layout, 1, 1, 1, tm=256)


def run(op, s, Q, K, V):
    B, S, Hq, D = Q.shape
    dO = empty_bf16(B, S, Hq, D).fill_(0x7FC0)
    lse = torch.full((B, Hq, S), float("nan"), dtype=torch.float32, device="cuda")
    op.run(s, [to_dev(Q), to_dev(K), to_dev(V), dO, lse])
    op.check()
    return from_dev_bf16(dO), lse.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("B,S,Hq,Hkv", [(2, 296, 4, 2), (1, 128, 2, 2), (1, 200, 8, 1)])
def test_attention_schedule_sweep(B, S, Hq, Hkv, causal):
    Q, K, V = inputs.attention(B, S, Hq, Hkv, 128, seed=61)
    O_ref, L_ref = oracle.attention_bf16(Q, K, V, causal=causal)
    op = att_op(B, S, Hq, Hkv, causal)
    n = 0
    for bn, st, ra, lay, loc, un, par in itertools.product((64, 128), (1, 2, 3, 4), (0, 1), (0, 1), (0, 1, 2), (1, 2),
                                                          (0, 1, 2)):
        try:
            s = sched(op, bn, st, ra, lay, loc, un, par)
        except rc.RcError:
            continue  # illegal here (shared memory, S % 8 for the transposed V, variant combinations)
        O, L = run(op, s, Q, K, V)
        assert rel_err(O, O_ref) <= TOL, (bn, st, ra, lay, loc, un, par, rel_err(O, O_ref))
        assert rel_err(L, L_ref) <= TOL_LSE, (bn, st, ra, lay, loc, un, par)
        n += 1
    assert n >= 40
    with pytest.raises(rc.RcError):  # row sums on the tensor core read V as given
        sched(op, 64, 2, 0, 1, 2, 1, 1)
    # each kernel family's canonical form: one issuing warp keeps P in shared memory and one S buffer,
    # split issue keeps P in tensor memory, so one Parallel transformation moves between them
    assert str(sched(op, 64, 2, 0, 0, 0, 2, 0)) == str(sched(op, 64, 2, 0, 0, 0, 1, 0))
    assert str(sched(op, 64, 2, 0, 0, 0, 1, 1)) == str(sched(op, 64, 2, 0, 0, 1, 1, 1))
    assert op.schedule(rc.T(rc.T_PARALLEL, 1)).knobs(0)["location"] == 1


@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("B,S,Hq,Hkv", [(2, 296, 4, 2), (1, 64, 2, 2), (1, 129, 2, 1), (1, 520, 8, 2), (2, 1000, 4, 1)])
def test_attention_two_query_tiles_sweep(B, S, Hq, Hkv, causal):
    # two 128-row query tiles per CTA: ragged sequences, a second tile with no row inside the
    # sequence (S = 64, 129), several CTAs per head, batch 2 (rows of the next sequence behind a
    # ragged key block are masked), every ring depth, query order and V layout
    Q, K, V = inputs.attention(B, S, Hq, Hkv, 128, seed=63)
    O_ref, L_ref = oracle.attention_bf16(Q, K, V, causal=causal)
    op = att_op(B, S, Hq, Hkv, causal)
    n = 0
    for st, ra, lay in itertools.product((1, 2, 3), (0, 1), (0, 1)):
        if lay == 1 and S % 8:
            with pytest.raises(rc.RcError):
                sched2q(op, st, ra, lay)
            continue
        O, L = run(op, sched2q(op, st, ra, lay), Q, K, V)
        assert rel_err(O, O_ref) <= TOL, (st, ra, lay, rel_err(O, O_ref))
        assert rel_err(L, L_ref) <= TOL_LSE, (st, ra, lay)
        n += 1
    assert n >= 6
    # canonical form: TileSize M = 256 fixes 128-key blocks, P in tensor memory, one S buffer per tile and
    # one softmax thread per row, whatever the other families' knobs were
    k = sched(op, 64, 2, 0, 0, 0, 2, 2, tm=256).knobs(0)
    assert (k["tile_m"], k["tile_n"], k["location"], k["unroll"], k["persistent"]) == (256, 128, 1, 1, 1)
    assert str(sched(op, 64, 2, 0, 0, 0, 2, 0, tm=256)) == str(sched2q(op, 2, 0, 0))
    with pytest.raises(rc.RcError):  # a 128-key K ring of four stages does not fit beside two query tiles
        sched2q(op, 4, 0, 0)


def test_attention_single_token_and_no_lse():
    Q, K, V = inputs.attention(1, 1, 4, 2, 128, seed=62)
    op = att_op(1, 1, 4, 2)
    O, L = run(op, op.schedule(rc.T(rc.T_LAYOUT, 0)), Q, K, V)
    for h in range(4):  # a single visible key returns its value row
        np.testing.assert_allclose(O[0, 0, h], inputs.bf16_bits_to_f64(V)[0, 0, h // 2], rtol=1e-2, atol=1e-2)
    dO = empty_bf16(1, 1, 4, 128)
    op.run(op.schedule(rc.T(rc.T_LAYOUT, 0)), [to_dev(Q), to_dev(K), to_dev(V), dO, None])
    op.check()


def test_attention_full_size_sampled_queries():
    # Llama-3-8B-shaped layer: batch 1, seq 2048, 32 query heads, 8 KV heads, d = 128, causal.
    B, S, Hq, Hkv = 1, 2048, 32, 8
    Q, K, V = inputs.attention(B, S, Hq, Hkv, 128, seed=4)
    qpos = np.array([0, 1, 63, 64, 127, 128, 129, 1000, 1023, 1024, 2000, 2046, 2047], dtype=np.int64)
    O_ref, L_ref = oracle.attention_bf16(Q, K, V, causal=True, qpos=qpos)
    op = att_op(B, S, Hq, Hkv)
    for s in [op.schedule(), sched(op, 128, 2, 1, 0), sched(op, 64, 3, 0, 1), sched(op, 64, 1, 1, 0),
              # split issue, one S buffer (two CTAs per SM at BN 64) or two, V as given or transposed
              sched(op, 64, 2, 1, 0, 1, 1, 1), sched(op, 64, 2, 0, 1, 1, 1, 1), sched(op, 64, 3, 1, 0, 1, 1, 1),
              sched(op, 128, 2, 1, 0, 1, 1, 1), sched(op, 128, 3, 0, 1, 1, 1, 1),
              sched(op, 64, 2, 1, 0, 1, 2, 1), sched(op, 64, 4, 1, 1, 1, 2, 1), sched(op, 128, 2, 1, 0, 1, 2, 1),
              # two softmax threads per row
              sched(op, 64, 2, 1, 0, 1, 1, 2), sched(op, 64, 3, 0, 1, 1, 1, 2), sched(op, 128, 2, 1, 0, 1, 1, 2),
              sched(op, 64, 2, 1, 0, 1, 2, 2),
              # row sums of P on the tensor core
              sched(op, 64, 2, 1, 0, 2, 1, 1), sched(op, 64, 3, 0, 0, 2, 1, 1), sched(op, 128, 2, 1, 0, 2, 1, 1),
              sched(op, 64, 2, 1, 0, 2, 2, 1), sched(op, 128, 2, 1, 0, 2, 1, 2),
              # two query tiles per CTA
              sched2q(op, 2, 1, 0), sched2q(op, 3, 0, 1), sched2q(op, 1, 1, 0)]:
        O, L = run(op, s, Q, K, V)
        assert rel_err(O[:, qpos], O_ref) <= TOL, str(s)
        assert rel_err(L[:, :, qpos], L_ref) <= TOL_LSE, str(s)


def test_flux_shaped_noncausal_attention_sampled_queries():
    # FLUX-style (DiT) self-attention: batch 1, 4096 image tokens, 24 heads (MHA), d = 128, no mask.
    B, S, H = 1, 4096, 24
    Q, K, V = inputs.attention(B, S, H, H, 128, seed=7)
    qpos = np.array([0, 1, 127, 128, 2047, 2048, 4000, 4095], dtype=np.int64)
    O_ref, L_ref = oracle.attention_bf16(Q, K, V, causal=False, qpos=qpos)
    op = att_op(B, S, H, H, causal=False)
    for s in [op.schedule(), sched(op, 64, 2, 0, 0, 1, 1, 1), sched(op, 64, 3, 1, 1, 1, 1, 1),
              sched(op, 128, 2, 1, 0, 1, 2, 1), sched(op, 64, 2, 1, 0, 1, 1, 2), sched(op, 64, 2, 0, 0, 2, 1, 1),
              sched(op, 128, 2, 0, 0, 2, 1, 1), sched2q(op, 2, 0, 0), sched2q(op, 3, 1, 0), sched2q(op, 2, 1, 1)]:
        O, L = run(op, s, Q, K, V)
        assert rel_err(O[:, qpos], O_ref) <= TOL, str(s)
        assert rel_err(L[:, :, qpos], L_ref) <= TOL_LSE, str(s)
