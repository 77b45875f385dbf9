"""MoE routing (bit-exact) and the routed SwiGLU FFN layer on the GPU against
the fp64 oracle. Routing ids, offsets and the permutation must be identical;
weights agree to fp32 rounding; layer outputs to 2e-2 normwise (bf16)."""
import itertools

import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import empty_bf16, from_dev_bf16, rel_err, to_dev, torch

pytestmark = pytest.mark.gpu
TOL = 2e-2


def run_route(logits, E, K, tile_m=4, renorm=True):
    T = logits.shape[0]
    fp32 = logits.dtype == np.float32
    op = rc.Op(rc.OP_MOE_ROUTE, tokens=T, experts=E, top_k=K, logits_fp32=int(fp32), renorm=int(renorm))
    ids = torch.empty(T, K, dtype=torch.int32, device="cuda")
    w = torch.empty(T, K, dtype=torch.float32, device="cuda")
    off = torch.empty(E + 1, dtype=torch.int32, device="cuda")
    perm = torch.empty(T * K, dtype=torch.int32, device="cuda")
    op.run(op.schedule(rc.T(rc.T_TILE_SIZE, tile_m, axis=0)), [to_dev(logits), ids, w, off, perm])
    op.check()
    return ids.cpu().numpy(), w.cpu().numpy(), off.cpu().numpy(), perm.cpu().numpy()


@pytest.mark.parametrize("T,E,K,fp32", [(4096, 64, 8, False), (1000, 16, 4, False), (333, 256, 16, False),
                                        (517, 33, 3, True), (64, 16, 16, False), (1, 8, 1, False)])
def test_routing_bit_exact(T, E, K, fp32):
    logits, _, _, _ = inputs.moe(T, 8, E, 8, seed=41, logits_fp32=fp32)
    r_ids, r_w, r_off, r_perm = oracle.moe_route(logits, K)
    for tm in (4, 8, 16):
        ids, w, off, perm = run_route(logits, E, K, tm)
        np.testing.assert_array_equal(ids, r_ids)
        np.testing.assert_array_equal(off, r_off)
        np.testing.assert_array_equal(perm, r_perm)
        np.testing.assert_allclose(w, r_w, rtol=2e-6, atol=1e-7)
    _, w_raw, _, _ = run_route(logits, E, K, renorm=False)
    np.testing.assert_allclose(w_raw, oracle.moe_route(logits, K, renorm=False)[1], rtol=2e-6, atol=1e-7)


def test_routing_ties_and_imbalance():
    T, E, K = 300, 64, 8
    L = np.zeros((T, E))
    L[100:, :] = np.random.default_rng(0).standard_normal((T - 100, E)).round(1)  # coarse values: many ties
    L[200:, :8] += 5.0  # 100 tokens all pick experts 0..7
    logits = inputs.to_bf16_bits(L)
    r = oracle.moe_route(logits, K)
    g = run_route(logits, E, K)
    for a, b in zip(g[:1] + g[2:], r[:1] + r[2:]):
        np.testing.assert_array_equal(a, b)
    assert list(g[0][0]) == list(range(8))  # all-equal row: lowest ids first


@pytest.mark.parametrize("fp32", [False, True])
def test_routing_nan_logits(fp32):
    # a NaN logit ranks below every number (read as -inf, ties by lower id) and gets weight 0;
    # rows with fewer than k numbers still route to k distinct experts below E
    T, E, K = 64, 64, 8
    logits, _, _, _ = inputs.moe(T, 8, E, 8, seed=46, logits_fp32=True)
    L = logits.astype(np.float64)
    rng = np.random.default_rng(3)
    L[0, :] = np.nan  # no number at all: ids 0..7
    L[1, 3:] = np.nan  # three numbers, then the five lowest NaN ids
    for t in range(2, T, 3):
        L[t, rng.choice(E, size=rng.integers(1, E), replace=False)] = np.nan
    lg = L.astype(np.float32) if fp32 else inputs.to_bf16_bits(L)
    r_ids, r_w, r_off, r_perm = oracle.moe_route(lg, K)
    assert list(r_ids[0]) == list(range(8))
    ids, w, off, perm = run_route(lg, E, K)
    np.testing.assert_array_equal(ids, r_ids)
    np.testing.assert_array_equal(off, r_off)
    np.testing.assert_array_equal(perm, r_perm)
    ok = np.isfinite(r_w).all(axis=1)  # the all-NaN row has no softmax
    assert ok.sum() == T - 1
    np.testing.assert_allclose(w[ok], r_w[ok], rtol=2e-6, atol=1e-7)


def moe_op(T, H, E, I, K):
    return rc.Op(rc.OP_MOE, tokens=T, hidden=H, experts=E, inter=I, top_k=K)


def moe_sched(op, tm, tn1, st1, tn2, st2, fuse, persistent=0, tile_k=64, tile_m=128, gather=0, split=0):
    # gather = 1: the grouped gate/up GEMM's producer gathers the token rows itself (compute location 1);
    # split = 1 (layout 1, CTA pairs): a segment's last remainder of at most 128 rows goes to a one-CTA launch
    return op.schedule(rc.T(rc.T_COMPUTE_LOCATION, gather, stage=1),
                       rc.T(rc.T_LAYOUT, split, stage=1), rc.T(rc.T_LAYOUT, split, stage=2),
                       rc.T(rc.T_TILE_SIZE, tm, axis=0, stage=0), rc.T(rc.T_TILE_SIZE, tn1, axis=1, stage=1),
                       rc.T(rc.T_PIPELINE_STAGES, st1, stage=1), rc.T(rc.T_TILE_SIZE, tn2, axis=1, stage=2),
                       rc.T(rc.T_PIPELINE_STAGES, st2, stage=2), rc.T(rc.T_FUSE, fuse, stage=2),
                       rc.T(rc.T_PARALLEL, persistent, stage=1), rc.T(rc.T_PARALLEL, persistent, stage=2),
                       rc.T(rc.T_TILE_SIZE, tile_k, axis=2, stage=1), rc.T(rc.T_TILE_SIZE, tile_k, axis=2, stage=2),
                       rc.T(rc.T_TILE_SIZE, tile_m, axis=0, stage=1), rc.T(rc.T_TILE_SIZE, tile_m, axis=0, stage=2))


def test_moe_layer_schedule_sweep():
    T, H, E, I, K = 200, 128, 8, 64, 2
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=42)
    ids, w, off, perm = oracle.moe_route(logits, K)
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    op = moe_op(T, H, E, I, K)
    dl, dX, d1, d2 = to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2)
    for tn1, tn2, fuse, st, pe, tk, tm, ga in itertools.product((32, 64, 128), (64, 128, 224, 256), (0, 1), (1, 3),
                                                                (0, 1), (64, 128), (128, 256), (0, 1)):
        try:  # CTA pairs (tm = 256) take 256 rows of one expert's segment
            s = moe_sched(op, 8, tn1, st, tn2, st, fuse, pe, tk, tm, ga)
        except rc.RcError:
            continue  # shared memory (K = 128, 3 stages, widest N); gather on pairs
        out = empty_bf16(T, H).fill_(0x7FC0)
        gi = torch.empty(T, K, dtype=torch.int32, device="cuda")
        gp = torch.empty(T * K, dtype=torch.int32, device="cuda")
        op.run(s, [dl, dX, d1, d2, out, gi, None, None, gp])
        op.check()
        np.testing.assert_array_equal(gi.cpu().numpy(), ids)
        np.testing.assert_array_equal(gp.cpu().numpy(), perm)
        err = rel_err(from_dev_bf16(out), ref)
        assert err <= TOL, (tn1, tn2, fuse, st, pe, tk, tm, ga, err)


@pytest.mark.parametrize("T,E,K,kinds", [(200, 8, 2, {"rest"}), (700, 16, 4, {"pairs"}),
                                         (1000, 5, 3, {"pairs", "rest"}), (2000, 12, 3, {"pairs", "rest"})])
def test_moe_split_segments(T, E, K, kinds):
    # CTA pairs with each segment's short remainder (1 .. 128 rows past its last whole or more than
    # half-full 256-row tile) in a second, one-CTA launch: both grouped GEMMs, fused and unfused combine,
    # persistent or not, ring depths that the one-CTA launch has to trim
    H, I = 128, 64
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=45 + T)
    ids, w, off, perm = oracle.moe_route(logits, K)
    rows = np.diff(off)
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    op = moe_op(T, H, E, I, K)
    dl, dX, d1, d2 = to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2)
    n = 0
    for tn1, tn2, fuse, st, pe, tk in itertools.product((64, 128), (128, 256), (0, 1), (3, 6), (0, 1), (64, 128)):
        try:
            s = moe_sched(op, 8, tn1, st, tn2, st, fuse, pe, tk, 256, 0, 1)
        except rc.RcError:
            continue  # shared memory of the pair ring
        assert s.knobs(1)["layout"] == 1 and s.knobs(2)["layout"] == 1
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(s, [dl, dX, d1, d2, out])
        op.check()
        err = rel_err(from_dev_bf16(out), ref)
        assert err <= TOL, (tn1, tn2, fuse, st, pe, tk, err)
        n += 1
    assert n >= 16
    # which launches this case exercises: a remainder of 1 .. 128 rows goes to the one-CTA launch, whole
    # pair tiles or a remainder of 129 .. 255 rows to the pair launch
    rem = rows % 256
    seen = set()
    if ((rem > 0) & (rem <= 128)).any():
        seen.add("rest")
    if ((rows >= 256) | (rem > 128)).any():
        seen.add("pairs")
    assert seen == kinds, (seen, rows.tolist())
    # single-CTA M tiles have nothing to split: the canonical form drops the layout
    assert moe_sched(op, 8, 64, 3, 128, 3, 0, tile_m=128, split=1).knobs(1)["layout"] == 0


def moe_sched_t(op, tn1, tn2, st, pe, tk, l1=2, l2=2, raster=(0, 1), fuse=0, tm1=128, tm2=128):
    # layout 2: each grouped GEMM computes W X^T (weights on UMMA M, a segment's token tile on N);
    # M tile 256: a CTA pair, 128 weight rows per CTA and the token tile's rows split between them
    return op.schedule(rc.T(rc.T_LAYOUT, l1, stage=1), rc.T(rc.T_LAYOUT, l2, stage=2),
                       rc.T(rc.T_TILE_SIZE, 8, axis=0, stage=0), rc.T(rc.T_TILE_SIZE, tn1, axis=1, stage=1),
                       rc.T(rc.T_TILE_SIZE, tn2, axis=1, stage=2), rc.T(rc.T_TILE_SIZE, tm1, axis=0, stage=1),
                       rc.T(rc.T_TILE_SIZE, tm2, axis=0, stage=2),
                       rc.T(rc.T_PIPELINE_STAGES, st, stage=1), rc.T(rc.T_PIPELINE_STAGES, st, stage=2),
                       rc.T(rc.T_PARALLEL, pe, stage=1), rc.T(rc.T_PARALLEL, pe, stage=2),
                       rc.T(rc.T_TILE_SIZE, tk, axis=2, stage=1), rc.T(rc.T_TILE_SIZE, tk, axis=2, stage=2),
                       rc.T(rc.T_LOOP_ORDER, raster[0], group=raster[1], stage=1),
                       rc.T(rc.T_LOOP_ORDER, raster[0], group=raster[1], stage=2), rc.T(rc.T_FUSE, fuse, stage=2))


@pytest.mark.parametrize("T,E,K,H,I", [(200, 8, 2, 128, 64), (1000, 5, 3, 256, 192), (2000, 12, 3, 384, 256),
                                       (37, 4, 4, 192, 64)])
def test_moe_exchanged_operands(T, E, K, H, I):
    # Layout 2 on both grouped GEMMs: token tiles of 64, 128 or 256 rows cut into whole 16-row units
    # (32-row units on CTA pairs; segments of 9 .. 700 rows), weight tiles past I or H (masked
    # columns), K of one or several ring laps, persistent or not, both raster orders, one CTA or a pair
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=47 + T)
    ids, w, off, perm = oracle.moe_route(logits, K)
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    op = moe_op(T, H, E, I, K)
    dl, dX, d1, d2 = to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2)
    n = 0
    for tn1, tn2, st, pe, tk, ra, tm in itertools.product((32, 64, 128), (64, 128, 256), (2, 4), (0, 1), (64, 128),
                                                          ((0, 1), (1, 8)), (128, 256)):
        try:
            s = moe_sched_t(op, tn1, tn2, st, pe, tk, raster=ra, tm1=tm, tm2=tm)
        except rc.RcError:
            continue  # shared memory
        assert s.knobs(1)["layout"] == 2 and s.knobs(2)["layout"] == 2
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(s, [dl, dX, d1, d2, out])
        op.check()
        err = rel_err(from_dev_bf16(out), ref)
        assert err <= TOL, (tn1, tn2, st, pe, tk, ra, tm, err)
        n += 1
    assert n >= 120
    # one stage exchanged, the other on M tiles of tokens (one CTA or a CTA pair)
    for l1, l2, tm2 in ((2, 0, 128), (0, 2, 128), (2, 0, 256), (2, 1, 256)):
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(moe_sched_t(op, 64, 128, 3, 1, 64, l1, l2, tm2=tm2), [dl, dX, d1, d2, out])
        op.check()
        assert rel_err(from_dev_bf16(out), ref) <= TOL, (l1, l2, tm2)


def test_moe_exchanged_operands_legality():
    op = moe_op(256, 128, 8, 64, 2)
    # persistent CTAs with 256-row token tiles keep a single accumulator of 512 TMEM columns
    assert moe_sched_t(op, 128, 256, 2, 1, 64).knobs(2)["persistent"] == 1
    with pytest.raises(rc.RcError):
        moe_sched_t(op, 64, 224, 2, 0, 64)  # token tiles of 64, 128 or 256 rows
    with pytest.raises(rc.RcError):
        moe_sched_t(op, 64, 128, 2, 0, 64, fuse=1)  # the atomic combine epilogue is not offered
    with pytest.raises(rc.RcError):
        moe_sched_t(op, 64, 128, 2, 0, 64, fuse=1, tm2=256)


def test_moe_layer_imbalanced_and_empty_experts():
    T, H, E, I, K = 300, 128, 16, 128, 4
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=43)
    L = inputs.bf16_bits_to_f64(logits)
    L[:, :4] += 8.0  # every token routes to experts 0..3: 300 rows each, 12 experts empty
    logits = inputs.to_bf16_bits(L)
    ids, w, off, _ = oracle.moe_route(logits, K)
    assert (np.diff(off)[4:] == 0).all() and (np.diff(off)[:4] == T).all()
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    op = moe_op(T, H, E, I, K)
    for fuse, pe, tm, ga, sp in itertools.product((0, 1), (0, 1), (128, 256), (0, 1), (0, 1)):
        if ga and tm == 256 or sp and tm == 128:
            continue
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(moe_sched(op, 4, 64, 2, 128, 2, fuse, pe, tile_m=tm, gather=ga, split=sp),
               [to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2), out])
        op.check()
        assert rel_err(from_dev_bf16(out), ref) <= TOL, (fuse, pe, tm, ga, sp)
    for tn1, tn2, pe, tm in itertools.product((32, 128), (64, 256), (0, 1), (128, 256)):  # exchanged operand roles
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(moe_sched_t(op, tn1, tn2, 2, pe, 64, tm1=tm, tm2=tm), [to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2), out])
        op.check()
        assert rel_err(from_dev_bf16(out), ref) <= TOL, (tn1, tn2, pe, tm)


def test_moe_full_size_sampled_tokens():
    # T=4096 tokens, H=7168, 64 experts with I=2048, top-8 softmax routing.
    T, H, E, I, K = 4096, 7168, 64, 2048, 8
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=6)
    ids, w, off, perm = oracle.moe_route(logits, K)
    tok = np.array([0, 1, 2047, 4095], dtype=np.int64)
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w, tok=tok)
    op = moe_op(T, H, E, I, K)
    dl, dX, d1, d2 = to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2)
    del W1, W2
    for s in [op.schedule(), moe_sched(op, 8, 128, 2, 256, 2, 0), moe_sched(op, 16, 64, 4, 128, 3, 1),
              moe_sched(op, 8, 128, 4, 256, 3, 0, 1), moe_sched(op, 8, 64, 3, 224, 2, 0, gather=1),
              moe_sched(op, 8, 128, 2, 224, 2, 1, 1, tile_k=128, gather=1),
              # CTA pairs with short remainders split off to one-CTA launches
              moe_sched(op, 8, 128, 3, 256, 4, 0, 1, tile_m=256, split=1),
              moe_sched(op, 8, 128, 3, 256, 3, 1, 0, tile_m=256, split=1),
              # exchanged operand roles: 256-row token tiles, and 128-row tiles on persistent CTAs
              moe_sched_t(op, 128, 256, 3, 0, 64), moe_sched_t(op, 64, 128, 4, 1, 64, raster=(1, 8)),
              moe_sched_t(op, 128, 224, 3, 0, 64, l2=0),
              moe_sched_t(op, 128, 256, 4, 1, 64, tm1=256, tm2=256), moe_sched_t(op, 64, 128, 2, 0, 128, tm1=256, tm2=256)]:
        out = empty_bf16(T, H)
        gi = torch.empty(T, K, dtype=torch.int32, device="cuda")
        go = torch.empty(E + 1, dtype=torch.int32, device="cuda")
        gp = torch.empty(T * K, dtype=torch.int32, device="cuda")
        op.run(s, [dl, dX, d1, d2, out, gi, None, go, gp])
        op.check()
        np.testing.assert_array_equal(gi.cpu().numpy(), ids)
        np.testing.assert_array_equal(go.cpu().numpy(), off)
        np.testing.assert_array_equal(gp.cpu().numpy(), perm)
        assert rel_err(from_dev_bf16(out)[tok], ref) <= TOL, str(s)


def test_moe_layer_256_experts():
    # the most segments a grouped GEMM takes (each CTA holds the segment table in shared memory,
    # eight segments per lane of the building warp); most experts get no or one row
    T, H, E, I, K = 96, 128, 256, 64, 6
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=44)
    ids, w, off, _ = oracle.moe_route(logits, K)
    ref = oracle.moe_ffn_bf16(X, W1, W2, ids, w)
    op = moe_op(T, H, E, I, K)
    for tm, fuse in itertools.product((128, 256), (0, 1)):
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(moe_sched(op, 8, 64, 2, 128, 2, fuse, tile_m=tm), [to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2), out])
        op.check()
        assert rel_err(from_dev_bf16(out), ref) <= TOL, (tm, fuse)
    for pe, tm in itertools.product((0, 1), (128, 256)):  # exchanged operand roles
        out = empty_bf16(T, H).fill_(0x7FC0)
        op.run(moe_sched_t(op, 32, 64, 2, pe, 64, tm1=tm, tm2=tm), [to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2), out])
        op.check()
        assert rel_err(from_dev_bf16(out), ref) <= TOL, (pe, tm)


def test_moe_host_path_matches_device_path():
    # rc_run_host copies W1 and W2 on a second stream while routing and the gate/up stage run;
    # the result must equal the device-buffer run bit for bit
    T, H, E, I, K = 256, 128, 8, 64, 2
    logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=45)
    op = moe_op(T, H, E, I, K)
    s = moe_sched(op, 8, 64, 2, 128, 2, 0)
    Yh = np.zeros((T, H), np.uint16)
    op.run_host(s, [logits, X, W1, W2, Yh])
    dY = empty_bf16(T, H)
    op.run(s, [to_dev(logits), to_dev(X), to_dev(W1), to_dev(W2), dY])
    op.check()
    np.testing.assert_array_equal(Yh, dY.cpu().numpy().view(np.uint16))
    ids, w, _, _ = oracle.moe_route(logits, K)
    assert rel_err(inputs.bf16_bits_to_f64(Yh), oracle.moe_ffn_bf16(X, W1, W2, ids, w)) <= TOL
