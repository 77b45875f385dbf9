"""The library's MCTS (rc_search_*) against the reference MCTS of oracle/mcts.py,
on a replayed measurement table (no GPU)."""
import itertools
import math

import pytest

import oracle.mcts as ref_mcts
from paper_2506_01374_gb300 import rc

# The fp32 GEMM schedule space of the 256^3 workload: CTA tiles {16,32,64}^3 x
# unroll {1,4}, written out here from the workload definition.
TILES = (16, 32, 64)
UNROLLS = (1, 4)
SPACE = [("tile", ax, v) for ax in range(3) for v in TILES] + [("unroll", 0, u) for u in UNROLLS]
P0 = (16, 16, 16, 1)


def ref_apply(p, tau):
    kind, ax, v = tau
    p = list(p)
    if kind == "tile":
        p[ax] = v
    else:
        p[3] = v
    return tuple(p)


def fake_ms(p):
    """Deterministic replayed 'measurement' of a program (ms)."""
    bm, bn, bk, u = p
    return 1.0 + ((bm * 7 + bn * 13 + bk * 3 + u * 5) % 17) / 10.0


def lib_program(s):
    k = s.knobs()
    return (k["tile_m"], k["tile_n"], k["tile_k"], k["unroll"])


def meas(p, fail=False):
    m = rc.Measurement()
    m.status = rc.ERR_PARITY if fail else rc.OK
    m.ms_median = 0.0 if fail else fake_ms(p)
    return m


def make_op():
    return rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256, flags=rc.EPI_BIAS | rc.EPI_RELU)


@pytest.mark.parametrize("seed,B,q", [(0, 2, 2), (7, 2, 0), (3, 4, 1)])
def test_trajectory_matches_reference(seed, B, q):
    op = make_op()
    assert [(t.kind, t.axis, t.value[0]) for t in op.transform_space()] == [
        (rc.T_TILE_SIZE if k == "tile" else rc.T_UNROLL, ax, v) for k, ax, v in SPACE]
    lib = rc.Search(op, seed=seed, branching=B, rollout=q)
    ref = ref_mcts.MCTS(P0, SPACE, ref_apply, seed=seed, B=B, q=q)
    res_lib, res_ref = [], []
    for it in range(40):
        nl = [lib_program(s) for s in lib.step(res_lib)]
        nr = ref.step(res_ref)
        assert nl == nr, f"iteration {it}"
        if not nl:
            break
        res_lib = [meas(p) for p in nl]
        res_ref = [fake_ms(p) for p in nr]
    st = lib.stats()
    assert st["nodes"] == len(ref.nodes)
    for i, nd in enumerate(ref.nodes):
        got = lib.node(i)
        assert got["N"] == nd.N and got["Q"] == pytest.approx(nd.Q, rel=1e-12)
        assert got["parent"] == (-1 if nd.parent is None else nd.parent)


def test_backprop_invariants():
    # Q and N of a node = its own rollout reward and visit + the sums over its children (Sec. 3.2)
    op = make_op()
    s = rc.Search(op, seed=11)
    res = []
    for _ in range(25):
        nxt = s.step(res)
        res = [meas(lib_program(x)) for x in nxt]
    n = s.stats()["nodes"]
    kids = {i: [] for i in range(n)}
    for i in range(1, n):
        kids[s.node(i)["parent"]].append(i)
    for i in range(n):
        nd = s.node(i)
        if nd["N"] == 0:
            continue
        assert nd["N"] == 1 + sum(s.node(c)["N"] for c in kids[i])
    root = s.node(0)
    assert root["N"] == 1 + sum(s.node(c)["N"] for c in kids[0])


def test_uct_closed_form_on_three_nodes():
    # Root with two visited children: UCT picks argmax Q/N + c sqrt(ln N_parent / N).
    ref = ref_mcts.MCTS(P0, SPACE, ref_apply, seed=0)
    a = ref_mcts.Node((32, 16, 16, 1), 0, 1)
    b = ref_mcts.Node((16, 32, 16, 1), 0, 1)
    ref.nodes += [a, b]
    ref.nodes[0].children = [1, 2]
    ref.nodes[0].N, a.N, b.N = 5, 3, 1
    a.Q, b.Q = 3.3, 0.9
    c = math.sqrt(2)
    ua = 3.3 / 3 + c * math.sqrt(math.log(5) / 3)
    ub = 0.9 / 1 + c * math.sqrt(math.log(5) / 1)
    assert ref._uct(1, 0) == pytest.approx(ua) and ref._uct(2, 0) == pytest.approx(ub)
    assert ub > ua  # the under-visited child wins here
    ref.nodes[0].expanded = True
    assert ref._select() == 2


def test_search_finds_exhaustive_optimum_and_is_deterministic():
    op = make_op()
    best_exhaustive = max(fake_ms(P0) / fake_ms(p) for p in itertools.product(TILES, TILES, TILES, UNROLLS))

    def run(seed):
        s = rc.Search(op, seed=seed)
        res, trace = [], []
        for _ in range(400):
            nxt = s.step(res)
            if not nxt:
                break
            trace += [x.hash for x in nxt]
            res = [meas(lib_program(x)) for x in nxt]
        return s, trace

    s1, t1 = run(5)
    s2, t2 = run(5)
    assert t1 == t2
    best, m = s1.best()
    assert fake_ms(P0) / m.ms_median == pytest.approx(best_exhaustive)
    assert s1.stats()["samples"] <= 54


def test_failed_candidates_get_zero_reward_and_search_continues():
    op = make_op()
    s = rc.Search(op, seed=2)
    nxt = s.step([])
    res = [meas(lib_program(x)) for x in nxt]
    for _ in range(5):
        nxt = s.step(res)
        res = [meas(lib_program(x), fail=True) for x in nxt]
    nxt = s.step(res)
    assert nxt  # still proposing
    assert s.stats()["best_reward"] == pytest.approx(1.0)  # only the root succeeded


def test_result_count_mismatch_is_an_error():
    s = rc.Search(make_op(), seed=0)
    s.step([])
    with pytest.raises(rc.RcError):
        s.step([])


def test_best_schedule_outlives_the_search():
    op = make_op()
    s = rc.Search(op, seed=4)
    res = []
    for _ in range(5):
        nxt = s.step(res)
        res = [meas(lib_program(x)) for x in nxt]
    best, m = s.best()
    knobs = best.knobs()
    del s
    import gc
    gc.collect()
    assert best.knobs() == knobs and best.hash == m.sched_hash


# ------------------------------------------------- one task of a composite op --

def _decoder_op():
    return rc.Op(rc.OP_DECODER_LAYER, tokens=512, hidden=1024, inter=2048, heads_q=8, heads_kv=2, head_dim=128)


def _stage_meas(s, noise):
    """Synthetic per-stage times: stage g's time from its own knobs; `noise` perturbs the others."""
    m = rc.Measurement()
    m.status = rc.OK
    m.n_stages = s.num_stages
    for g in range(s.num_stages):
        k = s.knobs(g)
        t = 1.0 + 0.01 * g + 1.0 / max(k["tile_n"], 1) + 0.1 / max(k["stages"], 1) + 0.05 * k["fuse"]
        m.stage_ms[g] = t + noise(g)
    m.ms_median = sum(m.stage_ms[g] for g in range(s.num_stages))
    return m


def _drive(srch, measure, samples):
    fed, res, pend = [], [], False
    while len(fed) < samples:
        nxt = srch.step(res)
        pend = False
        if not nxt:
            break
        res = [measure(s) for s in nxt]
        fed += list(zip(nxt, res))
        pend = True
    if pend:
        srch.step(res)
    return fed


def test_stage_mask_tunes_one_task_from_a_given_root():
    op = _decoder_op()
    root = op.schedule(rc.T(rc.T_FUSE, 1, stage=4), rc.T(rc.T_TILE_SIZE, 4, axis=0, stage=1))
    rng = iter(range(10 ** 6))

    def noise(g):  # the untouched stages' times jump around by up to 0.5 ms per measurement
        return 0.0 if g == 3 else 0.5 * ((next(rng) * 7919) % 101) / 100

    srch = rc.Search(op, seed=3, branching=4, stages=[3], root=root)
    fed = _drive(srch, lambda s: _stage_meas(s, noise), 120)
    assert fed[0][0].hash == root.hash  # the root is measured first
    for s, _ in fed:  # only stage 3 ever changes
        for g in range(6):
            if g != 3:
                assert s.knobs(g) == root.knobs(g)
    best, m = srch.best()
    # the objective is stage 3's own time: the best is the fastest stage-3 program seen, whatever the noise
    t3 = min(r.stage_ms[3] for _, r in fed)
    assert m.stage_ms[3] == pytest.approx(t3)
    assert srch.stats()["best_reward"] == pytest.approx(fed[0][1].stage_ms[3] / t3)


def test_stage_mask_and_root_are_validated():
    op = _decoder_op()
    with pytest.raises(rc.RcError) as e:
        rc.Search(op, stages=[6])
    assert e.value.status == rc.ERR_INVALID_ARG
    other = rc.Op(rc.OP_MLP, m=256, n=512, k=256)
    with pytest.raises(rc.RcError) as e:
        rc.Search(op, root=other.schedule())
    assert e.value.status == rc.ERR_INVALID_ARG
    # a task with a handful of programs is exhausted, not an error, for the caller
    srch = rc.Search(op, stages=[1], branching=4)
    fed = _drive(srch, lambda s: _stage_meas(s, lambda g: 0.0), 100)
    assert len({s.hash for s, _ in fed}) == 4  # TileSize tokens-per-CTA in {1, 2, 4, 8}
