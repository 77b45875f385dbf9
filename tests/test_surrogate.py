"""The learned surrogate f-hat of the search (rc_search_* with surrogate = 1).

Sec. 3.2: rollout programs are scored by a learned surrogate rather than run,
and proposals are screened by the cost model. The library's f-hat is checked
against the reference in oracle/surrogate.py (same definition, numpy fp64),
and that reference is pinned to closed forms and to an independent
least-squares solve. Measurements are synthetic (no GPU).
"""
import math

import numpy as np
import pytest

from oracle import surrogate as ref
from paper_2506_01374_gb300 import rc


def mlp_op():
    return rc.Op(rc.OP_MLP, m=2048, n=14336, k=4096)


def fake_stage_ms(g, k):
    """A synthetic, deterministic device time of one MLP stage from its knobs."""
    t = 1.0 + 0.5 * g
    t *= {32: 1.9, 64: 1.4, 128: 1.0, 224: 0.93, 256: 0.9}.get(k["tile_n"], 1.2)
    t *= 0.8 if k["tile_m"] == 256 else 1.0
    t *= {1: 1.6, 2: 1.1, 3: 1.0, 4: 1.02}.get(k["stages"], 1.05)
    t *= 0.97 if k["tile_k"] == 128 else 1.0
    t *= 1.0 + 0.07 * (k["split_k"] - 1)
    t *= 0.95 if k["persistent"] else 1.0
    t *= 0.9 if (g == 0 and k["fuse"]) else 1.0
    t *= 1.25 if (k["tile_n"] >= 224 and k["stages"] >= 4) else 1.0  # an interaction
    t *= 1.0 + 0.01 * ((k["raster"] * 3 + k["group"]) % 5)
    return t


def measure(s, per_stage=True):
    m = rc.Measurement()
    m.status = rc.OK
    st = [fake_stage_ms(g, s.knobs(g)) for g in range(2)]
    m.ms_median = sum(st)
    if per_stage:
        m.n_stages = 2
        for g in range(2):
            m.stage_ms[g] = st[g]
    return m


def run_search(samples, seed=0, surrogate=True, screen=1, per_stage=True, branching=4):
    op = mlp_op()
    srch = rc.Search(op, seed=seed, branching=branching, surrogate=surrogate, screen=screen)
    fed, res, best = [], [], math.inf
    while len(fed) < samples:
        nxt = srch.step(res)
        if not nxt:
            break
        res = [measure(s, per_stage) for s in nxt]
        for s, m in zip(nxt, res):
            fed.append(([s.knobs(0), s.knobs(1)], m.ms_median, [m.stage_ms[0], m.stage_ms[1]]))
            best = min(best, m.ms_median)
    if res:
        srch.step(res)  # consume the last batch (trains the model on it too)
    return srch, fed, best


# ------------------------------------------------------------ reference pins --

def test_reference_identical_rows_predict_geometric_mean():
    # one knob vector measured n times: the (nearly free) intercept takes the
    # mean log time and every indicator weight shrinks to 0
    k = rc.Op(rc.OP_LINEAR, m=64, n=64, k=64).schedule().knobs(0)
    ms = [1.0, 2.0, 4.0, 8.0]
    sur = ref.Surrogate([([k], t, [t]) for t in ms], per_stage=False)
    assert sur.predict_ms([k]) == pytest.approx(math.exp(np.mean(np.log(ms))), rel=1e-5)


def test_reference_recovers_an_additive_log_time():
    # log t = sum of per-knob effects over a replicated full factorial: with
    # many replicates the ridge penalty is negligible and every cell is fitted
    base = rc.Op(rc.OP_LINEAR, m=64, n=64, k=64).schedule().knobs(0)
    eff_n = {32: 0.3, 64: 0.0, 128: -0.2}
    eff_s = {1: 0.5, 2: 0.1, 3: 0.0}
    samples, cells = [], []
    for tn in eff_n:
        for st in eff_s:
            k = dict(base, tile_n=tn, stages=st)
            t = math.exp(1.0 + eff_n[tn] + eff_s[st])
            cells.append((k, t))
            samples += [([k], t, [t])] * 400
    sur = ref.Surrogate(samples, per_stage=False)
    for k, t in cells:
        assert sur.predict_ms([k]) == pytest.approx(t, rel=0.01)


def test_reference_solve_matches_augmented_least_squares():
    # the ridge solution is the least-squares solution of [X; sqrt(L)] w = [y; 0]
    rng = np.random.default_rng(3)
    base = rc.Op(rc.OP_LINEAR, m=64, n=64, k=64).schedule().knobs(0)
    samples = []
    for _ in range(60):
        k = dict(base, tile_n=int(rng.choice([32, 64, 128, 256])), stages=int(rng.integers(1, 5)),
                 persistent=int(rng.integers(0, 2)))
        samples.append(([k], float(rng.uniform(0.5, 3.0)), [0.0]))
    m = ref.Surrogate(samples, per_stage=False).models[0]
    X = np.zeros((len(m.rows), len(m.cols) + 1))
    X[:, 0] = 1.0
    for i, r in enumerate(m.rows):
        for n in r:
            X[i, m.cols[n]] = 1.0
    lam = np.full(X.shape[1], ref.LAMBDA)
    lam[0] = ref.LAMBDA_BIAS
    A = np.vstack([X, np.diag(np.sqrt(lam))])
    b = np.concatenate([np.asarray(m.ys), np.zeros(X.shape[1])])
    w, *_ = np.linalg.lstsq(A, b, rcond=None)
    np.testing.assert_allclose(m.w, w, rtol=1e-8, atol=1e-10)


# -------------------------------------------------------- library vs reference --

@pytest.mark.parametrize("per_stage", [True, False])
def test_library_surrogate_matches_reference(per_stage):
    srch, fed, _ = run_search(160, seed=1, per_stage=per_stage)
    st = srch.stats()
    n = st["model_samples"]
    assert n >= 24
    sur = ref.Surrogate(fed[:n], per_stage=per_stage)
    # predictions on schedules of the tree and on others
    op = mlp_op()
    probes = [op.schedule()] + [op.schedule(rc.T(rc.T_TILE_SIZE, tn, axis=1, stage=g), rc.T(rc.T_PIPELINE_STAGES, sg, stage=g))
                                for g in (0, 1) for tn in (64, 128) for sg in (2, 3)]
    for s in probes:
        want = sur.predict_ms([s.knobs(0), s.knobs(1)])
        assert srch.predict(s) == pytest.approx(want, rel=1e-9)


def test_surrogate_rollouts_are_not_measured():
    srch, fed, _ = run_search(200, seed=2)
    st = srch.stats()
    assert st["predicted"] > 0
    # after the fit only the expanded children are measured: fewer samples than nodes + measured rollouts
    assert st["samples"] < 2 * st["nodes"]


def test_surrogate_off_matches_plain_search_and_is_deterministic():
    a = run_search(120, seed=4, surrogate=False)[1]
    b = run_search(120, seed=4, surrogate=False)[1]
    assert [f[1] for f in a] == [f[1] for f in b]
    c = run_search(150, seed=4, surrogate=True, screen=3)[1]
    d = run_search(150, seed=4, surrogate=True, screen=3)[1]
    assert [f[1] for f in c] == [f[1] for f in d]
    with pytest.raises(rc.RcError):
        srch = rc.Search(mlp_op(), surrogate=False)
        srch.step([])
        srch.predict(mlp_op().schedule())


def test_screened_surrogate_search_is_more_sample_efficient():
    # on the synthetic landscape, best time after 300 measured programs,
    # averaged over seeds: screening by f-hat finds faster programs
    plain = np.mean([run_search(300, seed=s, surrogate=False)[2] for s in range(4)])
    screened = np.mean([run_search(300, seed=s, surrogate=True, screen=4)[2] for s in range(4)])
    assert screened < plain
