"""Reference learned surrogate f-hat for rollout rewards (CPU, numpy fp64).

TEST INFRASTRUCTURE ONLY: the tests use it to check the library's surrogate;
the product never imports it.

Sec. 3.2 scores a rollout program P_sim with a learned surrogate f-hat of the
objective instead of running it (reward = s * f-hat(P_sim)), and the cost model
screens proposals before they join the tree (appendix on proposal validity).
The surrogate is learned from the measurements the search has made:

  * a program is a knob vector per stage (tile sizes, unroll, pipeline stages,
    split-K, raster order and group, persistence, fusion, layout, vector
    width, compute location);
  * its features are 0/1 indicators: an intercept, one indicator per
    (stage, knob, value), and one per (stage, knob pair, value pair) for the
    knob pairs the kernels couple (tile M x N, N x K, N x stages, ...);
  * target: log of the measured device time; with per-stage times, one
    regression per stage on that stage's features and the op time predicted as
    the sum of exp(stage predictions); otherwise one regression of the op time;
  * fit: ridge regression, w = argmin ||X w - y||^2 + sum_j lambda_j w_j^2 with
    lambda = 1 for every indicator and 1e-6 for the intercept, i.e. the
    solution of (X^T X + diag(lambda)) w = X^T y; indicators never seen in
    training contribute 0 to a prediction.

Written from that definition with numpy.linalg.solve; shares nothing with the
library's implementation beyond the definition.
"""
from __future__ import annotations

import numpy as np

KNOBS = ("tile_m", "tile_n", "tile_k", "unroll", "stages", "split_k", "raster", "group", "persistent", "fuse",
         "layout", "vec", "location")
PAIRS = (("tile_m", "tile_n"), ("tile_n", "tile_k"), ("tile_n", "stages"), ("tile_k", "stages"),
         ("tile_m", "stages"), ("tile_m", "persistent"), ("tile_n", "persistent"), ("tile_n", "split_k"),
         ("persistent", "unroll"), ("tile_m", "unroll"), ("tile_n", "unroll"), ("persistent", "location"),
         ("tile_m", "fuse"), ("raster", "group"))
LAMBDA, LAMBDA_BIAS = 1.0, 1e-6


def indicators(stage: int, knobs: dict) -> list:
    """Names of the active indicators of one stage's knob vector (intercept excluded)."""
    out = [(stage, k, knobs[k]) for k in KNOBS]
    out += [(stage, a + "*" + b, (knobs[a], knobs[b])) for a, b in PAIRS]
    return out


class Ridge:
    def __init__(self):
        self.rows, self.ys = [], []

    def add(self, names: list, y: float):
        self.rows.append(names)
        self.ys.append(y)

    def fit(self):
        cols = {}
        for r in self.rows:
            for n in r:
                cols.setdefault(n, len(cols) + 1)
        X = np.zeros((len(self.rows), len(cols) + 1))
        X[:, 0] = 1.0
        for i, r in enumerate(self.rows):
            for n in r:
                X[i, cols[n]] = 1.0
        lam = np.full(len(cols) + 1, LAMBDA)
        lam[0] = LAMBDA_BIAS
        self.w = np.linalg.solve(X.T @ X + np.diag(lam), X.T @ np.asarray(self.ys))
        self.cols = cols
        return self

    def predict(self, names: list) -> float:
        return float(self.w[0] + sum(self.w[self.cols[n]] for n in names if n in self.cols))


class Surrogate:
    """f-hat over (knobs per stage, measurement) samples, fitted on all of them."""

    def __init__(self, samples: list, per_stage: bool):
        # samples: [(list of per-stage knob dicts, op ms, list of stage ms)]
        self.per_stage = per_stage
        S = len(samples[0][0])
        self.models = [Ridge() for _ in range(S if per_stage else 1)]
        for knobs, ms, stage_ms in samples:
            if per_stage:
                for g in range(S):
                    self.models[g].add(indicators(g, knobs[g]), float(np.log(stage_ms[g])))
            else:
                names = [n for g in range(S) for n in indicators(g, knobs[g])]
                self.models[0].add(names, float(np.log(ms)))
        for m in self.models:
            m.fit()

    def predict_ms(self, knobs: list) -> float:
        if self.per_stage:
            return float(sum(np.exp(self.models[g].predict(indicators(g, knobs[g]))) for g in range(len(knobs))))
        return float(np.exp(self.models[0].predict([n for g in range(len(knobs)) for n in indicators(g, knobs[g])])))
