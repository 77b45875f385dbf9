"""The benchmark's oracle check of the schedules it reports (bench.Workload.parity).

Every op the benchmark reports is first run once with its chosen schedule and
compared with the fp64 oracle on sampled outputs. These tests run that check
on small shapes of every workload, and plant a mistake in the oracle (on the
CPU side) to see the check refuse it.
"""
import numpy as np
import pytest

import bench
import oracle

pytestmark = pytest.mark.gpu

SMALL = {
    "mlp": {"tokens": 200, "hidden": 256, "inter": 384},
    "attention": {"seq": 296, "heads_q": 4, "heads_kv": 2},
    "attention_flux": {"seq": 256, "heads": 2},
    "conv2d": {"n": 1, "h": 16, "w": 16, "c": 64},
    "moe": {"tokens": 256, "hidden": 256, "experts": 8, "inter": 128, "top_k": 2},
    "decoder_layer": {"tokens": 128, "hidden": 256, "heads_q": 4, "heads_kv": 2, "inter": 256},
    "gemm_f32": {},
    "linear": {"m": 300, "n": 384, "k": 520},
}


@pytest.mark.parametrize("name", sorted(SMALL))
def test_parity_of_p0_and_a_tuned_schedule(name):
    wl = bench.Workload(name, SMALL[name])
    io = wl.device_io()
    par = wl.parity(wl.op.schedule(), io)
    assert par["ok"], par
    assert par["max_rel_err"] <= par["tol"]
    # a schedule from a short search must pass the same check
    _, best, m, _, _ = bench.search_best(wl.op, io, 24, seed=1, branching=2, finalists=2)
    assert wl.parity(best, io)["ok"]


def test_parity_refuses_a_wrong_result(monkeypatch):
    wl = bench.Workload("mlp", SMALL["mlp"])
    io = wl.device_io()
    good = oracle.mlp_bf16
    monkeypatch.setattr(oracle, "mlp_bf16", lambda *a, **k: 1.1 * good(*a, **k))  # planted in the oracle
    par = wl.parity(wl.op.schedule(), io)
    assert not par["ok"] and par["max_rel_err"] > par["tol"]


def test_parity_refuses_wrong_routing(monkeypatch):
    wl = bench.Workload("moe", SMALL["moe"])
    io = wl.device_io()
    good = oracle.moe_route

    def swapped(logits, k, renorm=True):
        ids, w, off, perm = good(logits, k, renorm)
        ids = ids.copy()
        ids[0, [0, 1]] = ids[0, [1, 0]]  # the first token's two picks in the wrong order
        return ids, w, off, perm

    monkeypatch.setattr(oracle, "moe_route", swapped)
    par = wl.parity(wl.op.schedule(), io)
    assert not par["routing_exact"] and not par["ok"]
