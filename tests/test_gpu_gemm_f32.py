"""fp32 GEMM+bias+ReLU on the GPU against the fp64 oracle, for every schedule of
the 54-point space (semantics preservation, Sec. 2) and ragged shapes."""
import itertools

import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import rel_err, torch

pytestmark = pytest.mark.gpu
TOL = 1e-4  # fp32 arithmetic, normwise max-relative error


def _sched(op, bm, bn, bk, u):
    return op.schedule(rc.T(rc.T_TILE_SIZE, bm, axis=0), rc.T(rc.T_TILE_SIZE, bn, axis=1),
                       rc.T(rc.T_TILE_SIZE, bk, axis=2), rc.T(rc.T_UNROLL, u))


def test_all_54_schedules_256_cube():
    A, B, bias = inputs.gemm_f32(256, 256, 256, seed=0)
    ref = oracle.gemm_bias_relu_f32(A, B, bias)
    op = rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256, flags=rc.EPI_BIAS | rc.EPI_RELU)
    dA, dB, db = (torch.from_numpy(x).cuda() for x in (A, B, bias))
    for bm, bn, bk, u in itertools.product((16, 32, 64), (16, 32, 64), (16, 32, 64), (1, 4)):
        dC = torch.full((256, 256), float("nan"), dtype=torch.float32, device="cuda")
        op.run(_sched(op, bm, bn, bk, u), [dA, dB, db, dC])
        op.check()
        got = dC.cpu().numpy().astype(np.float64)
        assert rel_err(got, ref) <= TOL, (bm, bn, bk, u)


@pytest.mark.parametrize("M,N,K", [(77, 45, 93), (1, 1, 1), (130, 67, 300), (64, 200, 17)])
def test_ragged_shapes(M, N, K):
    A, B, bias = inputs.gemm_f32(M, N, K, seed=1)
    op = rc.Op(rc.OP_GEMM_F32, m=M, n=N, k=K, flags=rc.EPI_BIAS | rc.EPI_RELU)
    ref = oracle.gemm_bias_relu_f32(A, B, bias)
    dA, dB, db = (torch.from_numpy(x).cuda() for x in (A, B, bias))
    for cfg in [(16, 16, 16, 1), (64, 32, 16, 4), (32, 64, 64, 4)]:
        dC = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        op.run(_sched(op, *cfg), [dA, dB, db, dC])
        op.check()
        assert rel_err(dC.cpu().numpy(), ref) <= TOL, cfg


def test_no_bias_no_relu_and_host_path():
    A, B, _ = inputs.gemm_f32(96, 80, 70, seed=2)
    op = rc.Op(rc.OP_GEMM_F32, m=96, n=80, k=70)
    C = np.zeros((96, 80), np.float32)
    op.run_host(op.schedule(rc.T(rc.T_TILE_SIZE, 32, axis=0)), [A, B, None, C])
    ref = oracle.gemm_bias_relu_f32(A, B, None, relu=False)
    assert rel_err(C, ref) <= TOL and (C < 0).any()


def test_measure_reports_times():
    A, B, bias = inputs.gemm_f32(256, 256, 256, seed=0)
    op = rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256, flags=rc.EPI_BIAS | rc.EPI_RELU)
    dA, dB, db = (torch.from_numpy(x).cuda() for x in (A, B, bias))
    dC = torch.empty(256, 256, dtype=torch.float32, device="cuda")
    ss = [_sched(op, 16, 16, 16, 1), _sched(op, 64, 64, 16, 4)]
    ms = op.measure(ss, [dA, dB, db, dC], warmup=2, repeats=5)
    for m in ms:
        assert m.status == rc.OK and 0 < m.ms_min <= m.ms_median and m.tflops > 0
