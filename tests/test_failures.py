"""Failure detection without faulting a GPU.

Host side (no GPU): illegal schedules, NULL and misaligned tensors and bad
handles come back as status codes before any device work. Device side: the
bounded-wait self-test makes an mbarrier wait run out (nothing arrives) and
checks that the kernel reports a timeout and the context stays usable.
"""
import ctypes

import numpy as np
import pytest

from paper_2506_01374_gb300 import inputs, rc


def test_null_and_misaligned_tensors_are_rejected_before_device_work():
    op = rc.Op(rc.OP_LINEAR, m=64, n=64, k=64)
    s = op.schedule()
    with pytest.raises(rc.RcError) as e:
        op.run(s, [None, None, None])
    assert e.value.status == rc.ERR_INVALID_ARG and "NULL" in str(e.value)
    buf = np.zeros(64 * 64 + 8, np.uint16)
    base = buf.ctypes.data + 2  # 2 bytes off a 16-byte boundary
    with pytest.raises(rc.RcError) as e:
        op.run(s, [base, base, base])
    assert e.value.status == rc.ERR_INVALID_ARG and "aligned" in str(e.value)


def test_schedule_of_another_op_is_rejected():
    a = rc.Op(rc.OP_LINEAR, m=64, n=64, k=64)
    b = rc.Op(rc.OP_GEMM_F32, m=64, n=64, k=64)
    buf = np.zeros(64 * 64 * 4, np.float32)
    with pytest.raises(rc.RcError) as e:
        a.run(b.schedule(), [buf, buf, buf])
    assert e.value.status == rc.ERR_INVALID_ARG


def test_null_handles_give_status_codes():
    L = rc.lib()
    assert L.rc_op_info(None, None) == rc.ERR_INVALID_ARG
    assert L.rc_schedule_knobs(None, 0, None) == rc.ERR_INVALID_ARG
    assert L.rc_search_step(None, None, 0, None, 0, None) == rc.ERR_INVALID_ARG
    assert rc.lib().rc_last_error()


@pytest.mark.gpu
def test_bounded_wait_reports_timeout_and_context_survives():
    import torch
    st = rc.selftest_bounded_wait(50.0)
    assert st == rc.ERR_DEVICE_TIMEOUT, rc.STATUS_NAMES.get(st, st)
    # the context is still usable: a normal op runs and is correct afterwards
    A, B, bias = inputs.gemm_f32(64, 64, 64, seed=3)
    op = rc.Op(rc.OP_GEMM_F32, m=64, n=64, k=64, flags=rc.EPI_BIAS | rc.EPI_RELU)
    C = torch.empty(64, 64, dtype=torch.float32, device="cuda")
    op.run(op.schedule(), [torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda(), torch.from_numpy(bias).cuda(), C])
    op.check()
    ref = np.maximum(A.astype(np.float64) @ B + bias, 0)
    assert np.max(np.abs(C.cpu().numpy() - ref)) / np.max(np.abs(ref)) < 1e-4


@pytest.mark.gpu
def test_measurement_budget_times_out_remaining_candidates():
    import torch
    A, B, bias = inputs.gemm_f32(256, 256, 256, seed=0)
    op = rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256, flags=rc.EPI_BIAS | rc.EPI_RELU)
    io = [torch.from_numpy(A).cuda(), torch.from_numpy(B).cuda(), torch.from_numpy(bias).cuda(),
          torch.empty(256, 256, dtype=torch.float32, device="cuda")]
    scheds = [op.schedule(rc.T(rc.T_UNROLL, u)) for u in (1, 4)] * 4
    ms = op.measure(scheds, io, warmup=1, repeats=3, budget_s=1e-9)
    assert ms[-1].status == rc.ERR_TIMEOUT
