"""The no-allocation routing entry point (rc_moe_route_noalloc).

It is meant for callers that cannot allocate device memory, such as a process
whose GPU memory is reserved by another allocator's pool, or a path where
cudaMalloc (which can synchronise the device) is not allowed. It must give
the same routing as the regular rc_run path: identical ids, offsets and
permutation, and weights within the routing tests' tolerance. Two calls in a
row, with different shapes, check that the shared fixed scratch carries
nothing over from one call to the next. The file sorts last so that a run
stopping at its first failure has already run every other test.
"""
import numpy as np
import pytest

import oracle
from paper_2506_01374_gb300 import inputs, rc

from .gpu_util import to_dev, torch

pytestmark = pytest.mark.gpu


def _buffers(T, E, K):
    return (torch.empty(T, K, dtype=torch.int32, device="cuda"), torch.empty(T, K, dtype=torch.float32, device="cuda"),
            torch.empty(E + 1, dtype=torch.int32, device="cuda"), torch.empty(T * K, dtype=torch.int32, device="cuda"))


def _host(bufs):
    return [b.cpu().numpy() for b in bufs]


def test_noalloc_routing_matches_regular_entry_point_two_calls():
    for T, E, K, fp32, seed in [(4096, 64, 8, False, 51), (777, 200, 6, True, 52)]:
        logits, _, _, _ = inputs.moe(T, 8, E, 8, seed=seed, logits_fp32=fp32)
        dl = to_dev(logits)
        op = rc.Op(rc.OP_MOE_ROUTE, tokens=T, experts=E, top_k=K, logits_fp32=int(fp32), renorm=1)
        regular = _buffers(T, E, K)
        op.run(op.schedule(), [dl, *regular])
        op.check()
        noalloc = _buffers(T, E, K)
        rc.moe_route_noalloc(dl, T, E, K, *noalloc, renorm=True, logits_fp32=fp32)
        torch.cuda.synchronize()
        r_ids, r_w, r_off, r_perm = _host(regular)
        n_ids, n_w, n_off, n_perm = _host(noalloc)
        np.testing.assert_array_equal(n_ids, r_ids)
        np.testing.assert_array_equal(n_off, r_off)
        np.testing.assert_array_equal(n_perm, r_perm)
        np.testing.assert_allclose(n_w, r_w, rtol=2e-6, atol=1e-7)
        assert n_off[-1] == T * K
        # and against the fp64 oracle's routing, so the check does not rest on the shared kernels alone
        o_ids, o_w, o_off, o_perm = oracle.moe_route(logits, K)
        np.testing.assert_array_equal(n_ids, o_ids)
        np.testing.assert_array_equal(n_off, o_off)
        np.testing.assert_array_equal(n_perm, o_perm)
        np.testing.assert_allclose(n_w, o_w, rtol=2e-6, atol=1e-7)


def test_noalloc_routing_rejects_too_many_experts():
    T, E, K = 16, 257, 4
    logits = torch.zeros(T, E, dtype=torch.int16, device="cuda")
    bufs = _buffers(T, E, K)
    with pytest.raises(rc.RcError) as e:
        rc.moe_route_noalloc(logits, T, E, K, *bufs)
    assert e.value.status == rc.ERR_INVALID_ARG and "exceeds" in str(e.value)
