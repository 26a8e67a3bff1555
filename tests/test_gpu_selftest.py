"""Failure detection without a GPU fault: a bounded barrier wait that nothing
completes gives up after its limit, records the timeout for the host, and the
context stays usable for the next call."""

import time

import numpy as np
import pytest
import torch

import workload as wl
from helpers import accepted_random, compare_condense, oracle_run

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wz():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_23265_gb300.wavezip as m
    assert torch.cuda.is_available()
    return m


def test_bounded_wait_times_out_and_reports(wz):
    timeout_ns = 20_000_000                        # 20 ms
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    status = wz.wz_selftest_bounded_wait(timeout_ns)
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert int(status.item()) & wz.STATUS_WAIT_TIMEOUT
    assert elapsed >= 0.9 * timeout_ns * 1e-9


def test_context_usable_after_a_timeout(wz):
    status = wz.wz_selftest_bounded_wait(1_000_000)
    torch.cuda.synchronize()
    assert int(status.item()) == wz.STATUS_WAIT_TIMEOUT
    X, Q = accepted_random(6, 9, 9, 64, 3, 0.3, seed=8)
    out = wz.wz_condense_ex(X.cuda(), Q.cuda(), 0.3)
    torch.cuda.synchronize()
    compare_condense(out, oracle_run(X, Q, 0.3), X.dtype)


def test_selftest_argument_errors(wz):
    st = torch.zeros((1,), dtype=torch.int32, device="cuda")
    for bad in (0, 2_000_000_000):
        with pytest.raises(wz.WaveZipError):
            wz.wz_selftest_bounded_wait(bad, st)
    assert wz._lib.wz_selftest_bounded_wait(1000, None, None) == wz.ERR_INVALID_ARG
