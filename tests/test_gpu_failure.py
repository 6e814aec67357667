"""Failure detection on the device, without a fault: every barrier wait in
the layer's pipelined kernels is bounded, and an expired wait records
PMPE_STATUS_PIPELINE_TIMEOUT in the audit status word and returns.  The
self-test entry point makes such a wait expire (a barrier nothing arrives on,
with a short limit); the host then reads the status, sees the error reported
through pmpe_audit_read, and the same CUDA context runs the layer correctly
afterwards."""
import time

import numpy as np
import pytest
import torch

from paper_2608_06690_gb300.configs import CONFIGS
from pmpe_testlib import check_against_oracle, check_audit, make_layer, run_gpu_layer, to_device

pytestmark = pytest.mark.gpu


def test_expired_wait_is_reported_and_the_context_stays_usable():
    from paper_2608_06690_gb300 import pmpe
    s = CONFIGS["tiny"].shape
    T, E = s.T, s.E
    audit = torch.zeros(pmpe.audit_words(T, E), dtype=torch.int32, device="cuda")
    limit_us = 20000
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    pmpe.selftest_wait_timeout(audit, limit_us)
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert elapsed >= limit_us * 1e-6, elapsed          # the wait really waited ...
    assert elapsed < 5.0, elapsed                       # ... and then gave up
    words = pmpe.audit_read(audit, T, E, check_status=False)
    assert words["status"] == pmpe.STATUS_PIPELINE_TIMEOUT
    assert words["shared_rows"] == 0 and not words["route_count"].any()
    with pytest.raises(pmpe.PmpeError) as e:
        pmpe.audit_read(audit, T, E)
    assert e.value.code == pmpe.ERR_DEVICE_STATUS
    # the context survives: the layer still runs and matches the oracle
    w, h, pol = make_layer(s, seed=5, policy="iid")
    wd, hd, pd = to_device(w, h, pol)
    gpu = run_gpu_layer(s, wd, hd, pd)
    assert gpu["audit"]["status"] == 0
    check_audit(s, pol, gpu)
    check_against_oracle(s, w, h, pol, gpu)


def test_reset_clears_a_recorded_timeout():
    from paper_2608_06690_gb300 import pmpe
    T, E = 4, 6
    audit = torch.zeros(pmpe.audit_words(T, E), dtype=torch.int32, device="cuda")
    pmpe.selftest_wait_timeout(audit, 1000)
    pmpe.selftest_wait_timeout(audit, 1000)   # ORs, does not add
    assert pmpe.audit_read(audit, T, E, check_status=False)["status"] == pmpe.STATUS_PIPELINE_TIMEOUT
    pmpe.audit_reset(audit, T, E)
    a = pmpe.audit_read(audit, T, E)
    assert a["status"] == 0 and np.all(a["exec_rows"] == 0)
