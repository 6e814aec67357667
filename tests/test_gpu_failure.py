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


def test_dispatch_mismatch_is_caught_by_the_execution_audit():
    """The execution audit counts what the expert tiles ran, checked against
    the route log row by row (Sec. 5.2, App. F.1: counts observed at the
    experts, independent of the router).  A dispatch corrupted on the host --
    a private expert's slot handed to a DENY token, every index still valid --
    makes the gate/up tiles run that token's row through the private expert;
    the audit shows it as exec != route for that expert and for both tokens,
    and as the dispatch-mismatch status bit, which pmpe_audit_read reports."""
    from paper_2608_06690_gb300 import pmpe
    from paper_2608_06690_gb300.inputs import LayerShape
    s = LayerShape(T=256, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True)
    w, h, pol = make_layer(s, seed=9, policy="iid")
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(s, wd)
    T, E, k = s.T, s.E, s.k
    audit = torch.zeros(pmpe.audit_words(T, E), dtype=torch.int32, device="cuda")
    idx = torch.empty((T, k), dtype=torch.int32, device="cuda")
    out = torch.empty_like(hd)
    layer.forward(hd, pd, out=out, topk_idx=idx, audit=audit, stages=pmpe.STAGE_ROUTE | pmpe.STAGE_PERMUTE)
    torch.cuda.synchronize()
    ws = layer.workspace(T)
    L = pmpe.workspace_layout(s)
    offsets = ws[L["offsets"]:L["offsets"] + 4 * (E + 1)].view(torch.int32).cpu().numpy()
    tos = ws[L["tok_of_slot"]:L["tok_of_slot"] + 4 * T * k].view(torch.int32)
    tau = (pol.numpy() == 1)
    e = next(e for e in range(s.E_pub, E) if offsets[e + 1] > offsets[e])   # a private expert with rows
    slot = int(offsets[e])
    t_orig = int(tos[slot].item())
    t_deny = int(np.nonzero(~tau)[0][0])
    tos[slot] = t_deny                     # host-side corruption of one dispatch entry
    torch.cuda.synchronize()
    # the gate/up tiles gather the rows named by tok_of_slot and count them
    layer.forward(hd, pd, out=out, topk_idx=idx, audit=audit, stages=pmpe.STAGE_GATEUP)
    torch.cuda.synchronize()
    with pytest.raises(pmpe.PmpeError) as err:
        pmpe.audit_read(audit, T, E)
    assert err.value.code == pmpe.ERR_DEVICE_STATUS
    a = pmpe.audit_read(audit, T, E, check_status=False)
    assert a["status"] & pmpe.STATUS_DISPATCH_MISMATCH
    assert a["exec_rows"][e] == a["route_count"][e] - 1
    others = np.arange(E) != e
    assert np.array_equal(a["exec_rows"][others], a["route_count"][others])
    assert a["route_priv_rows"][t_deny] == 0 and a["exec_priv_rows"][t_deny] == 1
    assert a["exec_priv_rows"][t_orig] == a["route_priv_rows"][t_orig] - 1
    # the uncorrupted forward is clean again
    pmpe.audit_reset(audit, T, E)
    layer.forward(hd, pd, out=out, topk_idx=idx, audit=audit)
    a = pmpe.audit_read(audit, T, E)
    assert a["status"] == 0 and np.array_equal(a["exec_rows"], a["route_count"])
