"""The paper's soft-router control on the GPU (Sec. 4.2 and App. E, the
control matrix's soft-router-only arm): routing over the concatenated public/private pool without the hard mask.
It is a negative control, not the method.  The GPU matches the oracle run
with the same control, private rows execute for DENY tokens (the audit
records them, route log and execution count agreeing), and the method run
on the same layer right afterwards is fail-closed again."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_06690_gb300.configs import CONFIGS
from paper_2608_06690_gb300.inputs import LayerShape
from pmpe_testlib import GAP_EPS, MAX_ABS_REL, MEAN_REL, check_audit, make_layer, oracle_layer, output_errors, \
    run_gpu_layer, to_device

pytestmark = pytest.mark.gpu

CASES = {
    "tiny_config_two_lists": (CONFIGS["tiny"].shape, 50),
    "ragged_three_lists": (LayerShape(T=300, H=256, I=128, E_pub=40, E_priv=16, E_sh=0, k=4, renormalize=True), 51),
    "shared_pool_softmax": (LayerShape(T=200, H=256, I=256, E_pub=16, E_priv=8, E_sh=2, k=3, renormalize=False), 52),
    "wide_pools_k6": (LayerShape(T=130, H=128, I=128, E_pub=96, E_priv=64, E_sh=0, k=6, renormalize=True), 53),
}


def _run_control(shape, w, h, pol):
    from paper_2608_06690_gb300 import pmpe
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    T, k, E = shape.T, shape.k, shape.E
    idx = torch.full((T, k), -1, dtype=torch.int32, device="cuda")
    wt = torch.zeros((T, k), dtype=torch.float32, device="cuda")
    audit = torch.zeros(pmpe.audit_words(T, E), dtype=torch.int32, device="cuda")
    out = layer.forward(hd, pd, topk_idx=idx, topk_w=wt, audit=audit, unmasked_control=True)
    torch.cuda.synchronize()
    a = pmpe.audit_read(audit, T, E)
    return layer, (hd, pd), dict(out=out.view(torch.int16).cpu().numpy().view(np.uint16), idx=idx.cpu().numpy(),
                                w=wt.cpu().numpy(), audit=a)


@pytest.mark.parametrize("name", list(CASES))
def test_control_matches_unmasked_oracle(name):
    shape, seed = CASES[name]
    w, h, pol = make_layer(shape, seed)
    _, _, g = _run_control(shape, w, h, pol)
    r = oracle.forward(oracle_layer(shape, w, h, pol, unmasked=True))
    ok = r["gap"] >= GAP_EPS
    assert np.all((g["idx"] >= 0) & (g["idx"] < shape.E))
    assert np.array_equal(g["idx"][ok], r["idx"][ok])
    np.testing.assert_allclose(g["w"][ok], r["w"][ok], rtol=0, atol=2e-5)
    mx, mean = output_errors(g["out"][ok], r["out"][ok])
    assert mx <= MAX_ABS_REL and mean <= MEAN_REL, (mx, mean)
    a = g["audit"]
    hist = np.bincount(g["idx"].reshape(-1), minlength=shape.E)
    assert np.array_equal(a["route_count"], hist)
    assert np.array_equal(a["exec_rows"], a["route_count"])
    assert np.array_equal(a["route_priv_rows"], (g["idx"] >= shape.E_pub).sum(1))
    assert np.array_equal(a["exec_priv_rows"], a["route_priv_rows"])
    assert a["shared_rows"] == shape.T * shape.E_sh


def test_control_runs_private_rows_for_deny_tokens_and_the_method_recovers():
    """The negative control: under the control, DENY tokens execute private
    rows; the method on the same layer, workspace and inputs executes none."""
    shape, seed = CASES["ragged_three_lists"]
    w, h, pol = make_layer(shape, seed)
    layer, (hd, pd), g = _run_control(shape, w, h, pol)
    tau = oracle.resolve(pol.numpy(), shape.T)
    assert g["audit"]["exec_priv_rows"][tau == 0].sum() > 0
    wd = layer.weights
    gm = run_gpu_layer(shape, wd, hd, pd)
    check_audit(shape, pol, gm)
    assert gm["audit"]["exec_priv_rows"][tau == 0].sum() == 0


def test_control_rejects_shapes_whose_merge_does_not_fit():
    """Pools of 8 + 8 chunks with k = 8 exceed the control's merge limit
    (chunks * k <= 96): rejected before any launch, output untouched."""
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=8, H=128, I=128, E_pub=256, E_priv=256, E_sh=0, k=8, renormalize=True)
    w, h, pol = make_layer(shape, 54)
    wd, hd, pd = to_device(w, h, pol)
    out = torch.full_like(hd, 7.0)
    ws = torch.empty(pmpe.workspace_size(shape), dtype=torch.uint8, device="cuda")
    d = pmpe.make_desc(shape, wd, hd, pd, out, ws, unmasked_control=True)
    import ctypes
    assert pmpe._lib.pmpe_moe_forward(ctypes.byref(d), None) == pmpe.ERR_UNSUPPORTED_SHAPE
    torch.cuda.synchronize()
    assert torch.all(out == 7.0)
