"""GPU parity of the private-branch backward (G2, Sec. 2.2; Sec. 3.2 trains
the private experts and the private router only) against the oracle's
backward_private, through the C ABI, on seeded inputs: renormalised top-k and
pool softmax, ragged expert row counts spanning several 128-row tiles, private
experts without rows, the all-DENY and empty batches."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_06690_gb300 import pmpe
from paper_2608_06690_gb300.inputs import LayerShape
from pmpe_testlib import GAP_EPS, make_layer, oracle_layer, to_device

pytestmark = pytest.mark.gpu

# Gradient tolerance: per tensor, max-abs error <= 2e-2 * max|ref| and
# sum|err| / sum|ref| <= 1e-2.  The GPU contracts BF16 operands with FP32
# accumulation and rounds three intermediates to BF16 (the SwiGLU input
# gradients dG, dU and the weighted activation w * act: 2^-9 relative each),
# which the weight gradients then sum over an expert's rows.
MAX_ABS_REL = 2e-2
MEAN_REL = 1e-2

GRADS = ("d_router", "d_gate", "d_up", "d_down")

CASES = {
    "renorm_ragged": (LayerShape(T=300, H=384, I=256, E_pub=24, E_priv=8, E_sh=0, k=4, renormalize=True), 51,
                      "iid"),
    "pool_softmax_with_shared": (LayerShape(T=200, H=256, I=256, E_pub=16, E_priv=8, E_sh=2, k=3,
                                            renormalize=False), 52, "iid"),
    # every token ALLOW, 4 private experts: ~250 rows each, two 128-row M tiles
    "all_allow_multi_tile": (LayerShape(T=500, H=256, I=128, E_pub=8, E_priv=4, E_sh=0, k=2, renormalize=True),
                             53, "allow"),
    # 64 private experts for ~45 ALLOW tokens x 2 picks: many experts without rows
    "sparse_pool_empty_experts": (LayerShape(T=90, H=128, I=128, E_pub=8, E_priv=64, E_sh=0, k=2,
                                             renormalize=True), 54, "iid"),
    "k12_pool_softmax": (LayerShape(T=150, H=256, I=128, E_pub=40, E_priv=16, E_sh=0, k=12, renormalize=False), 55,
                         "iid"),
    "k1": (LayerShape(T=100, H=128, I=128, E_pub=12, E_priv=5, E_sh=0, k=1, renormalize=True), 56, "iid"),
    "single_token": (LayerShape(T=1, H=256, I=128, E_pub=8, E_priv=4, E_sh=1, k=2, renormalize=False), 57, "allow"),
}


def _dout(shape: LayerShape, seed: int) -> torch.Tensor:
    g = torch.Generator().manual_seed(seed)
    return torch.randn((shape.T, shape.H), generator=g).to(torch.bfloat16)


def _gpu_backward(shape, w, h, pol, dout):
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    idx = torch.empty((shape.T, shape.k), dtype=torch.int32, device="cuda")
    wt = torch.empty((shape.T, shape.k), dtype=torch.float32, device="cuda")
    layer.forward(hd, pd, topk_idx=idx, topk_w=wt)
    g = layer.backward_private(hd, pd, dout.cuda().contiguous(), topk_idx=idx, topk_w=wt)
    torch.cuda.synchronize()
    return {n: v.cpu().numpy().astype(np.float64) for n, v in g.items()}, idx.cpu().numpy(), layer, (wd, hd, pd)


def _errors(got, ref):
    err = np.abs(got - ref)
    return float(err.max() / max(np.abs(ref).max(), 1e-30)), float(err.sum() / max(np.abs(ref).sum(), 1e-30))


@pytest.mark.parametrize("name", list(CASES))
def test_backward_parity_with_oracle(name):
    shape, seed, policy = CASES[name]
    w, h, pol = make_layer(shape, seed, policy=policy)
    L = oracle_layer(shape, w, h, pol)
    oidx, _, gap = oracle.route(L)
    dout = _dout(shape, seed)
    # a token whose k-th and (k+1)-th logits are closer than the gap rule may
    # route differently on the GPU; its gradient contributions are linear in
    # its dout row, so that row is zeroed on both sides
    dout[torch.from_numpy(gap < GAP_EPS)] = 0
    got, gidx, _, _ = _gpu_backward(shape, w, h, pol, dout)
    ok = gap >= GAP_EPS
    assert np.array_equal(gidx[ok], oidx[ok])
    ref = oracle.backward_private(L, dout.double().numpy())
    tau = oracle.resolve(None if pol is None else pol.numpy(), shape.T)
    for n in GRADS:
        if tau.sum() == 0 or not np.any(ref[n]):
            assert np.all(got[n] == 0.0), n
            continue
        mx, mean = _errors(got[n], ref[n])
        assert mx <= MAX_ABS_REL and mean <= MEAN_REL, (n, mx, mean)
    # experts without rows get exactly zero weight gradients
    rows = np.bincount(gidx[tau == 1].reshape(-1) - shape.E_pub, minlength=shape.E_priv) if tau.any() else \
        np.zeros(shape.E_priv, int)
    for q in np.flatnonzero(rows == 0):
        for n in ("d_gate", "d_up", "d_down"):
            assert np.all(got[n][q] == 0.0), (n, q)
    # Sec. 3.2: every expert that receives routing events receives nonzero,
    # finite gradients
    for n in GRADS:
        assert np.all(np.isfinite(got[n])), n
    for q in np.flatnonzero(rows > 0):
        for n in ("d_gate", "d_up", "d_down"):
            assert np.any(got[n][q] != 0.0), (n, q)


def test_backward_all_deny_and_empty_batch_give_zero_gradients():
    for T, policy in ((130, "deny"), (0, "deny")):
        shape = LayerShape(T=T, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True)
        w, h, pol = make_layer(shape, 58, policy=policy)
        got, _, _, _ = _gpu_backward(shape, w, h, pol, _dout(shape, 58))
        for n in GRADS:
            assert got[n].shape[0] == shape.E_priv
            assert np.all(got[n] == 0.0), (T, n)


def test_backward_g2_deny_rows_never_reach_private_gradients_and_is_deterministic():
    """G2 on the GPU: changing the upstream gradient of DENY tokens leaves the
    private gradients bitwise unchanged; a second run is bitwise identical
    (no atomics in the backward); the public weights are not written."""
    shape, seed, _ = CASES["renorm_ragged"]
    w, h, pol = make_layer(shape, seed, policy="iid")
    tau = oracle.resolve(pol.numpy(), shape.T)
    d1 = _dout(shape, 1)
    d2 = d1.clone()
    d2[torch.from_numpy(tau == 0)] = _dout(shape, 2)[torch.from_numpy(tau == 0)]
    g1, _, layer, (wd, hd, pd) = _gpu_backward(shape, w, h, pol, d1)
    before = {n: wd[n].clone() for n in wd if wd[n] is not None and not n.endswith("priv")}
    g2 = layer.backward_private(hd, pd, d2.cuda())
    g3 = layer.backward_private(hd, pd, d1.cuda())
    torch.cuda.synchronize()
    for n in GRADS:
        assert np.array_equal(g1[n], g2[n].cpu().numpy().astype(np.float64)), n
        assert np.array_equal(g1[n], g3[n].cpu().numpy().astype(np.float64)), n
    for n, v in before.items():
        assert torch.equal(v, wd[n]), n
    # the router gradient of a softmax sums to zero over the pool
    r = g1["d_router"]
    assert np.abs(r.sum(0)).max() <= 1e-3 * np.abs(r).max()


def test_backward_rejects_the_unmasked_control_and_a_short_workspace():
    shape = LayerShape(T=64, H=128, I=128, E_pub=8, E_priv=4, E_sh=0, k=2, renormalize=True)
    w, h, pol = make_layer(shape, 59, policy="iid")
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    out = layer.forward(hd, pd)
    dout = _dout(shape, 59).cuda()
    g = {n: torch.empty(1 << 20, dtype=torch.float32, device="cuda") for n in GRADS}
    nb = pmpe._lib.pmpe_moe_backward_workspace_size(shape.T, shape.H, shape.I, shape.E_pub, shape.E_priv,
                                                      shape.E_sh, shape.k)
    assert nb > 0
    bws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    args = [pmpe._ptr(dout)] + [pmpe._ptr(g[n]) for n in GRADS]
    desc = pmpe.make_desc(shape, wd, hd, pd, out, layer.workspace(shape.T), unmasked_control=True)
    rc = pmpe._lib.pmpe_moe_backward_private(pmpe.ctypes.byref(desc), *args, pmpe._ptr(bws), nb,
                                             pmpe._stream(None))
    assert rc == pmpe.ERR_UNSUPPORTED_SHAPE
    desc = pmpe.make_desc(shape, wd, hd, pd, out, layer.workspace(shape.T))
    rc = pmpe._lib.pmpe_moe_backward_private(pmpe.ctypes.byref(desc), *args, pmpe._ptr(bws), nb - 256,
                                             pmpe._stream(None))
    assert rc == pmpe.ERR_WORKSPACE
    torch.cuda.synchronize()
