"""The combined backward (the private-parameter gradients and the input
gradient in one pass, for a training step of the layer, Sec. 3.2) through the
C ABI: every output bitwise the one the two separate backward calls give --
which the parity tests of those calls tie to the oracle -- on shapes with both
pools, renormalised top-k and pool softmax, shared experts, experts without
rows, one token and the empty batch, and at the workloads' full sizes.  And
the training mode: a forward that saves its gate/up accumulators gives the
same output, and all three backward calls reading them give bitwise the
recomputation's results."""
import numpy as np
import pytest
import torch

from paper_2608_06690_gb300 import inputs as inp
from paper_2608_06690_gb300 import pmpe
from paper_2608_06690_gb300.configs import CONFIGS
from paper_2608_06690_gb300.inputs import LayerShape
from pmpe_testlib import make_layer, to_device

pytestmark = pytest.mark.gpu

GRADS = ("d_router", "d_gate", "d_up", "d_down")

CASES = {
    "renorm_ragged": (LayerShape(T=300, H=384, I=256, E_pub=24, E_priv=8, E_sh=0, k=4, renormalize=True), 81, "iid"),
    "pool_softmax_with_shared": (LayerShape(T=200, H=256, I=256, E_pub=16, E_priv=8, E_sh=2, k=3,
                                            renormalize=False), 82, "iid"),
    "all_allow_multi_tile": (LayerShape(T=500, H=256, I=128, E_pub=8, E_priv=4, E_sh=0, k=2, renormalize=True),
                             83, "allow"),
    "all_deny": (LayerShape(T=260, H=256, I=128, E_pub=8, E_priv=4, E_sh=1, k=2, renormalize=True), 84, "deny"),
    "sparse_pool_empty_experts": (LayerShape(T=90, H=128, I=128, E_pub=8, E_priv=64, E_sh=0, k=2,
                                             renormalize=True), 85, "iid"),
    "k12_pool_softmax": (LayerShape(T=150, H=256, I=128, E_pub=40, E_priv=16, E_sh=0, k=12, renormalize=False), 86,
                         "iid"),
    "single_token": (LayerShape(T=1, H=256, I=128, E_pub=8, E_priv=4, E_sh=1, k=2, renormalize=False), 87, "allow"),
}


def _dout(shape, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randn((shape.T, shape.H), generator=g).to(torch.bfloat16).cuda()


def _separate_and_combined(layer, h, pol, dout):
    layer.forward(h, pol)
    g_sep = {n: v.clone() for n, v in layer.backward_private(h, pol, dout).items()}
    dh_sep = layer.backward_input(h, pol, dout).clone()
    g, dh = layer.backward(h, pol, dout)
    torch.cuda.synchronize()
    return g_sep, dh_sep, g, dh


@pytest.mark.parametrize("name", list(CASES))
def test_combined_backward_is_bitwise_the_two_separate_passes(name):
    shape, seed, policy = CASES[name]
    w, h, pol = make_layer(shape, seed, policy=policy)
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    g_sep, dh_sep, g, dh = _separate_and_combined(layer, hd, pd, _dout(shape, seed))
    for n in GRADS:
        assert torch.equal(g[n], g_sep[n]), n
    assert torch.equal(dh, dh_sep)
    assert torch.all(torch.isfinite(dh))


def test_combined_backward_empty_batch():
    shape = LayerShape(T=0, H=256, I=128, E_pub=16, E_priv=8, E_sh=1, k=2, renormalize=True)
    w, h, pol = make_layer(shape, 88, policy="iid")
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    layer.forward(hd, pd)
    g, dh = layer.backward(hd, pd, torch.empty((0, shape.H), dtype=torch.bfloat16, device="cuda"))
    torch.cuda.synchronize()
    assert dh.shape == (0, shape.H)
    for n in GRADS:
        assert g[n].shape[0] == shape.E_priv and torch.all(g[n] == 0), n


@pytest.mark.parametrize("name", ["qwen3_prefill", "deepseek_v2_lite"])
def test_full_size_combined_backward_is_bitwise_the_two_separate_passes(name):
    cfg = CONFIGS[name]
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed, device="cuda", skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed, device="cuda", skew=cfg.skew)
    pd = cfg.policy(s.T).cuda()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(17)
    dout = torch.randn((s.T, s.H), generator=gen, device="cuda").to(torch.bfloat16)
    layer = pmpe.MoeLayer(s, w)
    g_sep, dh_sep, g, dh = _separate_and_combined(layer, h, pd, dout)
    for n in GRADS:
        assert torch.equal(g[n], g_sep[n]), n
    assert torch.equal(dh, dh_sep)


def _all_three(layer, h, pol, dout, save):
    out = layer.forward(h, pol, save_for_backward=save).clone()
    gp = {n: v.clone() for n, v in layer.backward_private(h, pol, dout).items()}
    di = layer.backward_input(h, pol, dout).clone()
    g, dh = layer.backward(h, pol, dout)
    torch.cuda.synchronize()
    return out, gp, di, g, dh


@pytest.mark.parametrize("name", ["renorm_ragged", "pool_softmax_with_shared", "sparse_pool_empty_experts",
                                  "single_token"])
def test_saved_gate_up_accumulators_give_bitwise_the_recomputed_backward(name):
    """A forward that saves its gate/up accumulators G | U gives the same
    output, and every backward call that reads them instead of recomputing
    the gate/up GEMM gives bitwise the recomputation's results."""
    shape, seed, policy = CASES[name]
    w, h, pol = make_layer(shape, seed, policy=policy)
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    dout = _dout(shape, seed + 1)
    ref = _all_three(layer, hd, pd, dout, save=False)
    got = _all_three(layer, hd, pd, dout, save=True)
    assert torch.equal(got[0].view(torch.int16), ref[0].view(torch.int16))
    for i in (1, 3):
        for n in GRADS:
            assert torch.equal(got[i][n], ref[i][n]), (i, n)
    assert torch.equal(got[2], ref[2]) and torch.equal(got[4], ref[4])
    # the buffer holds G | U of every dispatch row (some value written everywhere)
    R = shape.T * shape.k
    sg = layer._saved_buf[:R * 2 * shape.I].view(R, 2 * shape.I)
    assert torch.all(torch.isfinite(sg))


@pytest.mark.parametrize("name", ["qwen3_prefill", "deepseek_v2_lite"])
def test_full_size_saved_gate_up_accumulators_give_bitwise_the_recomputed_backward(name):
    cfg = CONFIGS[name]
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed, device="cuda", skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed, device="cuda", skew=cfg.skew)
    pd = cfg.policy(s.T).cuda()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(19)
    dout = torch.randn((s.T, s.H), generator=gen, device="cuda").to(torch.bfloat16)
    layer = pmpe.MoeLayer(s, w)
    ref = _all_three(layer, h, pd, dout, save=False)
    got = _all_three(layer, h, pd, dout, save=True)
    assert torch.equal(got[0].view(torch.int16), ref[0].view(torch.int16))
    for i in (1, 3):
        for n in GRADS:
            assert torch.equal(got[i][n], ref[i][n]), (i, n)
    assert torch.equal(got[2], ref[2]) and torch.equal(got[4], ref[4])
