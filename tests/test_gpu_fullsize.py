"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times: the CPU oracle checks every token of the layer (the full
layer arithmetic in fp64, OpenMP over the host's cores), and the properties
that hold at any size (audit closed forms, G1, dispatch order) are checked on
every token too.  The tokens the routing gap rule excuses are counted and
reported in the end-of-run parity summary."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_06690_gb300 import inputs as inp
from paper_2608_06690_gb300.configs import CONFIGS
from pmpe_testlib import check_against_oracle, check_audit, check_dispatch, run_gpu_layer

pytestmark = pytest.mark.gpu


def _sample_tokens(cfg, per_pool=12, seed=0):
    """Tokens spread over the requests, both pools represented (for the
    backward checks, whose oracle cost grows with the tokens of nonzero dout)."""
    pol = cfg.policy(cfg.shape.T).numpy()
    tau = oracle.resolve(pol, cfg.shape.T)
    g = np.random.default_rng(seed)
    picks = []
    for want in (1, 0):
        cand = np.nonzero(tau == want)[0]
        if len(cand):
            picks.append(g.choice(cand, size=min(per_pool, len(cand)), replace=False))
    return np.sort(np.concatenate(picks)).astype(np.int32)


@pytest.mark.parametrize("name", ["qwen3_prefill", "deepseek_v2_lite", "qwen3_decode"])
def test_full_size_workload_every_token(name):
    cfg = CONFIGS[name]
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed, device="cuda", skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed, device="cuda", skew=cfg.skew)
    pol = cfg.policy(s.T)
    gpu = run_gpu_layer(s, w, h, pol.cuda())
    # properties on all tokens
    check_audit(s, pol, gpu)
    check_dispatch(s, h.cpu(), gpu)
    # the oracle on every token (full layer arithmetic in fp64)
    w_cpu = {k: (None if v is None else v.cpu()) for k, v in w.items()}
    rep = check_against_oracle(s, w_cpu, h.cpu(), pol, gpu, name=f"{name} (full size)")
    assert rep["tokens"] == s.T
    # near-ties are rare: about 1e-4 over the spacing of the k-th and
    # (k+1)-th of the pool's logits
    assert rep["excused"] <= max(2, s.T // 100), rep


@pytest.mark.parametrize("name", ["qwen3_prefill", "deepseek_v2_lite"])
def test_full_size_backward_on_sampled_tokens(name):
    """The private-branch backward at full size, launched as the benchmark
    launches it.  dout is nonzero on sampled ALLOW and DENY tokens only, so
    the oracle computes every gradient element exactly from those tokens
    (every gradient term is linear in a token's dout row); all four gradients
    are compared element by element.  G2 on all tokens: random upstream
    gradients on every DENY token change no gradient bit."""
    from paper_2608_06690_gb300 import pmpe
    from pmpe_testlib import GAP_EPS, oracle_layer
    cfg = CONFIGS[name]
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed, device="cuda", skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed, device="cuda", skew=cfg.skew)
    pol = cfg.policy(s.T)
    w_cpu = {k: (None if v is None else v.cpu()) for k, v in w.items()}
    L = oracle_layer(s, w_cpu, h.cpu(), pol)
    toks = _sample_tokens(cfg, per_pool=12, seed=1)
    _, _, gap = oracle.route(L, tokens=toks)
    keep = toks[gap >= GAP_EPS]  # a token at a routing near-tie may pick another k-th expert
    gen = torch.Generator().manual_seed(11)
    dout = torch.zeros((s.T, s.H), dtype=torch.bfloat16)
    dout[torch.from_numpy(keep).long()] = torch.randn((len(keep), s.H), generator=gen).to(torch.bfloat16)
    layer = pmpe.MoeLayer(s, w)
    pd = pol.cuda()
    layer.forward(h, pd)
    g = {n: v.cpu().numpy().astype(np.float64) for n, v in layer.backward_private(h, pd, dout.cuda()).items()}
    ref = oracle.backward_private(L, dout.double().numpy())
    tau = oracle.resolve(pol.numpy(), s.T)
    assert tau[keep].sum() >= 8 and (tau[keep] == 0).sum() >= 8
    for n in ("d_router", "d_gate", "d_up", "d_down"):
        err = np.abs(g[n] - ref[n])
        mx = err.max() / np.abs(ref[n]).max()
        mean = err.sum() / np.abs(ref[n]).sum()
        assert mx <= 2e-2 and mean <= 1e-2, (n, mx, mean)
        # the same experts receive gradients (an expert no sampled row reached gets exact zeros)
        assert np.array_equal(np.abs(g[n]).reshape(s.E_priv, -1).max(1) == 0,
                              np.abs(ref[n]).reshape(s.E_priv, -1).max(1) == 0), n
    # G2 at full size: DENY rows of dout reach no private gradient
    d2 = dout.clone()
    deny = torch.from_numpy(tau == 0)
    d2[deny] = torch.randn((int(deny.sum()), s.H), generator=gen).to(torch.bfloat16)
    layer.forward(h, pd)
    g2 = layer.backward_private(h, pd, d2.cuda())
    for n in g:
        assert np.array_equal(g[n], g2[n].cpu().numpy().astype(np.float64)), n


@pytest.mark.parametrize("name", ["qwen3_prefill", "deepseek_v2_lite"])
def test_full_size_input_gradient_on_sampled_tokens(name):
    """The gradient of the layer's input at full size, launched as the
    benchmark launches it.  dout is nonzero on sampled ALLOW and DENY tokens
    only: the oracle computes their rows, which are compared element by
    element; every other row is exactly zero (each term is linear in the
    token's own dout row).  A second run is bitwise identical."""
    from paper_2608_06690_gb300 import pmpe
    from pmpe_testlib import GAP_EPS, oracle_layer
    cfg = CONFIGS[name]
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed, device="cuda", skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed, device="cuda", skew=cfg.skew)
    pol = cfg.policy(s.T)
    w_cpu = {k: (None if v is None else v.cpu()) for k, v in w.items()}
    L = oracle_layer(s, w_cpu, h.cpu(), pol)
    toks = _sample_tokens(cfg, per_pool=12, seed=2)
    _, _, gap = oracle.route(L, tokens=toks)
    keep = toks[gap >= GAP_EPS]
    gen = torch.Generator().manual_seed(12)
    dout = torch.zeros((s.T, s.H), dtype=torch.bfloat16)
    dout[torch.from_numpy(keep).long()] = torch.randn((len(keep), s.H), generator=gen).to(torch.bfloat16)
    layer = pmpe.MoeLayer(s, w)
    pd = pol.cuda()
    layer.forward(h, pd)
    dh = layer.backward_input(h, pd, dout.cuda())
    got = dh.cpu().numpy().astype(np.float64)
    ref = oracle.backward_input(L, dout.double().numpy())
    tau = oracle.resolve(pol.numpy(), s.T)
    assert tau[keep].sum() >= 8 and (tau[keep] == 0).sum() >= 8
    err = np.abs(got[keep] - ref[keep])
    assert err.max() / np.abs(ref[keep]).max() <= 2e-2 and err.sum() / np.abs(ref[keep]).sum() <= 1e-2
    rest = np.ones(s.T, bool)
    rest[keep] = False
    assert np.all(got[rest] == 0.0)
    layer.forward(h, pd)
    assert torch.equal(dh, layer.backward_input(h, pd, dout.cuda()))


@pytest.mark.parametrize("name", ["qwen3_prefill", "deepseek_v2_lite"])
def test_full_size_input_gradient_of_deny_tokens_ignores_private_weights(name):
    """G2 through the input gradient at full size: every private weight
    (router, gate, up, down) replaced by other random values leaves the DENY
    tokens' rows of d_hidden bitwise unchanged, while the ALLOW rows change."""
    from paper_2608_06690_gb300 import pmpe
    cfg = CONFIGS[name]
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed, device="cuda", skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed, device="cuda", skew=cfg.skew)
    pd = cfg.policy(s.T).cuda()
    tau = torch.from_numpy(oracle.resolve(cfg.policy(s.T).numpy(), s.T).astype(bool)).cuda()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(13)
    dout = torch.randn((s.T, s.H), generator=gen, device="cuda").to(torch.bfloat16)
    layer = pmpe.MoeLayer(s, w)
    layer.forward(h, pd)
    dh1 = layer.backward_input(h, pd, dout).clone()
    w2 = dict(w)
    for n in ("router_priv", "gate_priv", "up_priv", "down_priv"):
        w2[n] = (torch.randn(w[n].shape, generator=gen, device="cuda") * 0.02).to(torch.bfloat16)
    layer2 = pmpe.MoeLayer(s, w2)
    layer2.forward(h, pd)
    dh2 = layer2.backward_input(h, pd, dout)
    torch.cuda.synchronize()
    assert torch.equal(dh1[~tau], dh2[~tau])
    assert not torch.equal(dh1[tau], dh2[tau])
