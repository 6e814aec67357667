"""A 48-layer decode-shaped stack (64 requests of one token, alternating
ALLOW / DENY, residual add between layers) captured into one CUDA graph:
replaying the graph gives bit for bit the result of running the layers one
call at a time, twice in a row, and the audit counters accumulated inside
the graph satisfy the per-token closed form 48 * k * tau (Sec. 2.2, G1)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_06690_gb300 import inputs as inp
from paper_2608_06690_gb300 import pmpe
from paper_2608_06690_gb300.inputs import LayerShape

pytestmark = pytest.mark.gpu

N_LAYERS = 48
SHAPE = LayerShape(T=64, H=1024, I=256, E_pub=64, E_priv=16, E_sh=0, k=8, renormalize=True)


def _stack(layers, x_in, pol, x_out, audit):
    x = x_in
    out = torch.empty_like(x_in)
    for layer in layers:
        layer.forward(x, pol, out=out, audit=audit)
        x = (x.float() + out.float()).to(torch.bfloat16)
    x_out.copy_(x)


def test_48_layer_stack_replays_bitwise_from_a_cuda_graph():
    s = SHAPE
    ws = pmpe.Workspace("cuda")
    layers = [pmpe.MoeLayer(s, inp.make_weights(s, 7000 + l, device="cuda"), workspace=ws) for l in range(N_LAYERS)]
    x0 = inp.make_hidden(s, 7, device="cuda")
    pol = torch.tensor([1 if t % 2 == 0 else 0 for t in range(s.T)], dtype=torch.uint8, device="cuda")
    E = s.E
    audit_e = torch.zeros(pmpe.audit_words(s.T, E), dtype=torch.int32, device="cuda")
    eager = torch.empty_like(x0)
    _stack(layers, x0, pol, eager, audit_e)   # also sizes the shared workspace before capture
    torch.cuda.synchronize()

    x_in = x0.clone()
    x_out = torch.empty_like(x0)
    audit_g = torch.zeros_like(audit_e)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):                 # warm-up on the capture stream
        _stack(layers, x_in, pol, x_out, audit_g)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        _stack(layers, x_in, pol, x_out, audit_g)
    audit_g.zero_()
    for rep in range(2):
        x_out.fill_(0)
        graph.replay()
        torch.cuda.synchronize()
        assert torch.equal(x_out.view(torch.int16), eager.view(torch.int16)), rep
    a = pmpe.audit_read(audit_g, s.T, E)
    tau = oracle.resolve(pol.cpu().numpy(), s.T)
    assert np.array_equal(a["route_priv_rows"], 2 * N_LAYERS * s.k * tau.astype(np.uint32))
    assert np.array_equal(a["exec_priv_rows"], a["route_priv_rows"])
    assert np.array_equal(a["exec_rows"], a["route_count"])
    assert a["route_count"].sum() == 2 * N_LAYERS * s.T * s.k


def test_training_step_with_private_backward_replays_bitwise_from_a_cuda_graph():
    """One training step of a two-layer stack captured into one CUDA graph:
    the layers' forwards (the second fed the first one's output), then the
    top layer's private gradients and input gradient in one combined pass
    from the gate/up accumulators its forward saved;
    that input gradient in BF16 is the upstream gradient of the lower layer's
    private-branch backward.
    Each layer keeps its own workspace, which holds that layer's forward state
    for its backward.  Replaying the graph twice gives bit for bit the outputs,
    the four private gradients of each layer and the top layer's input
    gradient computed one call at a time."""
    s = LayerShape(T=512, H=512, I=256, E_pub=32, E_priv=8, E_sh=1, k=4, renormalize=True)
    layers = [pmpe.MoeLayer(s, inp.make_weights(s, 8000 + l, device="cuda")) for l in range(2)]
    x0 = inp.make_hidden(s, 8, device="cuda")
    pol = inp.policy_iid_mixed(s.T, 8).cuda()
    gen = torch.Generator(device="cuda")
    gen.manual_seed(9)
    dtop = torch.randn((s.T, s.H), generator=gen, device="cuda").to(torch.bfloat16)

    def step(x_in, outs):
        ins = [x_in, outs[0]]
        for l, layer in enumerate(layers):
            # the top layer keeps its gate/up accumulators for its backward
            layer.forward(ins[l], pol, out=outs[l], save_for_backward=(l == 1))
        g1, dh1 = layers[1].backward(ins[1], pol, dtop)  # both results in one pass
        g0 = layers[0].backward_private(ins[0], pol, dh1.to(torch.bfloat16))
        return [g0, g1, {"d_hidden": dh1}]

    outs_e = [torch.empty_like(x0) for _ in layers]
    res_e = step(x0, outs_e)   # also sizes every workspace before capture
    torch.cuda.synchronize()
    res_e = [{n: v.clone() for n, v in g.items()} for g in res_e]
    assert torch.all(torch.isfinite(res_e[2]["d_hidden"])) and res_e[2]["d_hidden"].abs().max() > 0
    assert res_e[0]["d_gate"].abs().max() > 0

    x_in = x0.clone()
    outs_g = [torch.empty_like(x0) for _ in layers]
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):                 # warm-up on the capture stream
        step(x_in, outs_g)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        res_g = step(x_in, outs_g)
    for rep in range(2):
        for o in outs_g:
            o.fill_(0)
        graph.replay()
        torch.cuda.synchronize()
        for l in range(len(layers)):
            assert torch.equal(outs_g[l].view(torch.int16), outs_e[l].view(torch.int16)), (rep, l)
        for i in range(len(res_e)):
            for n in res_e[i]:
                assert torch.equal(res_g[i][n], res_e[i][n]), (rep, i, n)
