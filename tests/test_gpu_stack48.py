"""The 48-layer Qwen3-shaped stack (16384 tokens in 64 requests, residual
add between layers, attention omitted; about 72 GB of BF16 weights resident
on the GPU): allow -> deny -> allow recovery is bitwise (Sec. 3.3, App.
F.3), 64 seeded adversarial policy vectors execute zero private rows wherever
the byte is not a valid ALLOW (Sec. 2.2 Eq. 1; App. F.1, the adversarial-suite table), and the
oracle, fed the GPU's own input to layers 0, 23 and 47 (teacher forcing),
matches the layer: every token of layer 47, 1024 tokens spread over the 64
requests at layers 0 and 23."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_06690_gb300 import inputs as inp
from paper_2608_06690_gb300 import pmpe
from paper_2608_06690_gb300.configs import CONFIGS
from pmpe_testlib import bf16_bits, check_against_oracle, check_audit, run_gpu_layer

pytestmark = pytest.mark.gpu

CHECK_LAYERS = (0, 23, 47)


@pytest.fixture(scope="module")
def stack():
    cfg = CONFIGS["qwen3_stack48"]
    s = cfg.shape
    free, _ = torch.cuda.mem_get_info()
    need = cfg.n_layers * 3 * (s.E_pub + s.E_priv) * s.I * s.H * 2 + (8 << 30)
    if free < need:
        pytest.skip(f"needs {need >> 30} GB free on the GPU, {free >> 30} GB available")
    ws = pmpe.Workspace("cuda")  # the layers run in sequence: one scratch buffer for all of them
    layers = [pmpe.MoeLayer(s, inp.make_weights(s, cfg.seed * 1000 + l, device="cuda"), workspace=ws)
              for l in range(cfg.n_layers)]
    x0 = inp.make_hidden(s, cfg.seed, device="cuda")
    yield cfg, layers, x0
    del layers
    torch.cuda.empty_cache()


def run_stack(layers, x0, pol, audit=None, keep=()):
    """x_{l+1} = bf16(x_l + moe_l(x_l)); returns the final x and, for the
    layers in `keep`, (x_l, moe_l(x_l))."""
    x = x0
    kept = {}
    out = torch.empty_like(x0)
    for l, layer in enumerate(layers):
        layer.forward(x, pol, out=out, audit=audit)
        if l in keep:
            kept[l] = (x.clone(), out.clone())
        x = (x.float() + out.float()).to(torch.bfloat16)
    return x, kept


def test_allow_deny_allow_recovery_is_bitwise(stack):
    cfg, layers, x0 = stack
    s = cfg.shape
    allow = inp.policy_const(s.T, inp.ALLOW).cuda()
    deny = inp.policy_const(s.T, inp.DENY).cuda()
    E = s.E
    a = torch.zeros(pmpe.audit_words(s.T, E), dtype=torch.int32, device="cuda")
    xa, _ = run_stack(layers, x0, allow, a)
    aa = pmpe.audit_read(a, s.T, E)
    pmpe.audit_reset(a, s.T, E)
    xd, _ = run_stack(layers, x0, deny, a)
    ad = pmpe.audit_read(a, s.T, E)
    pmpe.audit_reset(a, s.T, E)
    xr, _ = run_stack(layers, x0, allow, a)
    ar = pmpe.audit_read(a, s.T, E)
    L = cfg.n_layers
    assert torch.equal(xa.view(torch.int16), xr.view(torch.int16)), "recovery differs from the first ALLOW pass"
    assert not torch.equal(xa.view(torch.int16), xd.view(torch.int16))
    # DENY: zero private rows in every layer; ALLOW: private only
    assert ad["exec_rows"][s.E_pub:].sum() == 0 and ad["route_count"][s.E_pub:].sum() == 0
    assert np.all(ad["exec_priv_rows"] == 0)
    for x in (aa, ar):
        assert x["exec_rows"][:s.E_pub].sum() == 0
        assert np.all(x["exec_priv_rows"] == L * s.k)
        assert np.array_equal(x["exec_rows"], x["route_count"])
    assert np.array_equal(aa["route_count"], ar["route_count"])


def test_adversarial_policy_vectors_execute_no_private_rows(stack):
    cfg, layers, x0 = stack
    s = cfg.shape
    E, L = s.E, cfg.n_layers
    a = torch.zeros(pmpe.audit_words(s.T, E), dtype=torch.int32, device="cuda")
    vectors = inp.adversarial_policies(s.T, cfg.n_requests, cfg.seed, count=64)
    families = set()
    for fam, pol in vectors:
        families.add(fam)
        pmpe.audit_reset(a, s.T, E)
        run_stack(layers, x0, pol.cuda(), a)
        r = pmpe.audit_read(a, s.T, E)
        tau = oracle.resolve(pol.numpy(), s.T).astype(np.uint32)
        assert np.all(r["exec_priv_rows"][tau == 0] == 0), fam
        assert np.array_equal(r["exec_priv_rows"], L * s.k * tau), fam
        assert np.array_equal(r["route_priv_rows"], r["exec_priv_rows"]), fam
        assert np.array_equal(r["exec_rows"], r["route_count"]), fam
        assert r["route_count"][s.E_pub:].sum() == L * s.k * tau.sum(), fam
    assert families == {"all_malformed", "flipped_mid_request", "random_bytes"}


def test_teacher_forced_oracle_on_checked_layers(stack):
    """The stack runs once with the workload's policy; each checked layer is
    then re-run alone on the input it saw inside the stack, which must give
    the in-stack output bit for bit (the layer is deterministic and
    batch-invariant), and that run is compared with the oracle: every token
    of the last layer, 1024 tokens (16 per request) of layers 0 and 23."""
    cfg, layers, x0 = stack
    s = cfg.shape
    pol = cfg.policy(s.T)
    _, kept = run_stack(layers, x0, pol.cuda(), keep=CHECK_LAYERS)
    per_req = s.T // cfg.n_requests
    some = np.array([r * per_req + i for r in range(cfg.n_requests) for i in range(16)], np.int32)
    for l in CHECK_LAYERS:
        x_in, y = kept[l]
        gpu = run_gpu_layer(s, layers[l].weights, x_in, pol.cuda())
        assert np.array_equal(gpu["out"], bf16_bits(y)), f"layer {l}: re-run differs from the in-stack output"
        check_audit(s, pol, gpu)
        w_cpu = {k: (None if v is None else v.cpu()) for k, v in layers[l].weights.items()}
        toks = None if l == CHECK_LAYERS[-1] else some
        rep = check_against_oracle(s, w_cpu, x_in.cpu(), pol, gpu, tokens=toks,
                                   name=f"qwen3_stack48 layer {l} (teacher-forced)")
        assert rep["excused"] <= max(2, rep["tokens"] // 100), (l, rep)
        del gpu
