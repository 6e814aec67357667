"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times: the CPU oracle checks sampled tokens one by one, and the
properties that hold at any size (audit closed forms, G1, dispatch order) are
checked on every token."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_06690_gb300 import inputs as inp
from paper_2608_06690_gb300.configs import CONFIGS
from pmpe_testlib import check_against_oracle, check_audit, check_dispatch, run_gpu_layer

pytestmark = pytest.mark.gpu


def _sample_tokens(cfg, per_pool=12, seed=0):
    """Tokens spread over the requests, both pools represented."""
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
def test_full_size_workload(name):
    cfg = CONFIGS[name]
    s = cfg.shape
    w = inp.make_weights(s, cfg.seed, device="cuda", skew=cfg.skew)
    h = inp.make_hidden(s, cfg.seed, device="cuda", skew=cfg.skew)
    pol = cfg.policy(s.T)
    gpu = run_gpu_layer(s, w, h, pol.cuda())
    # properties on all tokens
    check_audit(s, pol, gpu)
    check_dispatch(s, h.cpu(), gpu)
    # the oracle on sampled tokens (full layer arithmetic in fp64)
    w_cpu = {k: (None if v is None else v.cpu()) for k, v in w.items()}
    toks = _sample_tokens(cfg) if s.T > 64 else None
    if toks is not None:
        rep = _check_sampled(s, w_cpu, h.cpu(), pol, gpu, toks)
    else:
        rep = check_against_oracle(s, w_cpu, h.cpu(), pol, gpu)
    assert rep["excused"] <= 2, rep


def _check_sampled(s, w_cpu, h_cpu, pol, gpu, toks):
    """check_against_oracle restricted to the sampled tokens."""
    from pmpe_testlib import GAP_EPS, MAX_ABS_REL, MEAN_REL, output_errors, oracle_layer
    L = oracle_layer(s, w_cpu, h_cpu, pol)
    r = oracle.forward(L, tokens=toks)
    tau = oracle.resolve(pol.numpy(), s.T)
    gi = gpu["idx"][toks]
    assert np.all((gi >= s.E_pub) == (tau[toks][:, None] == 1))
    ok = r["gap"] >= GAP_EPS
    assert np.array_equal(gi[ok], r["idx"][ok])
    np.testing.assert_allclose(gpu["w"][toks][ok], r["w"][ok], rtol=0, atol=2e-5)
    mx, mean = output_errors(gpu["out"][toks][ok], r["out"][ok])
    assert mx <= MAX_ABS_REL and mean <= MEAN_REL, (mx, mean)
    return dict(excused=int((~ok).sum()), max_abs_rel=mx, mean_rel=mean)
