"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: an
exhaustive enumeration, a closed form, a brute-force sort, a library routine
(torch.nn.functional in fp64, torch's BF16 conversion) or a hand-worked
fixture.  A plausible mistake in the oracle (a dropped mask, a wrong sign, a
transposed weight, swapped gate/up, a wrong softmax denominator, a wrong tie
break, an off-by-one in the dispatch order) fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2608_06690_gb300.inputs import LayerShape
from pmpe_testlib import make_layer, oracle_layer, bits_to_f64

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_worked.json")


# ------------------------------------------------------------------ BF16

def test_bf16_round_matches_torch_on_float32_values():
    """The oracle's double->BF16 rounding equals torch's float32->BF16
    round-to-nearest-even on values that are exact in float32 (so no double
    rounding is involved), including ties, subnormals and overflow."""
    g = torch.Generator().manual_seed(1)
    x = torch.randn(20000, generator=g) * torch.exp(torch.randn(20000, generator=g) * 8)
    ties = torch.tensor([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 2.0 ** -130, 3.0 * 2.0 ** -134,
                         3.3895e38, 3.4e38, -0.0, 0.0, 1e-45, 2.0 ** -126, 65504.0], dtype=torch.float32)
    x = torch.cat([x.float(), ties])
    want = x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.bf16_round(float(v)) for v in x.tolist()], dtype=np.uint16)
    assert np.array_equal(got, want)


# ---------------------------------------------------------------- resolve

def test_resolve_exhaustive_over_all_bytes():
    """Sec. 2.1 / App. B.1: only the trusted ALLOW value gives tau = 1;
    every other byte fails closed."""
    pol = np.arange(256, dtype=np.uint8)
    tau = oracle.resolve(pol, 256)
    assert tau[1] == 1 and tau.sum() == 1


def test_resolve_missing_metadata_is_deny():
    assert oracle.resolve(None, 37).sum() == 0


def test_policy_from_requests_closed_forms():
    """Per-request bytes expand to their requests' tokens; tokens after the
    last request are DENY; malformed offsets make the whole batch DENY."""
    g = np.random.default_rng(3)
    for _ in range(50):
        n = int(g.integers(1, 20))
        lens = g.integers(0, 40, size=n)
        T = int(lens.sum() + g.integers(0, 5))
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        rp = g.integers(0, 256, size=n).astype(np.uint8)
        rp[g.random(n) < 0.5] = 1
        got = oracle.policy_from_requests(rp, cu, T)
        want = np.concatenate([np.full(l, b, np.uint8) for l, b in zip(lens, rp)] + [np.zeros(T - lens.sum(), np.uint8)])
        assert np.array_equal(got, want)
    rp = np.array([1, 1, 1], np.uint8)
    for bad in ([1, 3, 5, 7], [0, 5, 3, 7], [0, 3, 5, 99]):   # cu[0] != 0, a decreasing step, past T
        assert oracle.policy_from_requests(rp, np.array(bad), 10).sum() == 0
    assert oracle.policy_from_requests(np.zeros(0, np.uint8), np.array([0]), 6).sum() == 0


# ---------------------------------------------------------------- routing

def _expected_topk(s_row, k):
    """Brute force: sort (score desc, id asc), keep the first k finite."""
    order = sorted(range(len(s_row)), key=lambda e: (-s_row[e], e))
    order = [e for e in order if s_row[e] != -math.inf]
    return order[:k], order


@pytest.mark.parametrize("renorm", [True, False])
def test_route_one_hot_rows_closed_form(renorm):
    """With h = one-hot(c), z_e = W_router[e, c] exactly; the oracle's top-k
    equals a brute-force sort of the eligible pool and its weights equal the
    softmax computed with math.exp."""
    s = LayerShape(T=96, H=64, I=16, E_pub=12, E_priv=6, E_sh=0, k=3, renormalize=renorm)
    w, _, pol = make_layer(s, seed=3)
    g = torch.Generator().manual_seed(5)
    cols = torch.randint(0, s.H, (s.T,), generator=g)
    h = torch.zeros(s.T, s.H)
    h[torch.arange(s.T), cols] = 1.0
    h = h.to(torch.bfloat16)
    L = oracle_layer(s, w, h, pol)
    idx, wt, gap = oracle.route(L)
    R = torch.cat([w["router_pub"], w["router_priv"]]).float().numpy()
    for t in range(s.T):
        allow = int(pol[t]) == 1
        srow = [float(R[e, cols[t]]) if ((e >= s.E_pub) == allow) else -math.inf for e in range(s.E)]
        top, order = _expected_topk(srow, s.k)
        assert list(idx[t]) == top
        m = srow[top[0]]
        ex = {e: math.exp(srow[e] - m) for e in order}
        denom = sum(ex[e] for e in (top if renorm else order))
        np.testing.assert_allclose(wt[t], [ex[e] / denom for e in top], rtol=1e-12)
        nxt = order[s.k] if len(order) > s.k else None
        assert gap[t] == (math.inf if nxt is None else srow[top[-1]] - srow[nxt])


def test_route_random_rows_brute_force_sort():
    """Random h: logits from numpy's float64 matmul rounded to fp32, masked,
    then a full sort -- equals the oracle's selection."""
    s = LayerShape(T=200, H=128, I=16, E_pub=20, E_priv=8, E_sh=0, k=4, renormalize=True)
    w, h, pol = make_layer(s, seed=11)
    L = oracle_layer(s, w, h, pol)
    idx, _, _ = oracle.route(L)
    R = torch.cat([w["router_pub"], w["router_priv"]]).double().numpy()
    Z = (h.double().numpy() @ R.T).astype(np.float32).astype(np.float64)
    for t in range(s.T):
        allow = int(pol[t]) == 1
        srow = [Z[t, e] if ((e >= s.E_pub) == allow) else -math.inf for e in range(s.E)]
        assert list(idx[t]) == _expected_topk(srow, s.k)[0]


@pytest.mark.parametrize("renorm", [True, False])
def test_route_equal_logits_tie_break_and_uniform_weights(renorm):
    """h = 0 makes every logit 0: the top-k are the k lowest ids of the pool
    and the weights are 1/k (renormalised) or 1/|pool| (pool softmax)."""
    s = LayerShape(T=4, H=32, I=8, E_pub=10, E_priv=5, E_sh=0, k=3, renormalize=renorm)
    w, _, _ = make_layer(s, seed=2)
    h = torch.zeros(s.T, s.H, dtype=torch.bfloat16)
    pol = torch.tensor([0, 1, 7, 1], dtype=torch.uint8)
    idx, wt, gap = oracle.route(oracle_layer(s, w, h, pol))
    assert idx.tolist() == [[0, 1, 2], [10, 11, 12], [0, 1, 2], [10, 11, 12]]
    for t in range(4):
        pool = s.E_priv if pol[t] == 1 else s.E_pub
        np.testing.assert_allclose(wt[t], [1 / s.k if renorm else 1 / pool] * s.k, rtol=1e-15)
    assert np.all(gap == 0.0)


def test_route_k_equals_pool_selects_whole_pool():
    s = LayerShape(T=16, H=32, I=8, E_pub=4, E_priv=4, E_sh=0, k=4, renormalize=False)
    w, h, pol = make_layer(s, seed=4)
    idx, wt, gap = oracle.route(oracle_layer(s, w, h, pol))
    for t in range(s.T):
        pool = set(range(4, 8)) if pol[t] == 1 else set(range(4))
        assert set(idx[t].tolist()) == pool
    np.testing.assert_allclose(wt.sum(1), 1.0, rtol=1e-12)   # pool softmax over the whole pool
    assert np.all(np.isinf(gap))


def test_unmasked_control_routes_over_the_whole_pool_brute_force():
    """The soft-router control (Sec. 4.2 and App. E, the soft-router-only
    arm of the control matrix): without the
    hard mask every expert of the concatenated pool is eligible.  Logits from
    numpy's float64 matmul rounded to fp32, a full sort over all E, and the
    softmax over all E (pool softmax) or over the top-k (renormalised)."""
    for renorm in (True, False):
        s = LayerShape(T=120, H=64, I=16, E_pub=12, E_priv=6, E_sh=0, k=3, renormalize=renorm)
        w, h, pol = make_layer(s, seed=21)
        idx, wt, gap = oracle.route(oracle_layer(s, w, h, pol, unmasked=True))
        R = torch.cat([w["router_pub"], w["router_priv"]]).double().numpy()
        Z = (h.double().numpy() @ R.T).astype(np.float32).astype(np.float64)
        for t in range(s.T):
            srow = list(Z[t])
            top, order = _expected_topk(srow, s.k)
            assert list(idx[t]) == top
            m = srow[top[0]]
            ex = {e: math.exp(srow[e] - m) for e in order}
            denom = sum(ex[e] for e in (top if renorm else order))
            np.testing.assert_allclose(wt[t], [ex[e] / denom for e in top], rtol=1e-12)
            assert gap[t] == srow[top[-1]] - srow[order[s.k]]


def test_unmasked_control_top1_is_the_better_masked_top1():
    """Without the mask, the best expert is the better of the best public
    expert (the masked DENY route) and the best private expert (the masked
    ALLOW route); and when the whole unmasked top-k lies in one pool, the
    renormalised weights equal that pool's masked ones."""
    s = LayerShape(T=300, H=128, I=16, E_pub=16, E_priv=8, E_sh=0, k=4, renormalize=True)
    w, h, _ = make_layer(s, seed=22)
    deny = torch.zeros(s.T, dtype=torch.uint8)
    allow = torch.ones(s.T, dtype=torch.uint8)
    i_d, w_d, _ = oracle.route(oracle_layer(s, w, h, deny))
    i_a, w_a, _ = oracle.route(oracle_layer(s, w, h, allow))
    i_u, w_u, _ = oracle.route(oracle_layer(s, w, h, deny, unmasked=True))
    R = torch.cat([w["router_pub"], w["router_priv"]]).double().numpy()
    Z = (h.double().numpy() @ R.T).astype(np.float32)
    one_pool = 0
    for t in range(s.T):
        a, b = i_d[t, 0], i_a[t, 0]
        best = a if (Z[t, a] > Z[t, b] or (Z[t, a] == Z[t, b] and a < b)) else b
        assert i_u[t, 0] == best
        if np.all(i_u[t] < s.E_pub):
            assert list(i_u[t]) == list(i_d[t]); np.testing.assert_allclose(w_u[t], w_d[t], rtol=1e-12); one_pool += 1
        elif np.all(i_u[t] >= s.E_pub):
            assert list(i_u[t]) == list(i_a[t]); np.testing.assert_allclose(w_u[t], w_a[t], rtol=1e-12); one_pool += 1
    assert one_pool > 0


def test_unmasked_control_executes_private_rows_for_deny_tokens():
    """The negative control: without the hard mask, DENY tokens reach private
    experts (the route log and the independent execution count both show it),
    which the masked layer never does (Sec. 2.2, G1)."""
    s = LayerShape(T=64, H=64, I=16, E_pub=8, E_priv=8, E_sh=0, k=2, renormalize=True)
    w, h, _ = make_layer(s, seed=23)
    deny = torch.zeros(s.T, dtype=torch.uint8)
    r_m = oracle.forward(oracle_layer(s, w, h, deny))
    r_u = oracle.forward(oracle_layer(s, w, h, deny, unmasked=True))
    assert r_m["exec_priv_rows"].sum() == 0 and r_m["route_priv_rows"].sum() == 0
    assert r_u["exec_priv_rows"].sum() > 0
    assert np.array_equal(r_u["exec_priv_rows"], r_u["route_priv_rows"])
    assert np.array_equal(r_u["route_priv_rows"], (r_u["idx"] >= s.E_pub).sum(1))


def test_route_k1_argmax_weight_one():
    s = LayerShape(T=50, H=64, I=8, E_pub=8, E_priv=3, E_sh=0, k=1, renormalize=True)
    w, h, pol = make_layer(s, seed=6)
    idx, wt, _ = oracle.route(oracle_layer(s, w, h, pol))
    assert np.all(wt == 1.0)


def test_weights_sum_rules():
    """Renormalised weights sum to 1; pool-softmax weights are each <= 1 and
    sum to at most 1."""
    for renorm in (True, False):
        s = LayerShape(T=64, H=64, I=8, E_pub=16, E_priv=8, E_sh=0, k=5, renormalize=renorm)
        w, h, pol = make_layer(s, seed=8)
        _, wt, _ = oracle.route(oracle_layer(s, w, h, pol))
        if renorm:
            np.testing.assert_allclose(wt.sum(1), 1.0, rtol=1e-12)
        else:
            assert np.all(wt <= 1.0) and np.all(wt.sum(1) <= 1.0 + 1e-12) and np.all(wt > 0)
        assert np.all(np.diff(wt, axis=1) <= 1e-15)               # descending score order


def test_mask_holds_against_adversarial_hidden_states():
    """Prompt content cannot change the pool (Sec. 3.1; App. F.1, the adversarial-suite table):
    hidden states built to maximise the *other* pool's logits still route
    inside the pool the policy selects."""
    s = LayerShape(T=8, H=64, I=8, E_pub=6, E_priv=4, E_sh=0, k=2, renormalize=True)
    w, _, _ = make_layer(s, seed=9)
    priv_dir = w["router_priv"].float().sum(0)
    pub_dir = w["router_pub"].float().sum(0)
    h = torch.stack([priv_dir * 50 * (i + 1) for i in range(4)] + [pub_dir * 50 * (i + 1) for i in range(4)])
    pol = torch.tensor([0, 0x7F, 0xFF, 2, 1, 1, 1, 1], dtype=torch.uint8)
    idx, _, _ = oracle.route(oracle_layer(s, w, h.to(torch.bfloat16), pol))
    assert np.all(idx[:4] < s.E_pub)
    assert np.all(idx[4:] >= s.E_pub)


# ---------------------------------------------------------------- experts

def _torch_mlp(h, g, u, d):
    """Textbook SwiGLU MLP in fp64 with the activation rounded to BF16."""
    a = (F.silu(F.linear(h, g)) * F.linear(h, u)).float().to(torch.bfloat16).double()
    return F.linear(a, d)


def test_expert_matches_textbook_swiglu():
    s = LayerShape(T=6, H=96, I=40, E_pub=3, E_priv=2, E_sh=2, k=1, renormalize=True)
    w, h, pol = make_layer(s, seed=10)
    L = oracle_layer(s, w, h, pol)
    for e in range(s.E):
        pool, j = ("pub", e) if e < s.E_pub else ("priv", e - s.E_pub)
        for t in range(s.T):
            y = oracle.expert(L, e, h[t])
            ref = _torch_mlp(h[t].double(), w[f"gate_{pool}"][j].double(), w[f"up_{pool}"][j].double(),
                             w[f"down_{pool}"][j].double()).numpy()
            np.testing.assert_allclose(y, ref, rtol=0, atol=1e-5 * np.abs(ref).max())
    for sidx in range(s.E_sh):
        y = oracle.expert(L, sidx, h[0], shared=True)
        ref = _torch_mlp(h[0].double(), w["gate_sh"][sidx].double(), w["up_sh"][sidx].double(),
                         w["down_sh"][sidx].double()).numpy()
        np.testing.assert_allclose(y, ref, rtol=0, atol=1e-5 * np.abs(ref).max())


def test_forward_single_expert_pools_reduce_to_dense_mlp():
    """E_pub = E_priv = k = 1 (renormalised): the layer is the dense SwiGLU
    MLP of the public expert under DENY and of the private one under ALLOW."""
    s = LayerShape(T=24, H=64, I=48, E_pub=1, E_priv=1, E_sh=0, k=1, renormalize=True)
    w, h, pol = make_layer(s, seed=12)
    r = oracle.forward(oracle_layer(s, w, h, pol))
    for t in range(s.T):
        pool = "priv" if pol[t] == 1 else "pub"
        ref = _torch_mlp(h[t].double(), w[f"gate_{pool}"][0].double(), w[f"up_{pool}"][0].double(),
                         w[f"down_{pool}"][0].double())
        np.testing.assert_allclose(r["out_f64"][t], ref.numpy(), rtol=0, atol=1e-5 * ref.abs().max().item())
        assert np.array_equal(r["out"][t], ref.float().to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16))


def test_forward_identical_experts_give_the_mlp():
    """If every routed expert has the same weights, the renormalised weights
    sum to 1 and the layer output is that one MLP, whatever the routing."""
    s = LayerShape(T=20, H=64, I=32, E_pub=6, E_priv=4, E_sh=0, k=3, renormalize=True)
    w, h, pol = make_layer(s, seed=13)
    for name in ("gate", "up", "down"):
        base = w[f"{name}_pub"][0]
        w[f"{name}_pub"] = base.expand(s.E_pub, *base.shape).contiguous()
        w[f"{name}_priv"] = base.expand(s.E_priv, *base.shape).contiguous()
    r = oracle.forward(oracle_layer(s, w, h, pol))
    ref = _torch_mlp(h.double(), w["gate_pub"][0].double(), w["up_pub"][0].double(), w["down_pub"][0].double())
    np.testing.assert_allclose(r["out_f64"], ref.numpy(), rtol=0, atol=1e-9 * ref.abs().max().item())


def test_forward_is_weighted_sum_of_routed_plus_shared_experts():
    """out = bf16(sum_j w_j MLP_{idx_j}(h) + sum_s MLP_s(h)) with the MLPs
    from torch.nn.functional; pins the combine order-free up to fp64."""
    s = LayerShape(T=12, H=64, I=32, E_pub=8, E_priv=4, E_sh=2, k=3, renormalize=False)
    w, h, pol = make_layer(s, seed=14)
    r = oracle.forward(oracle_layer(s, w, h, pol))
    for t in range(s.T):
        acc = torch.zeros(s.H, dtype=torch.float64)
        for j in range(s.k):
            e = int(r["idx"][t, j])
            pool, i = ("pub", e) if e < s.E_pub else ("priv", e - s.E_pub)
            acc += r["w"][t, j] * _torch_mlp(h[t].double(), w[f"gate_{pool}"][i].double(),
                                             w[f"up_{pool}"][i].double(), w[f"down_{pool}"][i].double())
        for sidx in range(s.E_sh):
            acc += _torch_mlp(h[t].double(), w["gate_sh"][sidx].double(), w["up_sh"][sidx].double(),
                              w["down_sh"][sidx].double())
        np.testing.assert_allclose(r["out_f64"][t], acc.numpy(), rtol=0, atol=1e-9 * acc.abs().max().item())


@pytest.mark.parametrize("unmasked", [False, True])
def test_logits_are_the_masked_fp32_matmul_and_reproduce_the_route(unmasked):
    """oracle.logits: numpy's float64 matmul of the BF16 values rounded to
    fp32, -inf outside the pool tau selects (none in the unmasked control);
    a brute-force sort of each row gives the oracle's top-k."""
    s = LayerShape(T=150, H=128, I=16, E_pub=20, E_priv=8, E_sh=0, k=4, renormalize=True)
    w, h, pol = make_layer(s, seed=21)
    L = oracle_layer(s, w, h, pol, unmasked=unmasked)
    got = oracle.logits(L)
    R = torch.cat([w["router_pub"], w["router_priv"]]).double().numpy()
    Z = (h.double().numpy() @ R.T).astype(np.float32).astype(np.float64)
    allow = (pol.numpy() == 1)[:, None]
    priv = (np.arange(s.E) >= s.E_pub)[None, :]
    want = Z if unmasked else np.where(allow == priv, Z, -np.inf)
    np.testing.assert_allclose(got, want, rtol=1e-6, atol=1e-7)
    assert np.array_equal(np.isinf(got), np.isinf(want))
    idx, _, _ = oracle.route(L)
    for t in range(s.T):
        assert list(idx[t]) == _expected_topk(list(got[t]), s.k)[0]
    toks = np.array([149, 3, 77], np.int32)
    assert np.array_equal(oracle.logits(L, tokens=toks), got[toks])


@pytest.mark.parametrize("renorm", [True, False])
def test_forward_forced_with_the_oracles_own_routing_is_the_forward(renorm):
    """Given the routing forward takes, forward_forced returns forward's
    output bits and weights (shared experts included)."""
    s = LayerShape(T=40, H=64, I=32, E_pub=9, E_priv=5, E_sh=1, k=3, renormalize=renorm)
    w, h, pol = make_layer(s, seed=22)
    L = oracle_layer(s, w, h, pol)
    r = oracle.forward(L)
    out, wt = oracle.forward_forced(L, r["idx"])
    assert np.array_equal(out, r["out"])
    np.testing.assert_array_equal(wt, r["w"])
    toks = np.array([5, 0, 39], np.int32)
    out2, _ = oracle.forward_forced(L, r["idx"][toks], tokens=toks)
    assert np.array_equal(out2, r["out"][toks])


def test_forward_forced_other_selections():
    """Any in-pool selection of identical experts gives that one MLP
    (renormalised weights sum to 1); with distinct experts a selection that
    swaps the k-th expert for the (k+1)-th changes the output by exactly the
    swapped terms, from torch.nn.functional MLPs and the logits' softmax."""
    s = LayerShape(T=16, H=64, I=32, E_pub=8, E_priv=4, E_sh=0, k=3, renormalize=True)
    w, h, pol = make_layer(s, seed=23)
    same = dict(w)
    for name in ("gate", "up", "down"):
        base = w[f"{name}_pub"][0]
        same[f"{name}_pub"] = base.expand(s.E_pub, *base.shape).contiguous()
        same[f"{name}_priv"] = base.expand(s.E_priv, *base.shape).contiguous()
    g = np.random.default_rng(4)
    tau = pol.numpy() == 1
    idx = np.stack([g.choice(np.arange(s.E_pub, s.E) if tau[t] else np.arange(s.E_pub), s.k, replace=False)
                    for t in range(s.T)]).astype(np.int32)
    out, wt = oracle.forward_forced(oracle_layer(s, same, h, pol), idx)
    np.testing.assert_allclose(wt.sum(1), 1.0, rtol=1e-12)
    ref = _torch_mlp(h.double(), same["gate_pub"][0].double(), same["up_pub"][0].double(),
                     same["down_pub"][0].double())
    assert np.array_equal(out, ref.float().to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16))
    # distinct experts: replace rank k-1 by the (k+1)-th best
    L = oracle_layer(s, w, h, pol)
    z = oracle.logits(L)
    r = oracle.forward(L)
    for t in range(s.T):
        order = _expected_topk(list(z[t]), s.k + 1)[0]
        sel = order[:s.k - 1] + [order[s.k]]
        o1, w1 = oracle.forward_forced(L, np.array([sel], np.int32), tokens=np.array([t], np.int32))
        ex = np.exp(z[t, sel] - z[t, order[0]])
        np.testing.assert_allclose(w1[0], ex / ex.sum(), rtol=1e-12)
        acc = torch.zeros(s.H, dtype=torch.float64)
        for j, e in enumerate(sel):
            pool, i = ("pub", e) if e < s.E_pub else ("priv", e - s.E_pub)
            acc += w1[0, j] * _torch_mlp(h[t].double(), w[f"gate_{pool}"][i].double(),
                                         w[f"up_{pool}"][i].double(), w[f"down_{pool}"][i].double())
        got = bits_to_f64(o1[0])
        np.testing.assert_allclose(got, acc.numpy(), rtol=0, atol=8e-3 * acc.abs().max().item())
        assert not np.array_equal(o1[0], r["out"][t])


# ------------------------------------------------------------------ audit

@pytest.mark.parametrize("policy", ["iid", "allow", "deny", "none"])
def test_audit_invariants(policy):
    """G1 (Sec. 2.2 Eq. 1) and the hook audit (Sec. 5.2, App. F.1): no
    private row executes for a token whose policy is not ALLOW; execution
    counts observed at the experts equal the route log; closed-form totals."""
    s = LayerShape(T=40, H=64, I=16, E_pub=10, E_priv=5, E_sh=1, k=2, renormalize=True)
    w, h, pol = make_layer(s, seed=15, policy=policy)
    r = oracle.forward(oracle_layer(s, w, h, pol))
    tau = oracle.resolve(None if pol is None else pol.numpy(), s.T)
    assert r["route_count"].sum() == s.T * s.k
    assert r["route_count"][s.E_pub:].sum() == s.k * tau.sum()
    assert r["route_count"][:s.E_pub].sum() == s.k * (s.T - tau.sum())
    assert np.array_equal(r["exec_rows"], r["route_count"])
    assert np.array_equal(r["route_priv_rows"], s.k * tau.astype(np.uint32))
    assert np.array_equal(r["exec_priv_rows"], r["route_priv_rows"])
    assert np.all(r["exec_priv_rows"][tau == 0] == 0)
    assert r["shared_rows"][0] == s.T * s.E_sh


# ---------------------------------------------------------------- permute

def test_permute_matches_brute_force_sort():
    g = torch.Generator().manual_seed(21)
    T, k, E = 57, 3, 11
    idx = np.stack([torch.randperm(E, generator=g)[:k].numpy() for _ in range(T)]).astype(np.int32)
    idx[5] = [0, 1, 2]                            # make sure some experts are hot
    counts, offsets, slot_of, tok_of_slot = oracle.permute(idx, E)
    rows = sorted(((int(idx[t, j]), t, j) for t in range(T) for j in range(k)))
    for slot, (e, t, j) in enumerate(rows):
        assert slot_of[t, j] == slot and tok_of_slot[slot] == t
    assert np.array_equal(counts, np.bincount(idx.reshape(-1), minlength=E))
    assert offsets[0] == 0 and np.array_equal(np.diff(offsets.astype(np.int64)), counts)


def test_permute_rejects_out_of_range_ids():
    with pytest.raises(ValueError):
        oracle.permute(np.array([[0, 5]], np.int32), 5)


# ----------------------------------------------------------------- golden

def _golden_layer(c):
    s = LayerShape(**c["shape"])
    bf = lambda v: torch.tensor(v, dtype=torch.float32).to(torch.bfloat16)
    t = {n: bf(c[n]) for n in ("hidden", "router_pub", "router_priv", "gate_pub", "up_pub", "down_pub",
                               "gate_priv", "up_priv", "down_priv")}
    for n in t:
        assert torch.equal(t[n].float(), torch.tensor(c[n], dtype=torch.float32)), "fixture not BF16-exact"
    return s, oracle.Layer(s, t, np.array(c["policy"], np.uint8))


@pytest.mark.parametrize("case", json.load(open(GOLDEN))["cases"], ids=lambda c: c["name"])
def test_golden_hand_worked(case):
    s, L = _golden_layer(case)
    r = oracle.forward(L)
    assert r["idx"].tolist() == case["expected_idx"]
    np.testing.assert_allclose(r["w"], case["expected_w"], rtol=1e-15)
    assert bits_to_f64(r["out"]).tolist() == case["expected_out"]


# ---------------------------------------------------- private-branch backward

def _bf16_step(t: torch.Tensor, index, up: bool) -> torch.Tensor:
    """A copy of BF16 tensor t with one element moved to the next BF16 value
    up or down (one unit in the last place)."""
    bits = t.view(torch.int16).clone()
    flat = bits.view(-1)
    i = int(np.ravel_multi_index(index, t.shape))
    v = int(flat[i]) & 0xFFFF
    mag, neg = v & 0x7FFF, v >> 15
    if (not neg) == up:
        mag += 1
    else:
        mag -= 1
    flat[i] = np.int16(np.uint16(mag | (neg << 15)).astype(np.int16))
    return bits.view(torch.bfloat16)


def _loss(s, w, h, pol, dout, unmasked=False):
    r = oracle.forward(oracle_layer(s, w, h, pol, unmasked=unmasked, exact=True))
    return float((r["out_f64"] * dout).sum()), r["idx"]


@pytest.mark.parametrize("renorm", [True, False])
def test_backward_matches_central_differences(renorm):
    """Central differences of sum(dout * out) over one-ULP BF16 steps of single
    private weights, on the forward without rounding (exact mode), routing
    unchanged under every step: router, gate, up and down gradients."""
    s = LayerShape(T=40, H=32, I=16, E_pub=6, E_priv=5, E_sh=0, k=2, renormalize=renorm)
    w, h, pol = make_layer(s, seed=31)
    w = {n: (v * 8).to(torch.bfloat16) if v is not None and n.endswith("priv") else v for n, v in w.items()}
    g = np.random.default_rng(5)
    dout = g.standard_normal((s.T, s.H))
    grads = oracle.backward_private(oracle_layer(s, w, h, pol, exact=True), dout)
    _, idx0 = _loss(s, w, h, pol, dout)
    checked = 0
    for name, gname in (("router_priv", "d_router"), ("gate_priv", "d_gate"), ("up_priv", "d_up"),
                        ("down_priv", "d_down")):
        G = grads[gname]
        picks = [np.unravel_index(int(i), G.shape) for i in np.argsort(-np.abs(G).ravel())[:4]]
        for index in picks:
            t0 = w[name]
            x = float(t0[index])
            wp, wm = dict(w), dict(w)
            wp[name] = _bf16_step(t0, index, True)
            wm[name] = _bf16_step(t0, index, False)
            lp, ip = _loss(s, wp, h, pol, dout)
            lm, im = _loss(s, wm, h, pol, dout)
            if not (np.array_equal(ip, idx0) and np.array_equal(im, idx0)):
                continue  # the step crossed a routing decision
            fd = (lp - lm) / (float(wp[name][index]) - float(wm[name][index]))
            assert fd == pytest.approx(G[index], rel=2e-3, abs=1e-9 * np.abs(G).max()), (gname, index, x)
            checked += 1
    assert checked >= 12


def test_backward_single_private_expert_is_the_dense_mlp_gradient():
    """E_priv = k = 1: every ALLOW token runs the one private expert with
    weight 1, so its gradients are torch.autograd's for the dense SwiGLU MLP
    (fp64, no rounding) summed over the ALLOW tokens, and the router gradient
    is exactly zero."""
    s = LayerShape(T=30, H=32, I=16, E_pub=3, E_priv=1, E_sh=0, k=1, renormalize=True)
    w, h, pol = make_layer(s, seed=32)
    dout = np.random.default_rng(6).standard_normal((s.T, s.H))
    r = oracle.backward_private(oracle_layer(s, w, h, pol, exact=True), dout)
    allow = oracle.resolve(pol.numpy(), s.T) == 1
    Wg = w["gate_priv"][0].double().requires_grad_()
    Wu = w["up_priv"][0].double().requires_grad_()
    Wd = w["down_priv"][0].double().requires_grad_()
    x = h.double()[torch.from_numpy(allow)]
    y = (F.silu(x @ Wg.T) * (x @ Wu.T)) @ Wd.T
    (y * torch.from_numpy(dout[allow])).sum().backward()
    np.testing.assert_allclose(r["d_gate"][0], Wg.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(r["d_up"][0], Wu.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(r["d_down"][0], Wd.grad.numpy(), rtol=1e-10, atol=1e-12)
    assert np.all(r["d_router"] == 0.0)


@pytest.mark.parametrize("renorm", [True, False])
def test_backward_g2_invariants(renorm):
    """G2: the upstream gradient of DENY tokens never reaches the private
    parameters (bitwise), and the router gradient sums to zero over the pool
    (softmax gradients are orthogonal to the constant vector).  Under the
    unmasked control, DENY tokens do reach them (the negative control)."""
    s = LayerShape(T=60, H=32, I=16, E_pub=6, E_priv=4, E_sh=0, k=2, renormalize=renorm)
    w, h, pol = make_layer(s, seed=33)
    tau = oracle.resolve(pol.numpy(), s.T)
    g = np.random.default_rng(7)
    d1 = g.standard_normal((s.T, s.H))
    d2 = d1.copy()
    d2[tau == 0] = g.standard_normal(((tau == 0).sum(), s.H))
    L = oracle_layer(s, w, h, pol)
    r1, r2 = oracle.backward_private(L, d1), oracle.backward_private(L, d2)
    for n in r1:
        assert np.array_equal(r1[n], r2[n]), n
    np.testing.assert_allclose(r1["d_router"].sum(0), 0.0, atol=1e-12 * np.abs(r1["d_router"]).max())
    Lu = oracle_layer(s, w, h, pol, unmasked=True)
    u1, u2 = oracle.backward_private(Lu, d1), oracle.backward_private(Lu, d2)
    assert any(not np.array_equal(u1[n], u2[n]) for n in u1)


# ------------------------------------------------- input gradient (backward)

@pytest.mark.parametrize("renorm", [True, False])
def test_input_gradient_matches_central_differences(renorm):
    """Central differences of sum(dout * out) over one-ULP BF16 steps of single
    hidden-state elements, on the forward without rounding (exact mode),
    routing unchanged under every step: the path through the routed experts
    (public for DENY, private for ALLOW tokens), the shared expert and the
    router of the token's pool."""
    s = LayerShape(T=24, H=32, I=16, E_pub=6, E_priv=5, E_sh=1, k=2, renormalize=renorm)
    w, h, pol = make_layer(s, seed=41)
    w = {n: (v * 8).to(torch.bfloat16) if v is not None else v for n, v in w.items()}
    g = np.random.default_rng(11)
    dout = g.standard_normal((s.T, s.H))
    dh = oracle.backward_input(oracle_layer(s, w, h, pol, exact=True), dout)
    _, idx0 = _loss(s, w, h, pol, dout)
    tau = oracle.resolve(pol.numpy(), s.T)
    checked = {0: 0, 1: 0}
    for pool in (0, 1):
        rows = np.flatnonzero(tau == pool)
        sub = np.abs(dh[rows])
        for flat in np.argsort(-sub.ravel())[:8]:
            r, c = np.unravel_index(int(flat), sub.shape)
            index = (int(rows[r]), int(c))
            hp, hm = _bf16_step(h, index, True), _bf16_step(h, index, False)
            lp, ip = _loss(s, w, hp, pol, dout)
            lm, im = _loss(s, w, hm, pol, dout)
            if not (np.array_equal(ip, idx0) and np.array_equal(im, idx0)):
                continue  # the step crossed a routing decision
            fd = (lp - lm) / (float(hp[index]) - float(hm[index]))
            assert fd == pytest.approx(dh[index], rel=2e-3, abs=1e-9 * np.abs(dh).max()), (index, pool)
            checked[pool] += 1
    assert checked[0] >= 4 and checked[1] >= 4, checked


def test_input_gradient_single_expert_pools_is_the_dense_mlp_gradient():
    """One expert per pool and k = 1: every token runs its pool's expert with
    weight 1 (the router contributes no gradient), plus the shared expert, so
    the input gradient is torch.autograd's for those dense SwiGLU MLPs (fp64,
    no rounding)."""
    s = LayerShape(T=20, H=32, I=16, E_pub=1, E_priv=1, E_sh=1, k=1, renormalize=True)
    w, h, pol = make_layer(s, seed=42)
    dout = np.random.default_rng(12).standard_normal((s.T, s.H))
    dh = oracle.backward_input(oracle_layer(s, w, h, pol, exact=True), dout)
    tau = oracle.resolve(pol.numpy(), s.T)

    def mlp(x, pre):
        Wg, Wu, Wd = (w[f"{n}_{pre}"][0].double() for n in ("gate", "up", "down"))
        return (F.silu(x @ Wg.T) * (x @ Wu.T)) @ Wd.T

    x = h.double().clone().requires_grad_()
    y = torch.where(torch.from_numpy(tau == 1)[:, None], mlp(x, "priv"), mlp(x, "pub")) + mlp(x, "sh")
    (y * torch.from_numpy(dout)).sum().backward()
    np.testing.assert_allclose(dh, x.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_input_gradient_pool_separation_and_linearity():
    """A DENY token's input gradient does not depend on the private weights
    and an ALLOW token's not on the public ones (bitwise): the mask of Sec. 3.1
    separates the backward paths as it separates the forward ones.  And the
    gradient is linear in dout."""
    s = LayerShape(T=40, H=32, I=16, E_pub=6, E_priv=4, E_sh=0, k=2, renormalize=False)
    w, h, pol = make_layer(s, seed=43)
    tau = oracle.resolve(pol.numpy(), s.T)
    dout = np.random.default_rng(13).standard_normal((s.T, s.H))
    base = oracle.backward_input(oracle_layer(s, w, h, pol), dout)
    for side, rows in (("priv", tau == 0), ("pub", tau == 1)):
        w2 = {n: ((v.float() * 1.5).to(torch.bfloat16) if v is not None and n.endswith(side) else v)
              for n, v in w.items()}
        other = oracle.backward_input(oracle_layer(s, w2, h, pol), dout)
        assert np.array_equal(base[rows], other[rows]), side
        assert not np.array_equal(base[~rows], other[~rows]), side
    np.testing.assert_allclose(oracle.backward_input(oracle_layer(s, w, h, pol), 2.5 * dout), 2.5 * base,
                               rtol=1e-12, atol=1e-14 * np.abs(base).max())
