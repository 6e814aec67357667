"""Seeded synthetic inputs for the policy-masked sparse-MoE layer.

This module only draws random numbers and lays them out; it holds none of the
layer's arithmetic (no routing, no softmax, no expert math).  It is the one
module that both the CUDA path's callers and the CPU oracle's tests use.

Recipe (shapes and distributions of the paper's two wrapped models, Sec. 4.1
Table 1 and App. C; the checkpoints themselves are not used):
  * weights ~ N(0, 0.02^2), hidden states ~ N(0, 1), both rounded to BF16 by
    torch's round-to-nearest-even conversion;
  * weight layouts follow the [out, in] convention of a linear layer:
    router [E, H], gate/up [E, I, H], down [E, H, I];
  * policies are one byte per token; requests are contiguous token spans.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

ALLOW = 0x01
DENY = 0x00


@dataclass(frozen=True)
class LayerShape:
    T: int            # tokens
    H: int            # hidden size
    I: int            # expert intermediate size
    E_pub: int        # public routed experts
    E_priv: int       # private routed experts
    E_sh: int         # always-on shared experts (0 if none)
    k: int            # top-k inside the selected pool
    renormalize: bool  # True: softmax renormalised over the top-k

    @property
    def E(self) -> int:
        return self.E_pub + self.E_priv


WEIGHT_NAMES = ("router_pub", "router_priv", "gate_pub", "up_pub", "down_pub",
                "gate_priv", "up_priv", "down_priv", "gate_sh", "up_sh", "down_sh")


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _normal(shape, std, g, device) -> torch.Tensor:
    return (torch.randn(shape, generator=g, device=device, dtype=torch.float32) * std).to(torch.bfloat16)


def make_weights(s: LayerShape, seed: int, device="cpu", std: float = 0.02, skew=None) -> dict:
    """Router and expert weights of one layer.  ``skew`` (a dict with keys
    beta, c, u_seed) adds the load-skew construction: router row e gets
    (b_e / c) * u with b_e = beta * Gumbel(0, 1) and u a seeded unit vector;
    the hidden states then get c * u (see ``make_hidden``)."""
    g = _gen(seed, device)
    w = {}
    w["router_pub"] = _normal((s.E_pub, s.H), std, g, device)
    w["router_priv"] = _normal((s.E_priv, s.H), std, g, device)
    for pool, n in (("pub", s.E_pub), ("priv", s.E_priv), ("sh", s.E_sh)):
        if n == 0:
            w[f"gate_{pool}"] = w[f"up_{pool}"] = w[f"down_{pool}"] = None
            continue
        w[f"gate_{pool}"] = _normal((n, s.I, s.H), std, g, device)
        w[f"up_{pool}"] = _normal((n, s.I, s.H), std, g, device)
        w[f"down_{pool}"] = _normal((n, s.H, s.I), std, g, device)
    if skew is not None:
        u = skew_direction(s.H, skew["u_seed"], device)
        gs = _gen(skew["u_seed"] + 1, device)
        for name, n in (("router_pub", s.E_pub), ("router_priv", s.E_priv)):
            unif = torch.rand((n,), generator=gs, device=device, dtype=torch.float64).clamp_(1e-12, 1 - 1e-12)
            gumbel = -torch.log(-torch.log(unif))
            b = skew["beta"] * gumbel
            w[name] = (w[name].float() + (b / skew["c"]).float()[:, None] * u[None, :]).to(torch.bfloat16)
    return w


def skew_direction(H: int, seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed, device)
    u = torch.randn((H,), generator=g, device=device, dtype=torch.float32)
    return u / u.norm()


def make_hidden(s: LayerShape, seed: int, device="cpu", std: float = 1.0, skew=None) -> torch.Tensor:
    g = _gen(seed + 1_000_003, device)
    h = torch.randn((s.T, s.H), generator=g, device=device, dtype=torch.float32) * std
    if skew is not None:
        h = h + skew["c"] * skew_direction(s.H, skew["u_seed"], device)[None, :]
    return h.to(torch.bfloat16)


# ----------------------------------------------------------------- policies

def policy_iid_mixed(T: int, seed: int, p_allow=0.45, p_deny=0.45) -> torch.Tensor:
    """Per-token bytes: ALLOW with p_allow, DENY with p_deny, otherwise a
    malformed byte drawn uniformly from 2..255."""
    g = _gen(seed + 17, "cpu")
    u = torch.rand((T,), generator=g)
    bad = torch.randint(2, 256, (T,), generator=g, dtype=torch.int64)
    out = torch.where(u < p_allow, torch.full_like(bad, ALLOW),
                      torch.where(u < p_allow + p_deny, torch.full_like(bad, DENY), bad))
    return out.to(torch.uint8)


def policy_requests(T: int, n_requests: int, n_allow: int, seed: int) -> torch.Tensor:
    """T tokens in n_requests equal contiguous requests; exactly n_allow of
    them, chosen by a seeded permutation, are ALLOW, the rest DENY."""
    assert T % n_requests == 0
    g = _gen(seed + 29, "cpu")
    perm = torch.randperm(n_requests, generator=g)
    req_policy = torch.zeros(n_requests, dtype=torch.uint8)
    req_policy[perm[:n_allow]] = ALLOW
    return req_policy.repeat_interleave(T // n_requests)


def policy_alternating(T: int, n_requests: int) -> torch.Tensor:
    """Request r is ALLOW for even r, DENY for odd r."""
    assert T % n_requests == 0
    req = torch.tensor([ALLOW if r % 2 == 0 else DENY for r in range(n_requests)], dtype=torch.uint8)
    return req.repeat_interleave(T // n_requests)


def policy_const(T: int, byte: int) -> torch.Tensor:
    return torch.full((T,), byte, dtype=torch.uint8)


def adversarial_policies(T: int, n_requests: int, seed: int, count: int = 64) -> list:
    """Seeded adversarial policy vectors, cycling through three families:
    all-malformed (every byte in 2..255), flipped mid-request (each request
    switches between ALLOW and DENY half-way, in a random direction), and
    random bytes (uniform 0..255, so about 1 in 256 tokens is ALLOW).
    Returns a list of (family, uint8 tensor)."""
    g = _gen(seed + 41, "cpu")
    L = T // n_requests
    out = []
    for i in range(count):
        fam = ("all_malformed", "flipped_mid_request", "random_bytes")[i % 3]
        if fam == "all_malformed":
            p = torch.randint(2, 256, (T,), generator=g, dtype=torch.int64).to(torch.uint8)
        elif fam == "flipped_mid_request":
            first = torch.randint(0, 2, (n_requests,), generator=g).to(torch.uint8)
            cut = torch.randint(1, L, (n_requests,), generator=g)
            pos = torch.arange(L)[None, :]
            before = (pos < cut[:, None]).to(torch.uint8)
            p = torch.where(before.bool(), first[:, None], 1 - first[:, None]).reshape(-1).to(torch.uint8)
        else:
            p = torch.randint(0, 256, (T,), generator=g, dtype=torch.int64).to(torch.uint8)
        out.append((fam, p))
    return out

