"""The five workloads of the policy-masked MoE layer, shaped like the paper's
two wrapped models (Sec. 4.1 Table 1, App. C.1 and C.3): a tiny layer for
exhaustive parity, a Qwen3-30B-A3B-shaped prefill layer, a DeepSeek-V2-Lite-
shaped layer with shared experts and skewed expert load, a Qwen3-shaped decode
step, and a 48-layer Qwen3-shaped stack.  Weights are random (the checkpoints
are not used); see ``inputs`` for the recipe.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable, Optional

from . import inputs as inp
from .inputs import LayerShape


@dataclass(frozen=True)
class Workload:
    name: str
    shape: LayerShape
    seed: int
    policy: Callable[[int], "object"]   # T -> uint8 tensor of policy bytes
    n_requests: int
    n_layers: int = 1
    skew: Optional[dict] = None
    note: str = ""
    extra: dict = field(default_factory=dict)


CONFIGS = {
    "tiny": Workload(
        name="tiny",
        shape=LayerShape(T=64, H=256, I=128, E_pub=16, E_priv=4, E_sh=0, k=2, renormalize=True),
        seed=0, n_requests=64,
        policy=lambda T: inp.policy_iid_mixed(T, 0),
        note="64 tokens, iid policy bytes 45% ALLOW / 45% DENY / 10% malformed"),
    "qwen3_prefill": Workload(
        name="qwen3_prefill",
        shape=LayerShape(T=4096, H=2048, I=768, E_pub=128, E_priv=32, E_sh=0, k=8, renormalize=True),
        seed=2, n_requests=16,
        policy=lambda T: inp.policy_requests(T, 16, 8, 2),
        note="16 requests x 256 tokens, 8 of 16 requests ALLOW"),
    "deepseek_v2_lite": Workload(
        name="deepseek_v2_lite",
        shape=LayerShape(T=8192, H=2048, I=1408, E_pub=64, E_priv=16, E_sh=2, k=6, renormalize=False),
        seed=3, n_requests=32,
        policy=lambda T: inp.policy_requests(T, 32, 8, 3),
        # beta chosen with tests/golden/calibrate_skew.py: the hottest public
        # expert gets 4.0x the mean public load (the private pool of 16 with
        # top-6 cannot exceed 16/6 = 2.67x; it reaches 1.66x)
        skew=dict(beta=0.175, c=4.0, u_seed=303),
        note="32 requests x 256 tokens, 8 of 32 ALLOW, Gumbel-skewed router, 2 shared experts"),
    "qwen3_decode": Workload(
        name="qwen3_decode",
        shape=LayerShape(T=64, H=2048, I=768, E_pub=128, E_priv=32, E_sh=0, k=8, renormalize=True),
        seed=4, n_requests=64,
        policy=lambda T: inp.policy_alternating(T, 64),
        note="64 requests x 1 token, ALLOW/DENY alternating"),
    "qwen3_stack48": Workload(
        name="qwen3_stack48",
        shape=LayerShape(T=16384, H=2048, I=768, E_pub=128, E_priv=32, E_sh=0, k=8, renormalize=True),
        seed=5, n_requests=64, n_layers=48,
        policy=lambda T: inp.policy_requests(T, 64, 32, 5),
        note="48 layers, residual add between layers, 64 requests x 256 tokens"),
}
