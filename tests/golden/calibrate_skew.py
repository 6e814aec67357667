"""Pick the Gumbel load-skew strength beta of the DeepSeek-V2-Lite-shaped
workload (8192 tokens, 64 public + 16 private experts, top-6, 2 shared
experts): the hottest routed expert of each pool should receive about 4x the
mean load.  Routing is computed by the CPU oracle only.

Usage: python tests/golden/calibrate_skew.py [beta ...]
"""
import os
import sys

import numpy as np

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__)))))
import oracle  # noqa: E402
from paper_2608_06690_gb300 import inputs as inp  # noqa: E402
from paper_2608_06690_gb300.configs import CONFIGS  # noqa: E402


def load_ratio(beta: float, T: int = 8192):
    cfg = CONFIGS["deepseek_v2_lite"]
    s = cfg.shape
    # the router weights are drawn before the expert weights, so a small I
    # gives the same routers and keeps this script fast
    s = inp.LayerShape(T, s.H, 128, s.E_pub, s.E_priv, 0, s.k, s.renormalize)
    skew = dict(cfg.skew, beta=beta)
    w = inp.make_weights(s, cfg.seed, skew=skew)
    h = inp.make_hidden(s, cfg.seed, skew=skew)
    pol = cfg.policy(T)
    L = oracle.Layer(s, dict(w, hidden=h), pol.numpy())
    idx, _, _ = oracle.route(L)
    cnt = np.bincount(idx.reshape(-1), minlength=s.E)
    pub, priv = cnt[:s.E_pub], cnt[s.E_pub:]
    return pub.max() / pub.mean(), priv.max() / priv.mean()


if __name__ == "__main__":
    betas = [float(b) for b in sys.argv[1:]] or [0.0, 0.5, 1.0, 1.5, 2.0, 3.0]
    for b in betas:
        r = load_ratio(b)
        print(f"beta={b:4.2f}  public max/mean={r[0]:.2f}  private max/mean={r[1]:.2f}")
