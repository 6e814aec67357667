"""Helpers shared by the test files: building seeded layers and comparing
results.  Nothing here computes the layer itself."""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_06690_gb300 import inputs as inp
from paper_2608_06690_gb300.inputs import LayerShape


def make_layer(shape: LayerShape, seed: int, device="cpu", policy="iid", skew=None):
    """Seeded layer: (weights dict, hidden [T,H] bf16, policy uint8 [T] or None)."""
    w = inp.make_weights(shape, seed, device=device, skew=skew)
    h = inp.make_hidden(shape, seed, device=device, skew=skew)
    if isinstance(policy, str):
        if policy == "iid":
            pol = inp.policy_iid_mixed(shape.T, seed)
        elif policy == "allow":
            pol = inp.policy_const(shape.T, inp.ALLOW)
        elif policy == "deny":
            pol = inp.policy_const(shape.T, inp.DENY)
        elif policy == "none":
            pol = None
        else:
            raise ValueError(policy)
    else:
        pol = policy
    return w, h, pol


def oracle_layer(shape, w, h, pol):
    import oracle
    t = dict(w)
    t["hidden"] = h
    return oracle.Layer(shape, t, None if pol is None else pol.cpu().numpy())


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def bits_to_f64(a: np.ndarray) -> np.ndarray:
    return (np.asarray(a, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def output_errors(got_bits: np.ndarray, ref_bits: np.ndarray):
    """(max-abs error / max|ref|, sum|err| / sum|ref|) of two BF16 arrays."""
    g = bits_to_f64(got_bits)
    r = bits_to_f64(ref_bits)
    err = np.abs(g - r)
    scale = max(np.abs(r).max(), 1e-30)
    return float(err.max() / scale), float(err.sum() / max(np.abs(r).sum(), 1e-30))


# The output tolerance: max-abs error <= 1e-2 * max|ref| and mean relative
# error (sum|err| / sum|ref|) <= 5e-3, BF16 inputs with FP32 accumulation.
MAX_ABS_REL = 1e-2
MEAN_REL = 5e-3
# Router gap rule: a token whose k-th and (k+1)-th fp32 logits (oracle) are
# closer than this may legitimately pick a different k-th expert.
GAP_EPS = 1e-4
