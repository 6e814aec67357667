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


def oracle_layer(shape, w, h, pol, unmasked=False, exact=False):
    import oracle
    t = dict(w)
    t["hidden"] = h
    return oracle.Layer(shape, t, None if pol is None else pol.cpu().numpy(), unmasked=unmasked, exact=exact)


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


# ------------------------------------------------------------ GPU helpers

def to_device(w: dict, h, pol, device="cuda"):
    wd = {k: (None if v is None else v.to(device).contiguous()) for k, v in w.items()}
    return wd, h.to(device).contiguous(), (None if pol is None else pol.to(device).contiguous())


def run_gpu_layer(shape: LayerShape, w: dict, h, pol, audit_reset=True, stages=None, stage_seq=None):
    """Run the layer through the C ABI; return outputs, the route log, the
    audit counters and the dispatch intermediates, all on the host.  With
    ``stage_seq``, one call per listed stage mask on the same workspace."""
    from paper_2608_06690_gb300 import pmpe
    layer = pmpe.MoeLayer(shape, w)
    T, k, E = shape.T, shape.k, shape.E
    idx = torch.full((T, k), -1, dtype=torch.int32, device="cuda")
    wt = torch.full((T, k), float("nan"), dtype=torch.float32, device="cuda")
    audit = torch.zeros(pmpe.audit_words(T, E), dtype=torch.int32, device="cuda")
    out = torch.full((T, shape.H), float("nan"), dtype=torch.bfloat16, device="cuda")
    for st in (stage_seq if stage_seq is not None else [pmpe.STAGE_ALL if stages is None else stages]):
        layer.forward(h, pol, out=out, topk_idx=idx, topk_w=wt, audit=audit, stages=st)
    torch.cuda.synchronize()
    a = pmpe.audit_read(audit, T, E, check_status=False)
    ws = layer.workspace(T)
    L = pmpe.workspace_layout(shape)
    R = T * k

    def region(name, dtype, n):
        nbytes = n * torch.tensor([], dtype=dtype).element_size()
        return ws[L[name]:L[name] + nbytes].view(dtype).cpu()

    return dict(out=bf16_bits(out), idx=idx.cpu().numpy(), w=wt.cpu().numpy(), audit=a,
                tau=region("tau", torch.uint8, T).numpy(),
                counts=region("counts", torch.int32, E).numpy().view(np.uint32),
                offsets=region("offsets", torch.int32, E + 1).numpy().view(np.uint32),
                slot_of=region("slot_of", torch.int32, R).numpy().reshape(T, k),
                tok_of_slot=region("tok_of_slot", torch.int32, R).numpy(),
                layer=layer)


# Parity reports of the tests in this session, printed at the end of the run
# by the terminal-summary hook in conftest.py: per checked layer, the tokens
# compared, the tokens excused by the gap rule and the errors.
PARITY_REPORT: list = []


def record_parity(name: str, rep: dict):
    PARITY_REPORT.append(dict(name=name, **{k: v for k, v in rep.items() if k != "oracle"}))


def check_excused_tokens(shape: LayerShape, L, toks_ex, gpu_idx, gpu_w, gpu_out):
    """Tokens at a routing near-tie (oracle gap z_(k) - z_(k+1) < GAP_EPS) may
    legitimately select another k-th expert.  For them: the GPU's selection
    must be a valid top-k of the oracle's logits up to GAP_EPS (its sorted
    logits match the oracle's top-k logits within GAP_EPS, all inside the
    pool), and its weights and output must match the oracle run on that same
    selection (oracle.forward_forced).  Returns (max_abs_rel, mean_rel) of
    those outputs, or (0, 0) when there are none."""
    import oracle
    if len(toks_ex) == 0:
        return 0.0, 0.0
    toks_ex = np.asarray(toks_ex, dtype=np.int32)
    z = oracle.logits(L, tokens=toks_ex)
    for p, t in enumerate(toks_ex):
        zs = np.sort(z[p])[::-1]
        mine = np.sort(z[p, gpu_idx[p]])[::-1]
        assert np.all(np.isfinite(mine)), f"token {t}: a selected expert lies outside the pool"
        assert len(set(gpu_idx[p].tolist())) == shape.k, f"token {t}: an expert selected twice"
        assert np.all(np.abs(mine - zs[:shape.k]) < GAP_EPS), f"token {t}: not a valid top-k at the near-tie"
    ref_out, ref_w = oracle.forward_forced(L, gpu_idx, tokens=toks_ex)
    # the GPU reports ids in descending score; at a near-tie two ids may swap
    # places, so weights are matched id by id
    for p in range(len(toks_ex)):
        wmap = dict(zip(gpu_idx[p].tolist(), ref_w[p].tolist()))
        np.testing.assert_allclose(gpu_w[p], [wmap[e] for e in gpu_idx[p].tolist()], rtol=0, atol=2e-5)
    return output_errors(gpu_out, ref_out)


def check_against_oracle(shape: LayerShape, w_cpu: dict, h_cpu, pol_cpu, gpu: dict, tokens=None,
                         name: str | None = None):
    """Compare a GPU run with the oracle on the same inputs, on all tokens
    or on the listed ``tokens``.  Returns a report dict; asserts the rules:
      * tau bit-exact; every routed id inside the pool tau selects;
      * top-k ids bit-exact except tokens whose oracle gap z_(k) - z_(k+1) is
        below GAP_EPS (counted and reported; their selection must be a valid
        top-k at the near-tie, and their weights and outputs must match the
        oracle run on the selection the GPU made);
      * routing weights within 2e-5 (absolute);
      * outputs within MAX_ABS_REL * max|ref| and MEAN_REL mean relative error.
    With ``name``, the report is recorded for the end-of-run summary.
    """
    import oracle
    L = oracle_layer(shape, w_cpu, h_cpu, pol_cpu)
    r = oracle.forward(L, tokens=tokens)
    toks = np.arange(shape.T) if tokens is None else np.asarray(tokens)
    tau = oracle.resolve(None if pol_cpu is None else pol_cpu.numpy(), shape.T)
    assert np.array_equal(gpu["tau"], tau), "resolved policy differs"
    gi = gpu["idx"]
    in_priv = gi >= shape.E_pub
    assert np.all((gi >= 0) & (gi < shape.E)), "routed id out of range"
    assert np.all(in_priv == (tau[:, None] == 1)), "a routed id lies outside the pool tau selects"
    excused = r["gap"] < GAP_EPS
    ok = ~excused
    assert np.array_equal(gi[toks][ok], r["idx"][ok]), "top-k ids differ on tokens outside the gap rule"
    np.testing.assert_allclose(gpu["w"][toks][ok], r["w"][ok], rtol=0, atol=2e-5)
    mx, mean = output_errors(gpu["out"][toks][ok], r["out"][ok])
    assert mx <= MAX_ABS_REL and mean <= MEAN_REL, (mx, mean)
    ex_t = toks[excused]
    ex_mx, ex_mean = check_excused_tokens(shape, L, ex_t, gi[ex_t], gpu["w"][ex_t], gpu["out"][ex_t])
    assert ex_mx <= MAX_ABS_REL and ex_mean <= MEAN_REL, (ex_mx, ex_mean)
    n_swapped = int(sum(not np.array_equal(gi[t], r["idx"][p]) for p, t in enumerate(toks) if excused[p]))
    rep = dict(tokens=int(len(toks)), excused=int(excused.sum()), excused_selection_differs=n_swapped,
               max_abs_rel=mx, mean_rel=mean, excused_max_abs_rel=ex_mx, excused_mean_rel=ex_mean, oracle=r)
    if name is not None:
        record_parity(name, rep)
    return rep


def check_audit(shape: LayerShape, pol_cpu, gpu: dict):
    """Audit invariants that hold at any size (G1 of Sec. 2.2 Eq. 1 and the
    hook audit of Sec. 5.2): route log == histogram of the routed ids,
    execution counts == route counts, no private row for a DENY token."""
    import oracle
    a = gpu["audit"]
    tau = oracle.resolve(None if pol_cpu is None else pol_cpu.numpy(), shape.T)
    hist = np.bincount(gpu["idx"].reshape(-1), minlength=shape.E).astype(np.uint32)
    assert a["status"] == 0, a["status"]
    assert np.array_equal(a["route_count"], hist)
    assert np.array_equal(gpu["counts"], hist)
    assert a["route_count"].sum() == shape.T * shape.k
    assert a["route_count"][shape.E_pub:].sum() == shape.k * tau.sum()
    assert np.array_equal(a["exec_rows"], a["route_count"]), "execution audit differs from the route log"
    assert np.array_equal(a["exec_tiles"] > 0, hist > 0), "an expert ran tiles without rows, or rows without tiles"
    assert np.array_equal(a["route_priv_rows"], shape.k * tau.astype(np.uint32))
    assert np.array_equal(a["exec_priv_rows"], a["route_priv_rows"])
    assert np.all(a["exec_priv_rows"][tau == 0] == 0), "a DENY token executed a private expert row"
    assert a["shared_rows"] == shape.T * shape.E_sh


def check_dispatch(shape: LayerShape, h_cpu, gpu: dict):
    """The dispatch grouping against the oracle's definition applied to the
    GPU's own route log, bit for bit: the expert offsets, and the stable slot
    order (expert-major, then token, then rank) in slot_of and tok_of_slot;
    plus the structure (slot_of a bijection onto [0, T*k) that tok_of_slot
    inverts).  The expert kernel gathers each slot's row from the hidden
    states through tok_of_slot, so these maps are what it runs on."""
    import oracle
    counts, offsets, slot_of_ref, tok_of_slot_ref = oracle.permute(gpu["idx"], shape.E)
    assert np.array_equal(gpu["offsets"], offsets)
    assert np.array_equal(gpu["slot_of"], slot_of_ref), "slot_of differs from the stable dispatch order"
    assert np.array_equal(gpu["tok_of_slot"], tok_of_slot_ref), "tok_of_slot differs from the stable dispatch order"
    T, k = gpu["idx"].shape
    so = gpu["slot_of"]
    assert np.array_equal(np.sort(so.reshape(-1)), np.arange(T * k)), "slot_of is not a bijection"
    tos = gpu["tok_of_slot"]
    assert np.array_equal(tos[so], np.repeat(np.arange(T), k).reshape(T, k)), "tok_of_slot does not invert slot_of"
    for e in range(shape.E):
        lo, hi = offsets[e], offsets[e + 1]
        assert np.array_equal(np.sort(tos[lo:hi]), tok_of_slot_ref[lo:hi]), f"expert {e} holds other tokens"
        mine = gpu["idx"] == e
        assert np.all((so[mine] >= lo) & (so[mine] < hi)), f"a row of expert {e} sits outside its slots"
