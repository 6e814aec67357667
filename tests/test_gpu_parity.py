"""GPU parity of the policy-masked MoE layer against the CPU oracle, through
the C ABI (libpmpe.so), on seeded inputs of sizes the oracle finishes in
seconds -- several tiles, ragged tails -- plus the edge cases of the method."""
import hashlib

import numpy as np
import pytest
import torch

import oracle
from paper_2608_06690_gb300 import inputs as inp
from paper_2608_06690_gb300.configs import CONFIGS
from paper_2608_06690_gb300.inputs import LayerShape
from pmpe_testlib import (bf16_bits, check_against_oracle, check_audit, check_dispatch, make_layer, run_gpu_layer,
                          to_device)

pytestmark = pytest.mark.gpu

CASES = {
    # name: (shape, seed, policy)
    "tiny_config": (CONFIGS["tiny"].shape, 0, "config"),
    "ragged_multi_tile": (LayerShape(T=300, H=384, I=256, E_pub=24, E_priv=8, E_sh=0, k=4, renormalize=True), 31,
                          "iid"),
    "no_renorm_with_shared": (LayerShape(T=200, H=256, I=256, E_pub=16, E_priv=8, E_sh=2, k=3, renormalize=False),
                              32, "iid"),
    "all_allow": (LayerShape(T=130, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True), 33, "allow"),
    "all_deny": (LayerShape(T=130, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True), 34, "deny"),
    "missing_metadata": (LayerShape(T=77, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True), 35,
                         "none"),
    "paper_pool_16_private_top8": (LayerShape(T=160, H=256, I=128, E_pub=32, E_priv=16, E_sh=0, k=8,
                                              renormalize=True), 36, "iid"),
    "k1_argmax": (LayerShape(T=100, H=128, I=128, E_pub=12, E_priv=5, E_sh=0, k=1, renormalize=True), 37, "iid"),
    "k_equals_pool": (LayerShape(T=90, H=128, I=128, E_pub=4, E_priv=4, E_sh=0, k=4, renormalize=False), 38, "iid"),
    "large_pools_256": (LayerShape(T=96, H=128, I=128, E_pub=256, E_priv=256, E_sh=0, k=6, renormalize=True), 39,
                        "iid"),
    "single_token": (LayerShape(T=1, H=256, I=128, E_pub=8, E_priv=4, E_sh=1, k=2, renormalize=True), 40, "allow"),
    # 512 experts x 104 router tiles: the stable dispatch order across many tiles
    "many_router_tiles_512_experts": (LayerShape(T=13000, H=128, I=128, E_pub=256, E_priv=256, E_sh=0, k=2,
                                                 renormalize=True), 45, "iid"),
    # k > 8 takes the router's sorting-network path; 40 public experts span two chunks
    "k12_two_chunks_pool_softmax": (LayerShape(T=150, H=256, I=128, E_pub=40, E_priv=16, E_sh=0, k=12,
                                               renormalize=False), 44, "iid"),
    # the expert launch's own routing (T <= 128) on a DeepSeek-like layer:
    # pool softmax, 64-expert public pool, shared experts, k = 6
    "small_batch_pool_softmax_shared": (LayerShape(T=96, H=256, I=128, E_pub=64, E_priv=16, E_sh=2, k=6,
                                                   renormalize=False), 50, "iid"),
    # the batch sizes on both sides of the in-launch routing's limit
    "t128_routed_in_launch": (LayerShape(T=128, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True),
                              51, "iid"),
    "t129_cluster_router": (LayerShape(T=129, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True),
                            52, "iid"),
    # H = 384: the routing lanes hold one or two 16-byte pieces of a row
    "h384_small_batch": (LayerShape(T=50, H=384, I=128, E_pub=24, E_priv=8, E_sh=0, k=4, renormalize=True), 53,
                         "iid"),
    # 9 rows of 8 KB per token: a ring of two tokens does not fit the bulk
    # combine's shared memory, so the thread-per-chunk combine runs
    "wide_rows_chunk_combine": (LayerShape(T=40, H=4096, I=128, E_pub=12, E_priv=8, E_sh=1, k=8, renormalize=True),
                                48, "iid"),
    # a 256-expert pool with k = 24 at H = 128: the chunk lists do not fit the
    # cluster router's shared memory, so the chunked router runs the method
    "k24_pool_256_chunked_router": (LayerShape(T=200, H=128, I=128, E_pub=256, E_priv=64, E_sh=0, k=24,
                                               renormalize=True), 47, "iid"),
}


def _setup(name):
    shape, seed, policy = CASES[name]
    if policy == "config":
        w, h, _ = make_layer(shape, seed)
        pol = CONFIGS["tiny"].policy(shape.T)
    else:
        w, h, pol = make_layer(shape, seed, policy=policy)
    return shape, w, h, pol


@pytest.mark.parametrize("name", list(CASES))
def test_parity_with_oracle(name):
    shape, w, h, pol = _setup(name)
    wd, hd, pd = to_device(w, h, pol)
    gpu = run_gpu_layer(shape, wd, hd, pd)
    rep = check_against_oracle(shape, w, h, pol, gpu, name=name)
    check_audit(shape, pol, gpu)
    check_dispatch(shape, h, gpu)
    assert rep["excused"] <= max(2, shape.T // 50), rep["excused"]


def test_expert_loads_0_1_and_152_rows():
    """Empty experts, a single-row expert and a 152-row expert (the shapes of
    the dispatch failures recorded in App. H) in one batch."""
    shape = LayerShape(T=200, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=1, renormalize=True)
    w, h, _ = make_layer(shape, 41)
    u = torch.zeros(shape.H)
    u[7] = 1.0
    hf = h.float()
    hf[:152] = hf[:152] * 0.01 + 8.0 * u          # 152 DENY rows pulled to public expert 3
    hf[152] = hf[152] * 0.01 - 8.0 * u            # one ALLOW row pulled to private expert 2
    rp = w["router_pub"].float()
    rp[3, 7] = 1.0
    rq = w["router_priv"].float()
    rq[2, 7] = -1.0
    w["router_pub"], w["router_priv"] = rp.to(torch.bfloat16), rq.to(torch.bfloat16)
    h = hf.to(torch.bfloat16)
    pol = torch.zeros(shape.T, dtype=torch.uint8)
    pol[152:] = 3                                  # malformed -> DENY
    pol[152] = 1
    wd, hd, pd = to_device(w, h, pol)
    gpu = run_gpu_layer(shape, wd, hd, pd)
    check_against_oracle(shape, w, h, pol, gpu)
    check_audit(shape, pol, gpu)
    check_dispatch(shape, h, gpu)
    counts = gpu["audit"]["route_count"]
    assert counts[3] >= 152 and counts[shape.E_pub + 2] == 1 and (counts == 0).any()


@pytest.mark.parametrize("T", [150, 100])
def test_exact_logit_ties_take_the_lower_id(T):
    """Exactly equal logits (Sec. 3.1 takes the top k after the mask; at an
    exact tie the lower expert id ranks first, the reading both sides
    implement): router rows duplicated in pairs, so every token's selection
    meets ties (at T = 150 the cluster router takes its exact selection path;
    at T = 100 the expert launch routes the tokens itself), and every fifth
    token with a zero hidden state, whose logits are all 0."""
    shape = LayerShape(T=T, H=256, I=128, E_pub=24, E_priv=8, E_sh=0, k=4, renormalize=True)
    w, h, pol = make_layer(shape, 49)
    for key in ("router_pub", "router_priv"):
        r = w[key].clone()
        r[1::2] = r[0::2]  # row 2i + 1 equals row 2i
        w[key] = r
    h = h.clone()
    h[::5] = 0
    wd, hd, pd = to_device(w, h, pol)
    gpu = run_gpu_layer(shape, wd, hd, pd)
    check_against_oracle(shape, w, h, pol, gpu)
    idx = gpu["idx"]
    base = np.where(gpu["tau"][:, None] == 1, shape.E_pub, 0)
    loc = idx - base
    # all-zero tokens: the pool's first k experts, in id order
    assert np.array_equal(loc[::5], np.tile(np.arange(shape.k), (len(loc[::5]), 1)))
    # twins (equal logits): 2i + 1 comes right after 2i, which is missing
    # from the selection only when 2i falls in the k-th place
    for t in range(shape.T):
        sel = list(loc[t])
        for j, e in enumerate(sel):
            if e % 2 == 1:
                assert j > 0 and sel[j - 1] == e - 1, (t, sel)
            elif j < len(sel) - 1:
                assert sel[j + 1] == e + 1, (t, sel)


@pytest.mark.parametrize("T", [96, 300])
def test_stage_by_stage_calls_match_the_oracle(T):
    """The layer run one stage per call on one workspace (route + dispatch,
    gate/up + down, combine): at T <= 128 the cluster router then writes the
    dispatch order itself; above, the dispatch kernel runs.  Outputs, route
    log, audit and dispatch order against the oracle."""
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=T, H=256, I=256, E_pub=24, E_priv=8, E_sh=1, k=4, renormalize=True)
    w, h, pol = make_layer(shape, 54)
    wd, hd, pd = to_device(w, h, pol)
    seq = [pmpe.STAGE_ROUTE | pmpe.STAGE_PERMUTE, pmpe.STAGE_GATEUP | pmpe.STAGE_DOWN, pmpe.STAGE_COMBINE]
    gpu = run_gpu_layer(shape, wd, hd, pd, stage_seq=seq)
    check_against_oracle(shape, w, h, pol, gpu)
    check_audit(shape, pol, gpu)
    check_dispatch(shape, h, gpu)


def test_zero_tokens_is_a_noop():
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=0, H=256, I=128, E_pub=8, E_priv=4, E_sh=0, k=2, renormalize=True)
    w, h, pol = make_layer(LayerShape(1, 256, 128, 8, 4, 0, 2, True), 42)
    wd, _, _ = to_device(w, h, pol)
    desc = pmpe.make_desc(shape, wd, None, None, None, None)
    pmpe.forward_desc(desc)
    torch.cuda.synchronize()


@pytest.mark.parametrize("T", [256, 96])
def test_determinism_recovery_and_batch_invariance(T):
    """Allow -> deny -> allow on the same inputs: the recovery pass is
    bitwise identical to the first allow pass (Sec. 3.3, App. F.3); a row's
    output is bitwise unchanged when other rows' policies flip (App. F.1,
    mixed-policy batches).  The forwards run back to back on one workspace
    with no host synchronisation, with the cluster router (T = 256) and with
    the routing inside the expert launch (T = 96)."""
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=T, H=256, I=256, E_pub=16, E_priv=8, E_sh=1, k=3, renormalize=True)
    w, h, _ = make_layer(shape, 43)
    wd, hd, _ = to_device(w, h, None)
    layer = pmpe.MoeLayer(shape, wd)
    allow = torch.full((shape.T,), 1, dtype=torch.uint8, device="cuda")
    deny = torch.zeros_like(allow)
    o_a = layer.forward(hd, allow).clone()
    o_d = layer.forward(hd, deny).clone()
    o_r = layer.forward(hd, allow).clone()
    assert torch.equal(o_a.view(torch.int16), o_r.view(torch.int16))
    assert not torch.equal(o_a.view(torch.int16), o_d.view(torch.int16))
    mixed = allow.clone()
    mixed[::2] = 0
    o_m = layer.forward(hd, mixed)
    assert torch.equal(o_m[1::2].view(torch.int16), o_a[1::2].view(torch.int16))
    assert torch.equal(o_m[::2].view(torch.int16), o_d[::2].view(torch.int16))


def test_adversarial_hidden_states_cannot_reach_private_pool():
    """Hidden states built to maximise the private router logits, under DENY
    and malformed bytes, execute zero private rows (Sec. 3.1; App. F.1, the adversarial-suite table)."""
    shape = LayerShape(T=128, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True)
    w, _, _ = make_layer(shape, 44)
    d = w["router_priv"].float().sum(0)
    scale = torch.linspace(1, 100, shape.T)[:, None]
    h = (d[None, :] * scale).to(torch.bfloat16)
    g = torch.Generator().manual_seed(44)
    pol = torch.randint(2, 256, (shape.T,), generator=g).to(torch.uint8)
    pol[::3] = 0
    wd, hd, pd = to_device(w, h, pol)
    gpu = run_gpu_layer(shape, wd, hd, pd)
    check_audit(shape, pol, gpu)
    assert gpu["audit"]["route_count"][shape.E_pub:].sum() == 0
    assert gpu["audit"]["exec_rows"][shape.E_pub:].sum() == 0


def _fingerprint(w: dict) -> str:
    """SHA-256 over (name, shape, dtype, raw bytes) of the public tensors."""
    hsh = hashlib.sha256()
    for name in ("router_pub", "gate_pub", "up_pub", "down_pub", "gate_sh", "up_sh", "down_sh"):
        t = w.get(name)
        if t is None:
            continue
        hsh.update(name.encode())
        hsh.update(str(tuple(t.shape)).encode())
        hsh.update(str(t.dtype).encode())
        hsh.update(bf16_bits(t).tobytes())
    return hsh.hexdigest()


def test_public_fingerprint_unchanged():
    """The frozen public weights hash the same before and after the layer
    runs (Sec. 3.2, App. C.1)."""
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=192, H=256, I=128, E_pub=16, E_priv=8, E_sh=2, k=2, renormalize=False)
    w, h, pol = make_layer(shape, 45)
    wd, hd, pd = to_device(w, h, pol)
    before = _fingerprint(wd)
    layer = pmpe.MoeLayer(shape, wd)
    for _ in range(3):
        layer.forward(hd, pd)
    torch.cuda.synchronize()
    assert _fingerprint(wd) == before


def test_invalid_arguments_launch_nothing():
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=64, H=256, I=128, E_pub=8, E_priv=4, E_sh=0, k=2, renormalize=True)
    w, h, pol = make_layer(shape, 46)
    wd, hd, pd = to_device(w, h, pol)
    ws = torch.empty(pmpe.workspace_size(shape), dtype=torch.uint8, device="cuda")
    out = torch.full_like(hd, 7.0)

    def call(s=shape, wts=wd, hid=hd, o=out, wsp=ws):
        return pmpe._lib.pmpe_moe_forward(
            pmpe.ctypes.byref(pmpe.make_desc(s, wts, hid, pd, o, wsp)), None)

    assert call() == pmpe.OK
    torch.cuda.synchronize()
    out.fill_(7.0)
    bad = [
        (dict(s=LayerShape(64, 256, 128, 8, 4, 0, 5, True)), pmpe.ERR_INVALID_ARG),     # k > private pool
        (dict(s=LayerShape(64, 256, 128, 8, 4, 0, 0, True)), pmpe.ERR_INVALID_ARG),     # k = 0
        (dict(s=LayerShape(64, 200, 128, 8, 4, 0, 2, True)), pmpe.ERR_UNSUPPORTED_SHAPE),  # H % 128
        (dict(wts=dict(wd, gate_priv=None)), pmpe.ERR_INVALID_ARG),
        (dict(hid=None), pmpe.ERR_INVALID_ARG),                                            # hidden = NULL
        (dict(wsp=ws[:100]), pmpe.ERR_WORKSPACE),
        (dict(wsp=ws[8:]), pmpe.ERR_UNSUPPORTED_SHAPE),                                    # misaligned
    ]
    for kw, want in bad:
        assert call(**kw) == want, kw
    torch.cuda.synchronize()
    assert torch.all(out == 7.0)


def test_policy_resolve_entry_point_all_bytes():
    from paper_2608_06690_gb300 import pmpe
    pol = torch.arange(256, dtype=torch.int32).to(torch.uint8).cuda()
    tau = pmpe.policy_resolve(pol, 256).cpu().numpy()
    assert np.array_equal(tau, oracle.resolve(np.arange(256, dtype=np.uint8), 256))
    tau0 = pmpe.policy_resolve(None, 50).cpu().numpy()
    assert tau0.sum() == 0


def test_audit_read_reports_status_and_accumulates():
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=64, H=256, I=128, E_pub=8, E_priv=4, E_sh=0, k=2, renormalize=True)
    w, h, pol = make_layer(shape, 47)
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    audit = torch.zeros(pmpe.audit_words(shape.T, shape.E), dtype=torch.int32, device="cuda")
    layer.forward(hd, pd, audit=audit)
    layer.forward(hd, pd, audit=audit)
    a = pmpe.audit_read(audit, shape.T, shape.E)
    assert a["route_count"].sum() == 2 * shape.T * shape.k
    assert np.array_equal(a["exec_rows"], a["route_count"])
    pmpe.audit_reset(audit, shape.T, shape.E)
    a = pmpe.audit_read(audit, shape.T, shape.E)
    assert a["route_count"].sum() == 0
    audit[0] = 1   # a status bit set by a kernel is reported as an error
    with pytest.raises(pmpe.PmpeError):
        pmpe.audit_read(audit, shape.T, shape.E)


def test_persistent_gemm_pair_matches_separate_launches():
    """The forward runs gate/up and down in one persistent launch, down tiles
    waiting for their activation rows; launching the two GEMMs one after the
    other computes every tile the same way, so the outputs are bitwise equal.
    Shared experts and ragged tiles are included."""
    from paper_2608_06690_gb300 import pmpe
    shape = LayerShape(T=700, H=256, I=256, E_pub=16, E_priv=8, E_sh=2, k=3, renormalize=False)
    w, h, pol = make_layer(shape, 45)
    wd, hd, pd = to_device(w, h, pol)
    layer = pmpe.MoeLayer(shape, wd)
    fused = layer.forward(hd, pd).clone()
    split = torch.full_like(fused, float("nan"))
    for st in (pmpe.STAGE_ROUTE | pmpe.STAGE_PERMUTE, pmpe.STAGE_GATEUP, pmpe.STAGE_DOWN, pmpe.STAGE_COMBINE):
        layer.forward(hd, pd, out=split, stages=st)
    torch.cuda.synchronize()
    assert torch.equal(fused.view(torch.int16), split.view(torch.int16))
    # and the pair alone, with its counters cleared by its own launch
    again = torch.full_like(fused, float("nan"))
    layer.forward(hd, pd, out=again, stages=pmpe.STAGE_ROUTE | pmpe.STAGE_PERMUTE)
    layer.forward(hd, pd, out=again, stages=pmpe.STAGE_GATEUP | pmpe.STAGE_DOWN)
    layer.forward(hd, pd, out=again, stages=pmpe.STAGE_COMBINE)
    torch.cuda.synchronize()
    assert torch.equal(fused.view(torch.int16), again.view(torch.int16))


def test_policy_from_requests_matches_oracle_and_feeds_the_layer():
    """Per-request policy bytes expanded on the device equal the oracle's
    expansion bit for bit (random partitions with empty requests and trailing
    tokens, malformed offsets failing closed), and the layer run on them
    equals the layer run on the per-token bytes."""
    from paper_2608_06690_gb300 import pmpe
    g = np.random.default_rng(9)
    for trial in range(40):
        n = int(g.integers(0, 30))
        lens = g.integers(0, 60, size=n)
        T = int(lens.sum() + g.integers(0, 8))
        cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        rp = g.integers(0, 256, size=n).astype(np.uint8)
        rp[g.random(n) < 0.5] = 1
        if trial % 5 == 4 and n >= 2:   # malformed offsets
            cu[int(g.integers(1, n + 1))] = -1 if trial % 10 == 4 else T + 1
        want = oracle.policy_from_requests(rp, cu, T)
        got = pmpe.policy_from_requests(torch.from_numpy(rp).cuda(), torch.from_numpy(cu).cuda(), T)
        torch.cuda.synchronize()
        assert np.array_equal(got.cpu().numpy(), want), (trial, cu, rp)
    shape = LayerShape(T=300, H=256, I=128, E_pub=16, E_priv=8, E_sh=0, k=2, renormalize=True)
    w, h, _ = make_layer(shape, 46)
    lens = np.array([70, 0, 100, 30, 100])
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    rp = np.array([1, 1, 0, 1, 9], np.uint8)
    wd, hd, _ = to_device(w, h, None)
    layer = pmpe.MoeLayer(shape, wd)
    pol_dev = pmpe.policy_from_requests(torch.from_numpy(rp).cuda(), torch.from_numpy(cu).cuda(), shape.T)
    pol_tok = torch.from_numpy(oracle.policy_from_requests(rp, cu, shape.T)).cuda()
    a = layer.forward(hd, pol_dev).clone()
    b = layer.forward(hd, pol_tok).clone()
    torch.cuda.synchronize()
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))
