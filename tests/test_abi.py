"""The C ABI without a GPU: the library builds for sm_103a, loads, exports
every function include/pmpe.h declares, and its host-only entry points
(sizes, layout, status text, argument validation) behave as documented.
No call here reaches a CUDA kernel."""
import ctypes
import os
import re
import shutil
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pmpe.h")

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                                reason="no CUDA toolkit to build the library")


@pytest.fixture(scope="module")
def pmpe():
    from paper_2608_06690_gb300 import build
    build.build()
    from paper_2608_06690_gb300 import pmpe as m
    return m


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^PMPE_API\s+[\w\s\*]*?\b(pmpe_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_documented_entry_points():
    names = declared_functions()
    for must in ("pmpe_moe_forward", "pmpe_policy_resolve", "pmpe_audit_read"):
        assert must in names


def test_every_declared_symbol_is_exported(pmpe):
    lib = ctypes.CDLL(pmpe.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(declared_functions()) == set(pmpe.EXPORTED)
    out = subprocess.run(["nm", "-D", "--defined-only", pmpe.LIB_PATH], capture_output=True, text=True).stdout
    exported = sorted(l.split()[-1] for l in out.splitlines() if " T " in l)
    assert exported == declared_functions()


def test_audit_words_and_fields(pmpe):
    import numpy as np
    T, E = 5, 7
    n = pmpe.audit_words(T, E)
    assert n == 2 + 3 * E + 2 * T
    f = pmpe.audit_fields(np.arange(n, dtype=np.uint32), T, E)
    assert f["status"] == 0 and f["shared_rows"] == 1
    assert f["route_count"][0] == 2 and f["exec_priv_rows"][-1] == n - 1


def test_workspace_size_and_layout(pmpe):
    from paper_2608_06690_gb300.inputs import LayerShape
    s = LayerShape(T=4096, H=2048, I=768, E_pub=128, E_priv=32, E_sh=0, k=8, renormalize=True)
    L = pmpe.workspace_layout(s)
    assert pmpe.workspace_size(s) == L["total"]
    R = s.T * s.k
    assert L["a_perm"] % 1024 == 0 and L["act"] % 1024 == 0 and L["y"] % 1024 == 0
    assert L["act"] >= L["a_perm"] + 2 * R * s.H and L["y"] >= L["act"] + 2 * R * s.I
    assert L["total"] >= L["y"] + 2 * R * s.H
    assert L["act_sh"] == 0 and L["y_sh"] == 0
    s2 = LayerShape(T=100, H=256, I=128, E_pub=8, E_priv=4, E_sh=2, k=2, renormalize=False)
    L2 = pmpe.workspace_layout(s2)
    assert L2["y_sh"] >= L2["act_sh"] + 2 * s2.T * s2.E_sh * s2.I
    # every region lies inside the workspace and no two overlap
    for sh, LL in ((s, L), (s2, L2)):
        T, E, R = sh.T, sh.E_pub + sh.E_priv, sh.T * sh.k
        slots = (T + 127) // 128 + 1
        ctas = slots * max((sh.E_pub + 31) // 32, (sh.E_priv + 31) // 32)
        ctas_all = slots * ((sh.E_pub + 31) // 32 + (sh.E_priv + 31) // 32)
        size = dict(tau=T, counts=4 * E, offsets=4 * (E + 1), topk_idx=4 * R, topk_w=4 * R, slot_of=4 * R,
                    ticket=4 * R, tok_of_slot=4 * R, w_of_slot=4 * R, tile_done=4 * slots,
                    router_lists=8 * ctas_all * 128 * sh.k, router_meta=16 * ctas_all * 128,
                    # readiness counters, then the expert kernel's tile and grid-barrier counters
                    gemm_ready=4 * ((R + 127) // 128 + E + (T + 127) // 128 + 6),
                    router_rows=2 * ctas * 128 * sh.H, a_perm=2 * R * sh.H, act=2 * R * sh.I, y=2 * R * sh.H,
                    act_sh=2 * T * sh.E_sh * sh.I, y_sh=2 * T * sh.H if sh.E_sh else 0,
                    tile_counts=4 * E * ((slots + 3) // 4 * 4))
        spans = sorted((LL[n], LL[n] + b, n) for n, b in size.items() if b)
        for (a0, a1, na), (b0, b1, nb) in zip(spans, spans[1:]):
            assert a1 <= b0, (na, nb)
        assert spans[-1][1] <= LL["total"]
        assert LL["router_meta"] % 16 == 0 and LL["router_lists"] % 8 == 0 and LL["router_rows"] % 1024 == 0
        assert LL["tile_done"] == LL["counts"] + 4 * E  # one memset clears these three
        assert LL["gemm_ready"] == LL["tile_done"] + 4 * slots
        gr_end = LL["gemm_ready"] + 4 * ((R + 127) // 128 + E + (T + 127) // 128 + 6)
        assert LL["tile_counts"] % 16 == 0 and gr_end <= LL["tile_counts"] <= gr_end + 12
    assert pmpe.workspace_size(LayerShape(64, 200, 128, 8, 4, 0, 2, True)) == 0    # H % 128
    assert pmpe.workspace_size(LayerShape(64, 256, 128, 8, 4, 0, 9, True)) == 0    # k > pool


def test_status_strings(pmpe):
    assert pmpe.status_string(0) == "ok"
    for c in (-1, -2, -3, -4, -5, -6):
        assert pmpe.status_string(c) not in ("ok", "unknown status")
    assert pmpe.status_string(-99) == "unknown status"


def test_validation_rejects_before_any_cuda_call(pmpe):
    """Invalid descriptors are rejected on the host; with fake (never
    dereferenced) device pointers nothing is launched."""
    from paper_2608_06690_gb300.inputs import LayerShape
    lib = pmpe._lib
    assert lib.pmpe_moe_forward(None, None) == pmpe.ERR_INVALID_ARG

    class Fake:
        def __init__(self, addr):
            self.addr = addr

        def data_ptr(self):
            return self.addr

        def numel(self):
            return 1 << 40

        def element_size(self):
            return 1

    p = Fake(0x10000000)
    W = {n: p for n in ("router_pub", "router_priv", "gate_pub", "up_pub", "down_pub", "gate_priv", "up_priv",
                        "down_priv")}

    def rc(shape, **over):
        args = dict(weights=W, hidden=p, policy=None, out=p, workspace=p)
        args.update(over)
        d = pmpe.make_desc(shape, args["weights"], args["hidden"], args["policy"], args["out"], args["workspace"])
        return lib.pmpe_moe_forward(ctypes.byref(d), None)

    ok = LayerShape(64, 256, 128, 8, 4, 0, 2, True)
    assert rc(LayerShape(64, 256, 128, 8, 4, 0, 5, True)) == pmpe.ERR_INVALID_ARG      # k > E_priv
    assert rc(LayerShape(64, 256, 128, 8, 4, 0, 0, True)) == pmpe.ERR_INVALID_ARG      # k < 1
    assert rc(LayerShape(-1, 256, 128, 8, 4, 0, 2, True)) == pmpe.ERR_INVALID_ARG     # T < 0
    assert rc(LayerShape(64, 192, 128, 8, 4, 0, 2, True)) == pmpe.ERR_UNSUPPORTED_SHAPE  # H % 128
    assert rc(LayerShape(64, 256, 64, 8, 4, 0, 2, True)) == pmpe.ERR_UNSUPPORTED_SHAPE   # I % 128
    assert rc(LayerShape(64, 256, 128, 300, 4, 0, 2, True)) == pmpe.ERR_UNSUPPORTED_SHAPE  # pool > 256
    assert rc(LayerShape(64, 256, 128, 40, 40, 0, 33, True)) == pmpe.ERR_UNSUPPORTED_SHAPE  # k > 32
    assert rc(ok, hidden=None) == pmpe.ERR_INVALID_ARG
    assert rc(ok, out=None) == pmpe.ERR_INVALID_ARG
    assert rc(ok, weights=dict(W, down_priv=None)) == pmpe.ERR_INVALID_ARG
    assert rc(LayerShape(64, 256, 128, 8, 4, 1, 2, True)) == pmpe.ERR_INVALID_ARG      # shared weights missing
    assert rc(ok, hidden=Fake(0x10000008)) == pmpe.ERR_UNSUPPORTED_SHAPE               # not 16-byte aligned
    assert rc(ok, workspace=None) == pmpe.ERR_WORKSPACE
    assert rc(ok, workspace=Fake(0x10000010)) == pmpe.ERR_WORKSPACE                   # not 256-byte aligned
    assert rc(LayerShape(0, 256, 128, 8, 4, 0, 2, True), hidden=None, out=None, workspace=None) == pmpe.OK
    assert lib.pmpe_policy_resolve(None, -1, None, None) == pmpe.ERR_INVALID_ARG
    assert lib.pmpe_policy_resolve(None, 0, None, None) == pmpe.OK
    assert lib.pmpe_audit_reset(None, 4, 4, None) == pmpe.ERR_INVALID_ARG
    assert lib.pmpe_audit_read(None, 4, 4, None, None, 10) == pmpe.ERR_INVALID_ARG
    d = pmpe.make_desc(ok, W, p, None, p, p, saved_gu=Fake(0x10000004))
    assert lib.pmpe_moe_forward(ctypes.byref(d), None) == pmpe.ERR_UNSUPPORTED_SHAPE     # saved G | U misaligned
    d = pmpe.make_desc(ok, W, p, None, p, p)
    d.unmasked_control = 2
    assert lib.pmpe_moe_forward(ctypes.byref(d), None) == pmpe.ERR_INVALID_ARG          # flag is 0 or 1
    d = pmpe.make_desc(LayerShape(64, 256, 128, 256, 256, 0, 8, True), W, p, None, p, p, unmasked_control=True)
    assert lib.pmpe_moe_forward(ctypes.byref(d), None) == pmpe.ERR_UNSUPPORTED_SHAPE     # merge too large
    assert lib.pmpe_policy_from_requests(None, None, 1, 4, None, None) == pmpe.ERR_INVALID_ARG
    assert lib.pmpe_policy_from_requests(p_ptr := ctypes.c_void_p(0x10000000), p_ptr, -1, 4, p_ptr, None) == \
        pmpe.ERR_INVALID_ARG
    assert lib.pmpe_policy_from_requests(None, ctypes.c_void_p(0x10000000), 0, 0, None, None) == pmpe.OK  # T = 0
    assert lib.pmpe_selftest_wait_timeout(None, 1000, None) == pmpe.ERR_INVALID_ARG
    assert lib.pmpe_selftest_wait_timeout(ctypes.c_void_p(0x10000000), 0, None) == pmpe.ERR_INVALID_ARG
    assert lib.pmpe_selftest_wait_timeout(ctypes.c_void_p(0x10000000), 1000001, None) == pmpe.ERR_INVALID_ARG


def test_backward_validation_rejects_before_any_cuda_call(pmpe):
    """The private-branch backward checks its gradient buffers, dout, the
    control flag and its scratch size on the host; fake device pointers are
    never dereferenced."""
    from paper_2608_06690_gb300.inputs import LayerShape
    lib = pmpe._lib
    shape = LayerShape(64, 256, 128, 8, 4, 0, 2, True)
    need = lib.pmpe_moe_backward_workspace_size(64, 256, 128, 8, 4, 0, 2)
    assert need >= 256 and need % 256 == 0
    assert lib.pmpe_moe_backward_workspace_size(64, 192, 128, 8, 4, 0, 2) == 0   # H % 128
    assert lib.pmpe_moe_backward_workspace_size(0, 256, 128, 8, 4, 0, 2) == 256  # empty batch: the floor
    # scratch grows with the routed rows
    assert lib.pmpe_moe_backward_workspace_size(128, 256, 128, 8, 4, 0, 2) > need

    class Fake:
        def __init__(self, addr):
            self.addr = addr

        def data_ptr(self):
            return self.addr

        def numel(self):
            return 1 << 40

        def element_size(self):
            return 1

    p = Fake(0x10000000)
    W = {n: p for n in ("router_pub", "router_priv", "gate_pub", "up_pub", "down_pub", "gate_priv", "up_priv",
                        "down_priv")}
    v = ctypes.c_void_p(p.addr)

    def rc(desc_ok=True, dout=v, grads=(v, v, v, v), bws=v, nbytes=need, unmasked=False):
        d = pmpe.make_desc(shape, W, p, None, p, p, unmasked_control=unmasked)
        return lib.pmpe_moe_backward_private(ctypes.byref(d) if desc_ok else None, dout, *grads, bws, nbytes, None)

    assert rc(desc_ok=False) == pmpe.ERR_INVALID_ARG
    assert rc(dout=None) == pmpe.ERR_INVALID_ARG
    assert rc(dout=ctypes.c_void_p(p.addr + 2)) == pmpe.ERR_INVALID_ARG
    assert rc(grads=(v, None, v, v)) == pmpe.ERR_INVALID_ARG
    assert rc(grads=(v, v, v, ctypes.c_void_p(p.addr + 4))) == pmpe.ERR_INVALID_ARG
    assert rc(unmasked=True) == pmpe.ERR_UNSUPPORTED_SHAPE
    assert rc(bws=None) == pmpe.ERR_WORKSPACE
    assert rc(nbytes=need - 256) == pmpe.ERR_WORKSPACE
    assert rc(bws=ctypes.c_void_p(p.addr + 16)) == pmpe.ERR_WORKSPACE


def test_backward_input_validation_rejects_before_any_cuda_call(pmpe):
    """The input-gradient backward checks dout, d_hidden, the control flag and
    its scratch size on the host; fake device pointers are never dereferenced."""
    from paper_2608_06690_gb300.inputs import LayerShape
    lib = pmpe._lib
    shape = LayerShape(64, 256, 128, 8, 4, 1, 2, True)
    need = lib.pmpe_moe_backward_input_workspace_size(64, 256, 128, 8, 4, 1, 2)
    assert need >= 256 and need % 256 == 0
    assert lib.pmpe_moe_backward_input_workspace_size(64, 192, 128, 8, 4, 1, 2) == 0   # H % 128
    assert lib.pmpe_moe_backward_input_workspace_size(0, 256, 128, 8, 4, 1, 2) == 256  # empty batch: the floor
    # scratch grows with the routed rows and with the shared experts
    assert lib.pmpe_moe_backward_input_workspace_size(128, 256, 128, 8, 4, 1, 2) > need
    assert lib.pmpe_moe_backward_input_workspace_size(64, 256, 128, 8, 4, 2, 2) > need

    class Fake:
        def __init__(self, addr):
            self.addr = addr

        def data_ptr(self):
            return self.addr

        def numel(self):
            return 1 << 40

        def element_size(self):
            return 1

    p = Fake(0x10000000)
    W = {n: p for n in ("router_pub", "router_priv", "gate_pub", "up_pub", "down_pub", "gate_priv", "up_priv",
                        "down_priv", "gate_sh", "up_sh", "down_sh")}
    v = ctypes.c_void_p(p.addr)

    def rc(desc_ok=True, dout=v, dh=v, bws=v, nbytes=need, unmasked=False):
        d = pmpe.make_desc(shape, W, p, None, p, p, unmasked_control=unmasked)
        return lib.pmpe_moe_backward_input(ctypes.byref(d) if desc_ok else None, dout, dh, bws, nbytes, None)

    assert rc(desc_ok=False) == pmpe.ERR_INVALID_ARG
    assert rc(dout=None) == pmpe.ERR_INVALID_ARG
    assert rc(dout=ctypes.c_void_p(p.addr + 2)) == pmpe.ERR_INVALID_ARG
    assert rc(dh=None) == pmpe.ERR_INVALID_ARG
    assert rc(dh=ctypes.c_void_p(p.addr + 4)) == pmpe.ERR_INVALID_ARG
    assert rc(unmasked=True) == pmpe.ERR_UNSUPPORTED_SHAPE
    assert rc(bws=None) == pmpe.ERR_WORKSPACE
    assert rc(nbytes=need - 256) == pmpe.ERR_WORKSPACE
    assert rc(bws=ctypes.c_void_p(p.addr + 16)) == pmpe.ERR_WORKSPACE


def test_backward_step_validation_rejects_before_any_cuda_call(pmpe):
    """The combined backward checks its gradient buffers, dout, d_hidden, the
    control flag and its scratch size on the host; fake device pointers are
    never dereferenced."""
    from paper_2608_06690_gb300.inputs import LayerShape
    lib = pmpe._lib
    shape = LayerShape(64, 256, 128, 8, 4, 1, 2, True)
    need = lib.pmpe_moe_backward_step_workspace_size(64, 256, 128, 8, 4, 1, 2)
    assert need >= 256 and need % 256 == 0
    assert lib.pmpe_moe_backward_step_workspace_size(64, 192, 128, 8, 4, 1, 2) == 0   # H % 128
    assert lib.pmpe_moe_backward_step_workspace_size(0, 256, 128, 8, 4, 1, 2) == 256  # empty batch: the floor
    # it holds the input gradient's scratch and more
    assert need > lib.pmpe_moe_backward_input_workspace_size(64, 256, 128, 8, 4, 1, 2)

    class Fake:
        def __init__(self, addr):
            self.addr = addr

        def data_ptr(self):
            return self.addr

        def numel(self):
            return 1 << 40

        def element_size(self):
            return 1

    p = Fake(0x10000000)
    W = {n: p for n in ("router_pub", "router_priv", "gate_pub", "up_pub", "down_pub", "gate_priv", "up_priv",
                        "down_priv", "gate_sh", "up_sh", "down_sh")}
    v = ctypes.c_void_p(p.addr)

    def rc(desc_ok=True, dout=v, grads=(v, v, v, v), dh=v, bws=v, nbytes=need, unmasked=False):
        d = pmpe.make_desc(shape, W, p, None, p, p, unmasked_control=unmasked)
        return lib.pmpe_moe_backward_step(ctypes.byref(d) if desc_ok else None, dout, *grads, dh, bws, nbytes, None)

    assert rc(desc_ok=False) == pmpe.ERR_INVALID_ARG
    assert rc(dout=None) == pmpe.ERR_INVALID_ARG
    assert rc(grads=(v, None, v, v)) == pmpe.ERR_INVALID_ARG
    assert rc(grads=(v, v, v, ctypes.c_void_p(p.addr + 4))) == pmpe.ERR_INVALID_ARG
    assert rc(dh=None) == pmpe.ERR_INVALID_ARG
    assert rc(dh=ctypes.c_void_p(p.addr + 8)) == pmpe.ERR_INVALID_ARG
    assert rc(unmasked=True) == pmpe.ERR_UNSUPPORTED_SHAPE
    assert rc(bws=None) == pmpe.ERR_WORKSPACE
    assert rc(nbytes=need - 256) == pmpe.ERR_WORKSPACE
    assert rc(bws=ctypes.c_void_p(p.addr + 16)) == pmpe.ERR_WORKSPACE


def test_optimizer_partition_matches_the_papers_trainable_parameter_counts(pmpe):
    """G2 optimizer partition (Sec. 2.2): the backward produces gradients for
    the private router and private experts only, and over the paper's two
    wrapped layers of 16 private experts their sizes add up to the trainable
    parameter counts the paper's model table prints."""
    import json
    from paper_2608_06690_gb300.inputs import LayerShape
    gold = json.load(open(os.path.join(ROOT, "tests", "golden", "trainable_parameters.json")))
    for c in gold["cases"]:
        s = LayerShape(T=1, H=c["H"], I=c["I"], E_pub=64, E_priv=c["E_priv"], E_sh=0, k=6, renormalize=True)
        shapes = pmpe.private_gradient_shapes(s)
        assert set(shapes) == {"d_router", "d_gate", "d_up", "d_down"}
        per_layer = sum(int(np.prod(v)) for v in shapes.values())
        assert c["wrapped_layers"] * per_layer == c["trainable_parameters"], c["model"]
    # the binding has no entry point that could write a public parameter's gradient
    assert not [n for n in pmpe.EXPORTED if "backward" in n and "pub" in n]
