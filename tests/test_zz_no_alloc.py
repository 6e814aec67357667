"""pmpe_moe_forward_noalloc: the forward for callers that cannot allocate
device memory where they run the layer (a plugin whose host owns all device
memory, a serving loop that must not pay cudaMalloc's synchronisation or risk
running out of memory mid-request).  Its scratch is a static device array of
the library instead of a caller workspace.

Checked through the C ABI against the regular entry point, bit for bit (both
run the same kernels on the same inputs), on two calls in a row with
different inputs (the shared array keeps the first call's contents, so the
second call shows that nothing stale leaks through), at a small ragged shape
with a shared expert and at the 64-token decode step of the Qwen3-shaped
layer.  This file is collected last so that a stopping run has already run
every other test."""
import ctypes

import pytest
import torch

from paper_2608_06690_gb300.configs import CONFIGS
from paper_2608_06690_gb300.inputs import LayerShape
from pmpe_testlib import make_layer, to_device

pytestmark = pytest.mark.gpu

SHAPES = {
    "ragged_with_shared_expert": LayerShape(T=200, H=512, I=256, E_pub=16, E_priv=8, E_sh=1, k=4, renormalize=True),
    "qwen3_decode_64_tokens": CONFIGS["qwen3_decode"].shape,
}


def _run(pmpe, entry, shape, wd, hd, pd, workspace=None):
    out = torch.full_like(hd, float("nan"))
    idx = torch.full((shape.T, shape.k), -1, dtype=torch.int32, device="cuda")
    wt = torch.full((shape.T, shape.k), float("nan"), dtype=torch.float32, device="cuda")
    audit = torch.zeros(pmpe.audit_words(shape.T, shape.E), dtype=torch.int32, device="cuda")
    desc = pmpe.make_desc(shape, wd, hd, pd, out, workspace, topk_idx=idx, topk_w=wt, audit=audit)
    rc = entry(ctypes.byref(desc), None)
    torch.cuda.synchronize()
    return rc, out, idx, wt, audit


@pytest.mark.parametrize("name", list(SHAPES))
def test_noalloc_matches_regular_entry_point_bitwise_on_two_calls(name):
    from paper_2608_06690_gb300 import pmpe
    shape = SHAPES[name]
    assert pmpe.workspace_size(shape) <= pmpe.STATIC_SCRATCH_BYTES
    for seed in (71, 72):   # two calls in a row, different inputs and policies
        w, h, pol = make_layer(shape, seed, device="cuda")
        wd, hd, pd = to_device(w, h, pol)
        ws = torch.empty(pmpe.workspace_size(shape), dtype=torch.uint8, device="cuda")
        rc0, out0, idx0, w0, a0 = _run(pmpe, pmpe._lib.pmpe_moe_forward, shape, wd, hd, pd, ws)
        rc1, out1, idx1, w1, a1 = _run(pmpe, pmpe._lib.pmpe_moe_forward_noalloc, shape, wd, hd, pd)
        assert rc0 == pmpe.OK and rc1 == pmpe.OK
        assert torch.equal(out0.view(torch.int16), out1.view(torch.int16)), "outputs differ"
        assert torch.equal(idx0, idx1)
        assert torch.equal(w0.view(torch.int32), w1.view(torch.int32))
        assert torch.equal(a0, a1)
        assert int(a1[0]) == 0  # status word


def test_noalloc_rejects_shapes_beyond_its_scratch():
    from paper_2608_06690_gb300 import pmpe
    big = LayerShape(T=4096, H=2048, I=768, E_pub=128, E_priv=32, E_sh=0, k=8, renormalize=True)
    assert pmpe.workspace_size(big) > pmpe.STATIC_SCRATCH_BYTES
    small = LayerShape(T=8, H=256, I=128, E_pub=8, E_priv=4, E_sh=0, k=2, renormalize=True)
    w, h, pol = make_layer(small, 73)
    wd, _, _ = to_device(w, h, pol)
    hd = torch.zeros((big.T, big.H), dtype=torch.bfloat16, device="cuda")
    out = torch.full_like(hd, 3.0)
    desc = pmpe.make_desc(big, wd, hd, None, out, None)
    assert pmpe._lib.pmpe_moe_forward_noalloc(ctypes.byref(desc), None) == pmpe.ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.all(out == 3.0)
