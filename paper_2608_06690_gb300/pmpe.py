"""ctypes binding over libpmpe.so (the C ABI of include/pmpe.h).

Argument marshalling only: every step of the layer runs in the library's
CUDA kernels.  PyTorch supplies device memory and streams.  If the library
has not been built this module raises on import -- there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

from .inputs import LayerShape

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libpmpe.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with `python -c 'import __graft_entry__ as g; g.build()'`")

_lib = ctypes.CDLL(LIB_PATH)

OK = 0
ERR_INVALID_ARG = -1
ERR_UNSUPPORTED_SHAPE = -2
ERR_WORKSPACE = -3
ERR_CUDA = -4
ERR_TIMEOUT = -5
ERR_DEVICE_STATUS = -6

STATUS_DISPATCH_MISMATCH = 0x1
STATUS_PIPELINE_TIMEOUT = 0x2
STATUS_BAD_EXPERT_ID = 0x4

STAGE_ROUTE = 0x01
STAGE_PERMUTE = 0x02
STAGE_GATEUP = 0x04
STAGE_DOWN = 0x08
STAGE_COMBINE = 0x10
STAGE_ALL = 0x1F

# Kernels one full forward launches: the router/top-k (with the policy
# resolve), one persistent launch that derives the dispatch order and runs the
# gate/up GEMM (rows gathered from the hidden states) and the down GEMM, and
# the combine; no memset.  For small experts (H * I < 2^20, the tiny test
# layer) the dispatch is a kernel of its own: 4.  (Where the persistent grid
# cannot be resident at once, the GEMMs take two launches as well.)
KERNELS_PER_FORWARD = 3


def kernels_per_forward(shape) -> int:
    """Kernels of this library one full forward of `shape` launches on a GPU
    where the persistent expert grid is resident at once (the rule the
    library applies when it launches the forward).  At most 128 tokens (H
    up to 2048, pools of at most 256 experts): a kernel clearing the expert
    launch's counters and the expert launch (routing, dispatch order, both
    GEMMs, combine).  Otherwise the router, the expert GEMMs and the
    combine, plus a dispatch kernel unless the expert launch derives the
    dispatch order (experts of at least 2^20 weights a projection)."""
    if shape.T <= 128 and shape.H <= 2048 and max(shape.E_pub, shape.E_priv) <= 256:
        return 2
    return 3 if shape.H * shape.I >= (1 << 20) else 4
# kernels one private-branch backward launches: the dispatched rows of the
# private experts, dout row gather, the dL/da GEMM, the gate/up recompute GEMM
# with the SwiGLU backward, router gradient, router weight-gradient partials
# and their reduction, the expert weight-gradient GEMM
KERNELS_PER_BACKWARD = 8


def kernels_per_backward_private(shape) -> int:
    """Kernels one private-branch backward launches: KERNELS_PER_BACKWARD,
    plus, for the pool softmax, the pool token lists and the logits GEMM."""
    return KERNELS_PER_BACKWARD + (0 if shape.renormalize else 2)


def kernels_per_backward_input(shape) -> int:
    """Kernels one input-gradient backward launches: the dispatched rows, the
    dout row gather, Z,
    the gate/up recompute with the SwiGLU backward and dA over the routed
    experts (the same three again over the shared experts, if any), the
    router's softmax gradient and the per-token sum; for the pool softmax
    also the pool token lists, the logits GEMM and the router-term GEMM."""
    return 7 + (3 if shape.E_sh > 0 else 0) + (0 if shape.renormalize else 3)


def kernels_per_backward_step(shape) -> int:
    """Kernels one combined backward launches: the dispatched rows, the dout
    row gather, Z, the
    gate/up recompute and dA over the routed experts (the same three over the
    shared experts, if any), the router's dz, its weight-gradient partials
    and their sum, the expert weight-gradient GEMM and the per-token sum; for
    the pool softmax also the pool token lists, the logits GEMM and the
    router-term GEMM."""
    return 9 + (3 if shape.E_sh > 0 else 0) + (0 if shape.renormalize else 3)

EXPORTED = ("pmpe_moe_workspace_size", "pmpe_moe_workspace_layout", "pmpe_audit_words", "pmpe_policy_resolve",
            "pmpe_moe_forward", "pmpe_moe_forward_stages", "pmpe_audit_reset", "pmpe_audit_read",
            "pmpe_status_string", "pmpe_moe_forward_noalloc", "pmpe_selftest_wait_timeout",
            "pmpe_policy_from_requests", "pmpe_moe_backward_workspace_size", "pmpe_moe_backward_private",
            "pmpe_moe_backward_input_workspace_size", "pmpe_moe_backward_input",
            "pmpe_moe_backward_step_workspace_size", "pmpe_moe_backward_step", "pmpe_saved_gu_floats")

# Bytes of the library's static scratch array used by pmpe_moe_forward_noalloc.
STATIC_SCRATCH_BYTES = 32 << 20

_vp = ctypes.c_void_p


class MoeDesc(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int), ("H", ctypes.c_int), ("I", ctypes.c_int), ("E_pub", ctypes.c_int),
                ("E_priv", ctypes.c_int), ("E_shared", ctypes.c_int), ("k", ctypes.c_int),
                ("renormalize", ctypes.c_int),
                ("hidden", _vp), ("policy", _vp),
                ("w_router_pub", _vp), ("w_router_priv", _vp),
                ("w_gate_pub", _vp), ("w_up_pub", _vp), ("w_down_pub", _vp),
                ("w_gate_priv", _vp), ("w_up_priv", _vp), ("w_down_priv", _vp),
                ("w_gate_sh", _vp), ("w_up_sh", _vp), ("w_down_sh", _vp),
                ("out", _vp), ("topk_idx", _vp), ("topk_w", _vp), ("audit", _vp),
                ("workspace", _vp), ("workspace_bytes", ctypes.c_size_t), ("unmasked_control", ctypes.c_int),
                ("saved_gu", _vp)]


class WorkspaceLayout(ctypes.Structure):
    _fields_ = [(n, ctypes.c_size_t) for n in ("total", "tau", "counts", "offsets", "topk_idx", "topk_w", "slot_of", "ticket",
                                                "tok_of_slot", "w_of_slot", "router_rows", "a_perm", "act", "y", "act_sh", "y_sh",
                                                "tile_done", "router_lists", "router_meta", "gemm_ready",
                                                "tile_counts")]


_lib.pmpe_moe_workspace_size.restype = ctypes.c_size_t
_lib.pmpe_moe_workspace_size.argtypes = [ctypes.c_int] * 7
_lib.pmpe_moe_workspace_layout.restype = ctypes.c_int
_lib.pmpe_moe_workspace_layout.argtypes = [ctypes.c_int] * 7 + [ctypes.POINTER(WorkspaceLayout)]
_lib.pmpe_audit_words.restype = ctypes.c_size_t
_lib.pmpe_audit_words.argtypes = [ctypes.c_int, ctypes.c_int]
_lib.pmpe_policy_resolve.restype = ctypes.c_int
_lib.pmpe_policy_resolve.argtypes = [_vp, ctypes.c_int, _vp, _vp]
_lib.pmpe_moe_forward.restype = ctypes.c_int
_lib.pmpe_moe_forward.argtypes = [ctypes.POINTER(MoeDesc), _vp]
_lib.pmpe_moe_forward_stages.restype = ctypes.c_int
_lib.pmpe_moe_forward_stages.argtypes = [ctypes.POINTER(MoeDesc), ctypes.c_uint, _vp]
_lib.pmpe_moe_forward_noalloc.restype = ctypes.c_int
_lib.pmpe_moe_forward_noalloc.argtypes = [ctypes.POINTER(MoeDesc), _vp]
_lib.pmpe_moe_backward_workspace_size.restype = ctypes.c_size_t
_lib.pmpe_moe_backward_workspace_size.argtypes = [ctypes.c_int] * 7
_lib.pmpe_moe_backward_private.restype = ctypes.c_int
_lib.pmpe_moe_backward_private.argtypes = [ctypes.POINTER(MoeDesc), _vp, _vp, _vp, _vp, _vp, _vp, ctypes.c_size_t, _vp]
_lib.pmpe_moe_backward_input_workspace_size.restype = ctypes.c_size_t
_lib.pmpe_moe_backward_input_workspace_size.argtypes = [ctypes.c_int] * 7
_lib.pmpe_moe_backward_input.restype = ctypes.c_int
_lib.pmpe_moe_backward_input.argtypes = [ctypes.POINTER(MoeDesc), _vp, _vp, _vp, ctypes.c_size_t, _vp]
_lib.pmpe_moe_backward_step_workspace_size.restype = ctypes.c_size_t
_lib.pmpe_moe_backward_step_workspace_size.argtypes = [ctypes.c_int] * 7
_lib.pmpe_moe_backward_step.restype = ctypes.c_int
_lib.pmpe_moe_backward_step.argtypes = [ctypes.POINTER(MoeDesc)] + [_vp] * 7 + [ctypes.c_size_t, _vp]
_lib.pmpe_saved_gu_floats.restype = ctypes.c_size_t
_lib.pmpe_saved_gu_floats.argtypes = [ctypes.c_int] * 4
_lib.pmpe_policy_from_requests.restype = ctypes.c_int
_lib.pmpe_policy_from_requests.argtypes = [_vp, _vp, ctypes.c_int, ctypes.c_int, _vp, _vp]
_lib.pmpe_selftest_wait_timeout.restype = ctypes.c_int
_lib.pmpe_selftest_wait_timeout.argtypes = [_vp, ctypes.c_int, _vp]
_lib.pmpe_audit_reset.restype = ctypes.c_int
_lib.pmpe_audit_reset.argtypes = [_vp, ctypes.c_int, ctypes.c_int, _vp]
_lib.pmpe_audit_read.restype = ctypes.c_int
_lib.pmpe_audit_read.argtypes = [_vp, ctypes.c_int, ctypes.c_int, _vp, _vp, ctypes.c_int]
_lib.pmpe_status_string.restype = ctypes.c_char_p
_lib.pmpe_status_string.argtypes = [ctypes.c_int]


class PmpeError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: {status_string(code)} ({code})")
        self.code = code


def status_string(code: int) -> str:
    return _lib.pmpe_status_string(code).decode()


def _check(code: int, what: str):
    if code != OK:
        raise PmpeError(code, what)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def workspace_size(s: LayerShape) -> int:
    return int(_lib.pmpe_moe_workspace_size(s.T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k))


def workspace_layout(s: LayerShape) -> dict:
    L = WorkspaceLayout()
    _check(_lib.pmpe_moe_workspace_layout(s.T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k, ctypes.byref(L)),
           "pmpe_moe_workspace_layout")
    return {n: int(getattr(L, n)) for n, _ in WorkspaceLayout._fields_}


def audit_words(T: int, E: int) -> int:
    return int(_lib.pmpe_audit_words(T, E))


def audit_fields(words: np.ndarray, T: int, E: int) -> dict:
    """Split an audit buffer read back to the host into its named counters."""
    a = np.asarray(words, dtype=np.uint32)
    return dict(status=int(a[0]), shared_rows=int(a[1]), route_count=a[2:2 + E], exec_rows=a[2 + E:2 + 2 * E],
                exec_tiles=a[2 + 2 * E:2 + 3 * E], route_priv_rows=a[2 + 3 * E:2 + 3 * E + T],
                exec_priv_rows=a[2 + 3 * E + T:2 + 3 * E + 2 * T])


def private_gradient_shapes(s: LayerShape) -> dict:
    """Shapes of the gradients the private-branch backward writes: the
    private router and the private experts' gate, up and down weights, the
    only parameters trained (G2, Sec. 2.2).  No public parameter has one."""
    return {"d_router": (s.E_priv, s.H), "d_gate": (s.E_priv, s.I, s.H), "d_up": (s.E_priv, s.I, s.H),
            "d_down": (s.E_priv, s.H, s.I)}


def policy_from_requests(req_policy, cu_seqlens, T: int, out=None, stream=None):
    """Per-token policy bytes (uint8 [T], device) from one byte per request
    and the requests' cumulative token offsets (int32 [n+1], device);
    fail-closed on malformed offsets."""
    if out is None:
        out = torch.empty(T, dtype=torch.uint8, device="cuda")
    n = cu_seqlens.numel() - 1
    _check(_lib.pmpe_policy_from_requests(_ptr(req_policy), _ptr(cu_seqlens), n, T, _ptr(out), _stream(stream)),
           "pmpe_policy_from_requests")
    return out


def policy_resolve(policy, T: int, tau=None, stream=None):
    """tau[t] = (policy[t] == 0x01) on the device; policy None = all DENY."""
    if tau is None:
        tau = torch.empty(T, dtype=torch.uint8, device="cuda")
    _check(_lib.pmpe_policy_resolve(_ptr(policy), T, _ptr(tau), _stream(stream)), "pmpe_policy_resolve")
    return tau


def audit_reset(audit, T: int, E: int, stream=None):
    _check(_lib.pmpe_audit_reset(_ptr(audit), T, E, _stream(stream)), "pmpe_audit_reset")


def audit_read(audit, T: int, E: int, stream=None, timeout_ms: int = 10000, check_status: bool = True) -> dict:
    host = torch.empty(audit_words(T, E), dtype=torch.int32).pin_memory()
    rc = _lib.pmpe_audit_read(_ptr(audit), T, E, ctypes.c_void_p(host.data_ptr()), _stream(stream), timeout_ms)
    if rc == ERR_DEVICE_STATUS and not check_status:
        rc = OK
    _check(rc, "pmpe_audit_read")
    return audit_fields(host.numpy().view(np.uint32).copy(), T, E)


def selftest_wait_timeout(status, limit_us: int, stream=None):
    """Enqueue the bounded-wait self-test: a barrier wait that can never
    complete expires after ``limit_us`` microseconds and ORs
    STATUS_PIPELINE_TIMEOUT into the device word ``status[0]``."""
    _check(_lib.pmpe_selftest_wait_timeout(_ptr(status), int(limit_us), _stream(stream)),
           "pmpe_selftest_wait_timeout")


def make_desc(s: LayerShape, weights: dict, hidden, policy, out, workspace, topk_idx=None, topk_w=None,
              audit=None, unmasked_control: bool = False, saved_gu=None) -> MoeDesc:
    """Fill the C descriptor from torch tensors (device pointers only)."""
    W = weights
    return MoeDesc(s.T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k, int(bool(s.renormalize)),
                   _ptr(hidden), _ptr(policy),
                   _ptr(W["router_pub"]), _ptr(W["router_priv"]),
                   _ptr(W["gate_pub"]), _ptr(W["up_pub"]), _ptr(W["down_pub"]),
                   _ptr(W["gate_priv"]), _ptr(W["up_priv"]), _ptr(W["down_priv"]),
                   _ptr(W.get("gate_sh")), _ptr(W.get("up_sh")), _ptr(W.get("down_sh")),
                   _ptr(out), _ptr(topk_idx), _ptr(topk_w), _ptr(audit),
                   _ptr(workspace), 0 if workspace is None else workspace.numel() * workspace.element_size(),
                   int(bool(unmasked_control)), _ptr(saved_gu))


def forward_desc(desc: MoeDesc, stages: int = STAGE_ALL, stream=None):
    """Enqueue the layer (or a subset of its stages) for a prepared descriptor."""
    if stages == STAGE_ALL:
        rc = _lib.pmpe_moe_forward(ctypes.byref(desc), _stream(stream))
    else:
        rc = _lib.pmpe_moe_forward_stages(ctypes.byref(desc), stages, _stream(stream))
    _check(rc, "pmpe_moe_forward")


class Workspace:
    """A device scratch buffer that grows on demand; layers that run one after
    another on the same stream can share one."""

    def __init__(self, device="cuda"):
        self.device = torch.device(device)
        self._buf = None

    def get(self, nbytes: int) -> torch.Tensor:
        if self._buf is None or self._buf.numel() < nbytes:
            self._buf = torch.empty(max(nbytes, 1), dtype=torch.uint8, device=self.device)
        return self._buf


class MoeLayer:
    """One policy-masked MoE layer with its weights resident on the GPU and
    a reusable workspace.  ``forward`` enqueues the C-ABI call on the
    current stream and returns the output tensor."""

    def __init__(self, shape: LayerShape, weights: dict, device="cuda", workspace: "Workspace | None" = None):
        self.shape = shape
        self.weights = weights
        self.device = torch.device(device)
        self._ws = workspace if workspace is not None else Workspace(self.device)
        self._bws = None
        self._route_out = (None, None)  # the last forward's caller-owned route outputs
        self._saved_gu = None           # the last forward's saved G | U, when it saved them
        self._saved_buf = None

    def workspace(self, T: int) -> torch.Tensor:
        return self._ws.get(workspace_size(self._shape_T(T)))

    def _shape_T(self, T: int) -> LayerShape:
        s = self.shape
        return LayerShape(T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k, s.renormalize)

    def forward(self, hidden, policy, out=None, topk_idx=None, topk_w=None, audit=None, stages=STAGE_ALL,
                stream=None, unmasked_control: bool = False, save_for_backward: bool = False):
        """Enqueue the layer on ``stream`` (default: the current stream).
        ``unmasked_control`` runs the paper's soft-router control instead of
        the method: routing over the concatenated pool without the hard mask.
        ``save_for_backward`` also keeps the gate and up accumulators of the
        routed rows and the shared experts (FP32, owned by the layer), which
        the backward calls after this forward then read instead of
        recomputing them."""
        T = hidden.shape[0]
        s = self._shape_T(T)
        assert hidden.is_contiguous() and hidden.dtype == torch.bfloat16 and hidden.shape == (T, s.H)
        if policy is not None:
            assert policy.dtype == torch.uint8 and policy.numel() == T and policy.is_contiguous()
        if out is None:
            out = torch.empty_like(hidden)
        saved = None
        if save_for_backward:
            n = _lib.pmpe_saved_gu_floats(T, s.I, s.E_sh, s.k)
            if self._saved_buf is None or self._saved_buf.numel() < n:
                self._saved_buf = torch.empty(max(n, 4), dtype=torch.float32, device=hidden.device)
            saved = self._saved_buf
        desc = make_desc(s, self.weights, hidden, policy, out, self.workspace(T), topk_idx, topk_w, audit,
                         unmasked_control, saved)
        forward_desc(desc, stages, stream)
        self._route_out = (topk_idx, topk_w)
        self._saved_gu = saved
        return out

    def backward_private(self, hidden, policy, dout, topk_idx=None, topk_w=None, stream=None) -> dict:
        """Gradients of sum(dout * out) with respect to the private parameters
        (router, gate, up, down; FP32) for the forward just run with the same
        hidden states and policy on the same stream (its workspace holds the
        route and the activations; the route outputs default to those that
        forward wrote).  The public parameters get none."""
        T = hidden.shape[0]
        s = self._shape_T(T)
        assert dout.is_contiguous() and dout.dtype == torch.bfloat16 and dout.shape == (T, s.H)
        dev = hidden.device
        g = {n: torch.empty(shp, dtype=torch.float32, device=dev) for n, shp in private_gradient_shapes(s).items()}
        nb = _lib.pmpe_moe_backward_workspace_size(s.T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k)
        if nb == 0:
            raise PmpeError(ERR_UNSUPPORTED_SHAPE, "pmpe_moe_backward_workspace_size")
        if self._bws is None or self._bws.numel() < nb:
            self._bws = torch.empty(nb, dtype=torch.uint8, device=dev)
        bws = self._bws
        if topk_idx is None and topk_w is None:
            topk_idx, topk_w = self._route_out
        # the descriptor's output pointer is never written by the backward
        desc = make_desc(s, self.weights, hidden, policy, dout, self.workspace(T), topk_idx, topk_w,
                         saved_gu=self._saved_gu)
        _check(_lib.pmpe_moe_backward_private(ctypes.byref(desc), _ptr(dout), _ptr(g["d_router"]), _ptr(g["d_gate"]),
                                              _ptr(g["d_up"]), _ptr(g["d_down"]), _ptr(bws), bws.numel(),
                                              _stream(stream)), "pmpe_moe_backward_private")
        return g

    def backward(self, hidden, policy, dout, topk_idx=None, topk_w=None, stream=None):
        """Both backward results of the forward just run with the same hidden
        states and policy on the same stream, in one pass: the private
        parameters' gradients (as backward_private) and the gradient of the
        hidden states (as backward_input), each bitwise as those calls give."""
        T = hidden.shape[0]
        s = self._shape_T(T)
        assert dout.is_contiguous() and dout.dtype == torch.bfloat16 and dout.shape == (T, s.H)
        dev = hidden.device
        g = {n: torch.empty(shp, dtype=torch.float32, device=dev) for n, shp in private_gradient_shapes(s).items()}
        d_hidden = torch.empty((T, s.H), dtype=torch.float32, device=dev)
        nb = _lib.pmpe_moe_backward_step_workspace_size(s.T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k)
        if nb == 0:
            raise PmpeError(ERR_UNSUPPORTED_SHAPE, "pmpe_moe_backward_step_workspace_size")
        if self._bws is None or self._bws.numel() < nb:
            self._bws = torch.empty(nb, dtype=torch.uint8, device=dev)
        bws = self._bws
        if topk_idx is None and topk_w is None:
            topk_idx, topk_w = self._route_out
        desc = make_desc(s, self.weights, hidden, policy, dout, self.workspace(T), topk_idx, topk_w,
                         saved_gu=self._saved_gu)
        _check(_lib.pmpe_moe_backward_step(ctypes.byref(desc), _ptr(dout), _ptr(g["d_router"]), _ptr(g["d_gate"]),
                                           _ptr(g["d_up"]), _ptr(g["d_down"]), _ptr(d_hidden), _ptr(bws),
                                           bws.numel(), _stream(stream)), "pmpe_moe_backward_step")
        return g, d_hidden

    def backward_input(self, hidden, policy, dout, topk_idx=None, topk_w=None, stream=None) -> torch.Tensor:
        """Gradient of sum(dout * out) with respect to the hidden states [T, H]
        (FP32), through the frozen layer, for the forward just run with the
        same hidden states and policy on the same stream: the routed experts
        of each token's pool, the shared experts and that pool's router."""
        T = hidden.shape[0]
        s = self._shape_T(T)
        assert dout.is_contiguous() and dout.dtype == torch.bfloat16 and dout.shape == (T, s.H)
        dev = hidden.device
        d_hidden = torch.empty((T, s.H), dtype=torch.float32, device=dev)
        nb = _lib.pmpe_moe_backward_input_workspace_size(s.T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k)
        if nb == 0:
            raise PmpeError(ERR_UNSUPPORTED_SHAPE, "pmpe_moe_backward_input_workspace_size")
        if self._bws is None or self._bws.numel() < nb:
            self._bws = torch.empty(nb, dtype=torch.uint8, device=dev)
        bws = self._bws
        if topk_idx is None and topk_w is None:
            topk_idx, topk_w = self._route_out
        desc = make_desc(s, self.weights, hidden, policy, dout, self.workspace(T), topk_idx, topk_w,
                         saved_gu=self._saved_gu)
        _check(_lib.pmpe_moe_backward_input(ctypes.byref(desc), _ptr(dout), _ptr(d_hidden), _ptr(bws), bws.numel(),
                                            _stream(stream)), "pmpe_moe_backward_input")
        return d_hidden
