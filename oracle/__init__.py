"""ctypes wrapper over the CPU oracle in ``pmpe_oracle.c``.

TEST INFRASTRUCTURE ONLY: the slow, obviously-correct definition of the
policy-masked sparse-MoE layer forward (arXiv 2608.06690, Sec. 3.1 Eq. 4 and
App. B.1) that the GPU path is checked against.  Only ``tests/``, the smoke
check and the benchmark's CPU-baseline leg may import this package.  It
shares no code with the CUDA library and imports nothing from it.

Parity status per function (what pins it is in ``tests/test_oracle.py``):
  resolve       exhaustive over all 256 byte values + NULL
  route         brute-force sort, closed forms (one-hot rows, equal logits)
  expert        textbook SwiGLU MLP via torch.nn.functional (fp64)
  forward       reduces to a dense MLP (E_pool = k = 1, shared weights), audit
                invariants, hand-worked golden fixture
  permute       brute-force sort by (expert, token, rank)
  logits        numpy float64 matmul rounded to fp32 under the mask; its
                sorted order reproduces route
  forward_forced  equals forward bitwise when given forward's own routing;
                a swapped selection changes exactly the swapped terms
  bf16_round    torch's float32 -> bfloat16 rounding on float32-exact values
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pmpe_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

_u16p = ctypes.POINTER(ctypes.c_uint16)
_u8p = ctypes.POINTER(ctypes.c_uint8)
_i32p = ctypes.POINTER(ctypes.c_int32)
_u32p = ctypes.POINTER(ctypes.c_uint32)
_f64p = ctypes.POINTER(ctypes.c_double)


class _Layer(ctypes.Structure):
    _fields_ = [
        ("T", ctypes.c_int), ("H", ctypes.c_int), ("I", ctypes.c_int),
        ("E_pub", ctypes.c_int), ("E_priv", ctypes.c_int), ("E_sh", ctypes.c_int), ("k", ctypes.c_int),
        ("renormalize", ctypes.c_int),
        ("hidden", _u16p), ("policy", _u8p),
        ("router_pub", _u16p), ("router_priv", _u16p),
        ("gate_pub", _u16p), ("up_pub", _u16p), ("down_pub", _u16p),
        ("gate_priv", _u16p), ("up_priv", _u16p), ("down_priv", _u16p),
        ("gate_sh", _u16p), ("up_sh", _u16p), ("down_sh", _u16p),
        ("unmasked", ctypes.c_int), ("exact", ctypes.c_int),
    ]


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/liboracle.so`` (gcc, OpenMP if present)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    base = ["gcc", "-O2", "-shared", "-fPIC", "-o", _LIB + ".tmp", _SRC, "-lm"]
    try:
        subprocess.run(base[:2] + ["-fopenmp"] + base[2:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


_lib = None


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        lib.oracle_bf16_round.restype = ctypes.c_uint16
        lib.oracle_bf16_round.argtypes = [ctypes.c_double]
        lib.oracle_bf16_value.restype = ctypes.c_double
        lib.oracle_bf16_value.argtypes = [ctypes.c_uint16]
        lib.oracle_resolve.restype = None
        lib.oracle_resolve.argtypes = [_u8p, ctypes.c_int, _u8p]
        lib.oracle_route.restype = ctypes.c_int
        lib.oracle_route.argtypes = [ctypes.POINTER(_Layer), _i32p, ctypes.c_int, _i32p, _f64p, _f64p, ctypes.c_int]
        lib.oracle_expert.restype = ctypes.c_int
        lib.oracle_expert.argtypes = [ctypes.POINTER(_Layer), ctypes.c_int, ctypes.c_int, _u16p, _f64p]
        lib.oracle_forward.restype = ctypes.c_int
        lib.oracle_forward.argtypes = [ctypes.POINTER(_Layer), _i32p, ctypes.c_int, _u16p, _f64p, _i32p, _f64p,
                                       _f64p, _u32p, _u32p, _u32p, _u32p, _u32p, ctypes.c_int]
        lib.oracle_logits.restype = ctypes.c_int
        lib.oracle_logits.argtypes = [ctypes.POINTER(_Layer), _i32p, ctypes.c_int, _f64p, ctypes.c_int]
        lib.oracle_forward_forced.restype = ctypes.c_int
        lib.oracle_forward_forced.argtypes = [ctypes.POINTER(_Layer), _i32p, ctypes.c_int, _i32p, _u16p, _f64p,
                                              ctypes.c_int]
        lib.oracle_permute.restype = ctypes.c_int
        lib.oracle_permute.argtypes = [_i32p, ctypes.c_int, ctypes.c_int, ctypes.c_int, _u32p, _u32p, _i32p, _i32p]
        _lib = lib
    return _lib


def _bits(x) -> np.ndarray:
    """BF16 tensor / uint16 array -> contiguous uint16 numpy array of the raw bits."""
    if isinstance(x, np.ndarray):
        assert x.dtype == np.uint16
        return np.ascontiguousarray(x)
    import torch
    assert x.dtype == torch.bfloat16, x.dtype
    return x.detach().to("cpu").contiguous().view(torch.int16).numpy().view(np.uint16)


def _ptr(a, typ):
    return None if a is None else a.ctypes.data_as(typ)


class Layer:
    """One layer's inputs as the oracle sees them (BF16 bit arrays on the host).

    ``tensors`` maps names (hidden, router_pub, router_priv, gate_pub, up_pub,
    down_pub, gate_priv, up_priv, down_priv, and optionally gate_sh, up_sh,
    down_sh) to BF16 tensors or uint16 arrays; ``policy`` is a uint8 array of
    T bytes or None (missing metadata).  ``unmasked`` selects the paper's
    soft-router control: routing over the concatenated pool without the hard
    mask (a negative control, not the method).  ``exact`` removes the
    rounding of logits (fp32) and activations (BF16): the smooth function the
    finite-difference pins of the backward differentiate.
    """

    def __init__(self, shape, tensors: dict, policy, unmasked: bool = False, exact: bool = False):
        self.shape = shape
        self._keep = {}
        for name in ("hidden", "router_pub", "router_priv", "gate_pub", "up_pub", "down_pub",
                     "gate_priv", "up_priv", "down_priv", "gate_sh", "up_sh", "down_sh"):
            v = tensors.get(name)
            self._keep[name] = None if v is None else _bits(v)
        if policy is not None:
            if not isinstance(policy, np.ndarray):
                policy = policy.detach().to("cpu").numpy()
            policy = np.ascontiguousarray(policy, dtype=np.uint8)
        self._keep["policy"] = policy
        s = shape
        k = self._keep
        self.c = _Layer(s.T, s.H, s.I, s.E_pub, s.E_priv, s.E_sh, s.k, int(bool(s.renormalize)),
                        _ptr(k["hidden"], _u16p), _ptr(k["policy"], _u8p),
                        _ptr(k["router_pub"], _u16p), _ptr(k["router_priv"], _u16p),
                        _ptr(k["gate_pub"], _u16p), _ptr(k["up_pub"], _u16p), _ptr(k["down_pub"], _u16p),
                        _ptr(k["gate_priv"], _u16p), _ptr(k["up_priv"], _u16p), _ptr(k["down_priv"], _u16p),
                        _ptr(k["gate_sh"], _u16p), _ptr(k["up_sh"], _u16p), _ptr(k["down_sh"], _u16p),
                        int(bool(unmasked)), int(bool(exact)))


def bf16_round(x: float) -> int:
    return int(_load().oracle_bf16_round(float(x)))


def bf16_value(bits: int) -> float:
    return float(_load().oracle_bf16_value(int(bits)))


def bf16_bits_to_f64(a: np.ndarray) -> np.ndarray:
    """uint16 BF16 bits -> float64 values (exact widening)."""
    return (np.asarray(a, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def resolve(policy, T: int) -> np.ndarray:
    tau = np.zeros(T, dtype=np.uint8)
    pol = None if policy is None else np.ascontiguousarray(policy, dtype=np.uint8)
    _load().oracle_resolve(_ptr(pol, _u8p), T, tau.ctypes.data_as(_u8p))
    return tau


def policy_from_requests(req_policy, cu_seqlens, T: int) -> np.ndarray:
    """Per-token policy bytes from one byte per request and the cumulative
    token offsets of the requests (fail-closed on malformed offsets)."""
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    rp = np.ascontiguousarray(req_policy, dtype=np.uint8)
    out = np.zeros(T, dtype=np.uint8)
    _load().oracle_policy_from_requests(_ptr(rp, _u8p), _ptr(cu, _i32p), len(cu) - 1, T, out.ctypes.data_as(_u8p))
    return out


def backward_private(layer: Layer, dout) -> dict:
    """Gradients of sum(dout * out) with respect to the private parameters
    (d_router [E_priv,H], d_gate / d_up [E_priv,I,H], d_down [E_priv,H,I],
    float64), for the routing the forward takes; public parameters get none."""
    s = layer.shape
    d = np.ascontiguousarray(dout, dtype=np.float64).reshape(s.T, s.H)
    r = dict(d_router=np.zeros((s.E_priv, s.H)), d_gate=np.zeros((s.E_priv, s.I, s.H)),
             d_up=np.zeros((s.E_priv, s.I, s.H)), d_down=np.zeros((s.E_priv, s.H, s.I)))
    rc = _load().oracle_backward_private(ctypes.byref(layer.c), d.ctypes.data_as(_f64p),
                                         *(r[n].ctypes.data_as(_f64p) for n in ("d_router", "d_gate", "d_up", "d_down")))
    if rc != 0:
        raise ValueError("oracle_backward_private rejected the layer description")
    return r


def backward_input(layer: Layer, dout) -> np.ndarray:
    """Gradient of sum(dout * out) with respect to the layer's input hidden
    states [T, H] (float64), through the frozen public, private and shared
    weights and the router of each token's pool, for the routing the forward
    takes.  No parameter gets a gradient here."""
    s = layer.shape
    d = np.ascontiguousarray(dout, dtype=np.float64).reshape(s.T, s.H)
    dh = np.zeros((s.T, s.H))
    rc = _load().oracle_backward_input(ctypes.byref(layer.c), d.ctypes.data_as(_f64p), dh.ctypes.data_as(_f64p))
    if rc != 0:
        raise ValueError("oracle_backward_input rejected the layer description")
    return dh


def _token_list(layer: Layer, tokens):
    if tokens is None:
        return None, layer.shape.T
    tl = np.ascontiguousarray(tokens, dtype=np.int32)
    return tl, len(tl)


def route(layer: Layer, tokens=None, nthreads: int = 0):
    """Routing only: (idx [n,k] int32 global ids, w [n,k] f64, gap [n] f64)."""
    tl, n = _token_list(layer, tokens)
    k = layer.shape.k
    idx = np.zeros((n, k), np.int32)
    w = np.zeros((n, k), np.float64)
    gap = np.zeros(n, np.float64)
    rc = _load().oracle_route(ctypes.byref(layer.c), _ptr(tl, _i32p), n, idx.ctypes.data_as(_i32p),
                              w.ctypes.data_as(_f64p), gap.ctypes.data_as(_f64p), nthreads)
    if rc != 0:
        raise ValueError("oracle_route rejected the layer description")
    return idx, w, gap


def expert(layer: Layer, e: int, h_row, shared: bool = False) -> np.ndarray:
    h = _bits(h_row).reshape(-1)
    y = np.zeros(layer.shape.H, np.float64)
    rc = _load().oracle_expert(ctypes.byref(layer.c), e, int(shared), h.ctypes.data_as(_u16p),
                               y.ctypes.data_as(_f64p))
    if rc != 0:
        raise ValueError("oracle_expert rejected its arguments")
    return y


def forward(layer: Layer, tokens=None, nthreads: int = 0) -> dict:
    """Full layer forward over ``tokens`` (None = all T).  Returns a dict with
    out (uint16 BF16 bits [n,H]), out_f64, idx, w, gap, route_count,
    route_priv_rows, exec_rows, exec_priv_rows, shared_rows."""
    tl, n = _token_list(layer, tokens)
    s = layer.shape
    E = s.E_pub + s.E_priv
    r = dict(out=np.zeros((n, s.H), np.uint16), out_f64=np.zeros((n, s.H), np.float64),
             idx=np.zeros((n, s.k), np.int32), w=np.zeros((n, s.k), np.float64), gap=np.zeros(n, np.float64),
             route_count=np.zeros(E, np.uint32), route_priv_rows=np.zeros(n, np.uint32),
             exec_rows=np.zeros(E, np.uint32), exec_priv_rows=np.zeros(n, np.uint32),
             shared_rows=np.zeros(1, np.uint32))
    rc = _load().oracle_forward(ctypes.byref(layer.c), _ptr(tl, _i32p), n,
                                r["out"].ctypes.data_as(_u16p), r["out_f64"].ctypes.data_as(_f64p),
                                r["idx"].ctypes.data_as(_i32p), r["w"].ctypes.data_as(_f64p),
                                r["gap"].ctypes.data_as(_f64p), r["route_count"].ctypes.data_as(_u32p),
                                r["route_priv_rows"].ctypes.data_as(_u32p), r["exec_rows"].ctypes.data_as(_u32p),
                                r["exec_priv_rows"].ctypes.data_as(_u32p), r["shared_rows"].ctypes.data_as(_u32p),
                                nthreads)
    if rc != 0:
        raise ValueError("oracle_forward rejected the layer description")
    return r


def logits(layer: Layer, tokens=None, nthreads: int = 0) -> np.ndarray:
    """Masked logits s = z + m(tau) [n, E] (float64 holding fp32 values;
    -inf outside the pool tau selects), as the routing decision sees them."""
    tl, n = _token_list(layer, tokens)
    E = layer.shape.E_pub + layer.shape.E_priv
    s = np.zeros((n, E), np.float64)
    if _load().oracle_logits(ctypes.byref(layer.c), _ptr(tl, _i32p), n, s.ctypes.data_as(_f64p), nthreads) != 0:
        raise ValueError("oracle_logits rejected the layer description")
    return s


def forward_forced(layer: Layer, idx, tokens=None, nthreads: int = 0):
    """The layer output for a GIVEN routing idx [n, k] (global ids, rank
    order) of the tokens: (out uint16 BF16 bits [n, H], w [n, k])."""
    tl, n = _token_list(layer, tokens)
    s = layer.shape
    ii = np.ascontiguousarray(idx, dtype=np.int32).reshape(n, s.k)
    out = np.zeros((n, s.H), np.uint16)
    w = np.zeros((n, s.k), np.float64)
    rc = _load().oracle_forward_forced(ctypes.byref(layer.c), _ptr(tl, _i32p), n, ii.ctypes.data_as(_i32p),
                                       out.ctypes.data_as(_u16p), w.ctypes.data_as(_f64p), nthreads)
    if rc != 0:
        raise ValueError("oracle_forward_forced rejected its arguments")
    return out, w


def permute(idx: np.ndarray, E: int):
    """(counts [E], offsets [E+1], slot_of [T,k], tok_of_slot [T*k])."""
    idx = np.ascontiguousarray(idx, dtype=np.int32)
    T, k = idx.shape
    counts = np.zeros(E, np.uint32)
    offsets = np.zeros(E + 1, np.uint32)
    slot_of = np.zeros((T, k), np.int32)
    tok_of_slot = np.zeros(T * k, np.int32)
    rc = _load().oracle_permute(idx.ctypes.data_as(_i32p), T, k, E, counts.ctypes.data_as(_u32p),
                                offsets.ctypes.data_as(_u32p), slot_of.ctypes.data_as(_i32p),
                                tok_of_slot.ctypes.data_as(_i32p))
    if rc != 0:
        raise ValueError("expert id out of range")
    return counts, offsets, slot_of, tok_of_slot
