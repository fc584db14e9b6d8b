"""CPU oracle for the DO-loss hot path (test infrastructure only).

A plain, single-threaded C statement of the paper's definitions in double
precision (``doloss_oracle.c``), wrapped here with ctypes over numpy arrays.
Only the tests, the package smoke check and the benchmark's CPU-baseline leg
use it; the product path never imports it.  It shares no code with the CUDA
library.

Each function works on one problem (one layer) and cites the passage of
"Function Over Form: Distributional Orthogonalization in Mixture-of-Experts"
that it follows in the C source.  Pins that tie every function to something
other than itself live in ``tests/test_oracle.py``; no function here is
"parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "doloss_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

GATE_SIGMOID_NORM = 0
GATE_SOFTMAX = 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, no fast-math) into oracle/_build."""
    os.makedirs(_BUILD, exist_ok=True)
    fresh = os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)
    if fresh and not force:
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P, I64, I32, D = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_double
        sig = {
            "oracle_select": ([P, I64, I32, I32, P], None),
            "oracle_pack": ([P, I64, I32, P], None),
            "oracle_counts": ([P, I64, I32, P], None),
            "oracle_hamming": ([P, I64, I64, I32, P], None),
            "oracle_hamming_bits": ([P, I64, I32, P], None),
            "oracle_gate": ([P, I64, I32, I32, P], None),
            "oracle_direction": ([P, P, I64, I64, I32, I32, P], None),
            "oracle_loss": ([P, P, I32, I64, I32, D], D),
            "oracle_dloss_dp": ([P, P, I64, I64, I32, I64, I32, D, P], None),
            "oracle_gate_backward": ([P, P, I64, I64, I32, I32, D, P], None),
            "oracle_origin_do": ([P, I32], I64),
            "oracle_forward_backward": ([P, I64, I32, I32, I32, D, D, P, P, P, P, P, P], ctypes.c_int),
            "oracle_route": ([P, I64, I32, I32, I32, P, P], None),
            "oracle_dispatch": ([P, I64, I32, I32, P, P, P], None),
            "oracle_bf16_to_double": ([P, I64, P], None),
            "oracle_direction_mode": ([P, P, I64, I64, I32, I32, I32, P], None),
            "oracle_route_backward": ([P, P, P, I64, I32, I32, I32, P], None),
            "oracle_router_logits": ([P, P, I64, I32, I32, P], None),
            "oracle_router_grad": ([P, P, P, I64, I32, I32, P, P], None),
        }
        for name, (args, res) in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
        return lib


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a, a.ctypes.data


def select(z, k):
    """Top-K load bits f [T,E] uint8 (Sec. 3.1.1, Eq. 1)."""
    z, pz = _c(z, np.float32)
    T, E = z.shape
    f = np.empty((T, E), np.uint8)
    _load().oracle_select(pz, T, E, k, f.ctypes.data)
    return f


def pack(f):
    """Signatures [E, ceil(T/32)] uint32 from f [T,E]."""
    f, pf = _c(f, np.uint8)
    T, E = f.shape
    bits = np.empty((E, (T + 31) // 32), np.uint32)
    _load().oracle_pack(pf, T, E, bits.ctypes.data)
    return bits


def counts(f):
    f, pf = _c(f, np.uint8)
    T, E = f.shape
    n = np.empty(E, np.int32)
    _load().oracle_counts(pf, T, E, n.ctypes.data)
    return n


def hamming(f, t0=0, t1=None):
    """G_ij = sum_t |f_it - f_jt| over tokens [t0, t1) (Eq. gij_cij)."""
    f, pf = _c(f, np.uint8)
    T, E = f.shape
    t1 = T if t1 is None else t1
    D = np.zeros((E, E), np.int32)
    _load().oracle_hamming(pf, t0, t1, E, D.ctypes.data)
    return D


def hamming_bits(bits, T):
    bits, pb = _c(bits, np.uint32)
    E = bits.shape[0]
    D = np.empty((E, E), np.int32)
    _load().oracle_hamming_bits(pb, T, E, D.ctypes.data)
    return D


def gate(z, gate_kind=GATE_SIGMOID_NORM):
    z, pz = _c(z, np.float32)
    T, E = z.shape
    p = np.empty((T, E), np.float64)
    _load().oracle_gate(pz, T, E, gate_kind, p.ctypes.data)
    return p


def direction(z, f, gate_kind=GATE_SIGMOID_NORM, t0=0, t1=None):
    """C_ij = sum_t p_it (f_it - f_jt) over tokens [t0, t1) (Eq. gij_cij)."""
    z, pz = _c(z, np.float32)
    f, pf = _c(f, np.uint8)
    T, E = z.shape
    t1 = T if t1 is None else t1
    C = np.zeros((E, E), np.float64)
    _load().oracle_direction(pz, pf, t0, t1, E, gate_kind, C.ctypes.data)
    return C


def loss(D, C, m, k, d_scale=1.0):
    """L_DO = 1/(m^2 k) sum_ij (d_scale D_ij) C_ij (Eq. do_loss / global_do)."""
    D, pD = _c(D, np.int32)
    C, pC = _c(C, np.float64)
    return float(_load().oracle_loss(pD, pC, D.shape[0], m, k, d_scale))


def dloss_dp(D, f, m, k, d_scale=1.0, t0=0, t1=None):
    """dL/dp [T,E] float64 with G and F held constant (Sec. 3.1.3)."""
    D, pD = _c(D, np.int32)
    f, pf = _c(f, np.uint8)
    T, E = f.shape
    t1 = T if t1 is None else t1
    g = np.zeros((T, E), np.float64)
    _load().oracle_dloss_dp(pD, pf, t0, t1, E, m, k, d_scale, g.ctypes.data)
    return g


def gate_backward(z, g, gate_kind=GATE_SIGMOID_NORM, grad_scale=1.0, t0=0, t1=None):
    z, pz = _c(z, np.float32)
    g, pg = _c(g, np.float64)
    T, E = z.shape
    t1 = T if t1 is None else t1
    dz = np.zeros((T, E), np.float64)
    _load().oracle_gate_backward(pz, pg, t0, t1, E, gate_kind, grad_scale, dz.ctypes.data)
    return dz


def origin_do(D):
    D, pD = _c(D, np.int32)
    return int(_load().oracle_origin_do(pD, D.shape[0]))


def forward_backward(z, k, gate_kind=GATE_SIGMOID_NORM, d_scale=1.0, grad_scale=1.0,
                     with_grad=True):
    """Whole path for one problem z [T,E] fp32.

    Returns dict(bits [E,W] u32, counts [E] i32, D [E,E] i32, loss float,
    origin_do int, dz [T,E] float64 or None)."""
    z, pz = _c(z, np.float32)
    T, E = z.shape
    bits = np.empty((E, (T + 31) // 32), np.uint32)
    n = np.empty(E, np.int32)
    D = np.empty((E, E), np.int32)
    lossv = ctypes.c_double(0.0)
    odo = ctypes.c_int64(0)
    dz = np.empty((T, E), np.float64) if with_grad else None
    rc = _load().oracle_forward_backward(
        pz, T, E, k, gate_kind, d_scale, grad_scale, bits.ctypes.data, n.ctypes.data,
        D.ctypes.data, ctypes.addressof(lossv), ctypes.addressof(odo),
        dz.ctypes.data if dz is not None else None)
    if rc != 0:
        raise MemoryError("oracle_forward_backward ran out of host memory")
    return dict(bits=bits, counts=n, D=D, loss=lossv.value, origin_do=odo.value, dz=dz)


def route(z, k, gate_kind=GATE_SIGMOID_NORM):
    """Chosen experts ids [T,k] int32 (selection order) and their re-normalized
    weights combine [T,k] float64 (Sec. 3.1.1)."""
    z, pz = _c(z, np.float32)
    T, E = z.shape
    ids = np.empty((T, k), np.int32)
    comb = np.empty((T, k), np.float64)
    _load().oracle_route(pz, T, E, k, gate_kind, ids.ctypes.data, comb.ctypes.data)
    return ids, comb


def dispatch(ids, E):
    """Expert-grouped order of the (token, choice) pairs: offsets [E+1],
    rows [T*k] (token of each row), pos [T,k] (row of each pair)."""
    ids, pi = _c(ids, np.int32)
    T, k = ids.shape
    offsets = np.empty(E + 1, np.int32)
    rows = np.empty(T * k, np.int32)
    pos = np.empty((T, k), np.int32)
    _load().oracle_dispatch(pi, T, E, k, offsets.ctypes.data, rows.ctypes.data, pos.ctypes.data)
    return offsets, rows, pos


def bf16_to_double(h):
    """Exact values of bf16 bit patterns (uint16 array)."""
    h, ph = _c(h, np.uint16)
    out = np.empty(h.shape, np.float64)
    _load().oracle_bf16_to_double(ph, h.size, out.ctypes.data)
    return out


def router_logits(X, Wr):
    """z [T,E] float64 = X Wr^T for bf16 bit patterns X [T,H], Wr [E,H] (uint16)."""
    X, px = _c(X, np.uint16)
    Wr, pw = _c(Wr, np.uint16)
    T, H = X.shape
    E = Wr.shape[0]
    z = np.empty((T, E), np.float64)
    _load().oracle_router_logits(px, pw, T, H, E, z.ctypes.data)
    return z


def router_grad(X, Wr, dz, with_dx=False):
    """dW [E,H] (and dX [T,H]) float64 of z = X Wr^T for the upstream dz [T,E]."""
    X, px = _c(X, np.uint16)
    Wr, pw = _c(Wr, np.uint16)
    dz, pd = _c(dz, np.float64)
    T, H = X.shape
    E = Wr.shape[0]
    dW = np.empty((E, H), np.float64)
    dX = np.empty((T, H), np.float64) if with_dx else None
    _load().oracle_router_grad(px, pw, pd, T, H, E, dW.ctypes.data,
                               dX.ctypes.data if dX is not None else None)
    return (dW, dX) if with_dx else dW


def direction_mode(z, f, gate_kind=GATE_SIGMOID_NORM, mode=0):
    """C_ij with the dense p (mode 0, the path's reading) or the re-normalized
    top-K weights (mode 1)."""
    z, pz = _c(z, np.float32)
    f, pf = _c(f, np.uint8)
    T, E = z.shape
    C = np.zeros((E, E), np.float64)
    _load().oracle_direction_mode(pz, pf, 0, T, E, gate_kind, mode, C.ctypes.data)
    return C


def route_backward(z, ids, g, gate_kind=GATE_SIGMOID_NORM):
    """dz [T,E] float64: the gradient of the combine weights to the logits for
    the upstream gradient g [T,k] of the weights."""
    z, pz = _c(z, np.float32)
    ids, pi = _c(ids, np.int32)
    g, pg = _c(g, np.float64)
    T, E = z.shape
    k = ids.shape[1]
    dz = np.empty((T, E), np.float64)
    _load().oracle_route_backward(pz, pi, pg, T, E, k, gate_kind, dz.ctypes.data)
    return dz
