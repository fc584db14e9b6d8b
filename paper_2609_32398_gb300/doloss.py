"""Python binding of libdoloss (include/doloss.h) over torch CUDA tensors.

Argument marshalling only: every step of the DO-loss path runs in the CUDA
kernels of libdoloss.so.  torch supplies device memory and the current
stream.  There is no CPU fallback: if the library is not built, or a call
fails, these functions raise.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

GATE_SIGMOID_NORM = 0
GATE_SOFTMAX = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libdoloss.so")
_lock = threading.Lock()
_lib = None

EXPORTS = {
    # name: (argtypes, restype)
    "do_signatures": (["p", "i64", "i32", "i32", "i32", "p", "p", "p"], "i32"),
    "do_pairwise_hamming": (["p", "i64", "i32", "i32", "p", "p"], "i32"),
    "do_pairwise_hamming_accumulate": (["p", "i64", "i32", "i32", "p", "p"], "i32"),
    "do_loss_fwd_bwd": (["p", "p", "p", "i64", "i32", "i32", "i32", "i32", "f32", "f32", "p",
                         "p", "p", "p", "sz", "p"], "i32"),
    "do_forward_backward": (["p", "i64", "i32", "i32", "i32", "i32", "f32", "p", "p", "p", "p",
                             "p", "p", "p", "sz", "p"], "i32"),
    "do_workspace_size": (["i64", "i32", "i32", "i32"], "sz"),
    "do_routed_workspace_size": (["i64", "i32", "i32", "i32"], "sz"),
    "do_device_status": (["p", "p"], "i32"),
    "do_forward_backward_host": (["p", "i64", "i32", "i32", "i32", "i32", "f32", "p", "p", "p",
                                  "p", "p", "sz", "p"], "i32"),
    "do_host_buffer_size": (["i64", "i32", "i32", "i32"], "sz"),
    "do_forward_backward_host_async": (["p", "i64", "i32", "i32", "i32", "i32", "f32", "p", "p",
                                        "sz", "p"], "i32"),
    "do_status_string": (["i32"], "str"),
    "do_selftest_wait_limit": (["p", "p"], "i32"),
    "do_forward_backward_static": (["p", "i64", "i32", "i32", "i32", "i32", "f32", "p", "p", "p",
                                    "p", "p", "p", "p", "p"], "i32"),
    "do_routing": (["p", "i64", "i32", "i32", "i32", "i32", "p", "p", "p", "p", "p", "p", "p", "sz",
                    "p"], "i32"),
    "do_routing_workspace_size": (["i64", "i32", "i32", "i32"], "sz"),
    "do_route_backward": (["p", "p", "p", "i64", "i32", "i32", "i32", "i32", "i32", "p", "p", "p"],
                          "i32"),
    "do_accumulate_distances": (["p", "i32", "i32", "p", "p"], "i32"),
    "do_offdiag_variance": (["p", "i64", "i32", "i32", "i32", "p", "p"], "i32"),
    "do_routed_forward": (["p", "i64", "i32", "i32", "i32", "i32", "p", "p", "p", "p", "p", "p", "p",
                           "p", "p", "p", "sz", "p"], "i32"),
    "do_routed_backward": (["p", "i64", "i32", "i32", "i32", "i32", "f32", "f32", "p", "p", "p", "p",
                            "p", "p", "p", "p", "sz", "p"], "i32"),
    "do_forward_backward_routed": (["p", "i64", "i32", "i32", "i32", "i32", "f32", "p", "p", "p",
                                    "p", "p", "p", "p", "p", "p", "p", "p", "p", "sz", "p"], "i32"),
    "do_maxvio": (["p", "p", "i32", "i32", "i32", "p", "p", "p", "p"], "i32"),
    "do_router_backward": (["p", "p", "p", "i64", "i32", "i32", "i32", "p", "p", "p", "sz", "p"],
                           "i32"),
    "do_router_backward_workspace_size": (["i64", "i32", "i32", "i32"], "sz"),
    "do_router_forward_backward": (["p", "p", "i64", "i32", "i32", "i32", "i32", "i32", "f32", "p",
                                    "p", "p", "p", "p", "p", "p", "p", "sz", "p"], "i32"),
    "do_rem_allocate": (["p", "p", "p", "i32", "i32", "i32", "p", "p", "p", "p", "p", "p"], "i32"),
}

_CT = {"p": ctypes.c_void_p, "i64": ctypes.c_int64, "i32": ctypes.c_int32,
       "f32": ctypes.c_float, "sz": ctypes.c_size_t, "str": ctypes.c_char_p}


class DoLossError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed with status {status}: {status_string(status)}")


def lib():
    """The loaded libdoloss.so; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"{LIB_PATH} is missing: build it with "
                    "`python -c 'import __graft_entry__ as g; g.build()'`")
            l = ctypes.CDLL(LIB_PATH)
            for name, (args, res) in EXPORTS.items():
                fn = getattr(l, name)
                fn.argtypes = [_CT[a] for a in args]
                fn.restype = _CT[res]
            _lib = l
        return _lib


def status_string(status: int) -> str:
    return lib().do_status_string(int(status)).decode()


def _check(fn: str, status: int):
    if status != 0:
        raise DoLossError(fn, status)


def _stream(t: torch.Tensor) -> int:
    return torch.cuda.current_stream(t.device).cuda_stream


def _ptr(t):
    return None if t is None else t.data_ptr()


def _as3d(logits: torch.Tensor) -> torch.Tensor:
    if logits.dim() == 2:
        logits = logits.unsqueeze(0)
    if logits.dim() != 3 or logits.dtype != torch.float32 or not logits.is_cuda:
        raise ValueError("logits must be a CUDA float32 tensor of shape [L, T, E] or [T, E]")
    if not logits.is_contiguous():
        raise ValueError("logits must be contiguous")
    return logits


def words(T: int) -> int:
    return (T + 31) // 32


def workspace_size(T: int, E: int, k: int, L: int = 1) -> int:
    return int(lib().do_workspace_size(T, E, k, L))


def new_workspace(T: int, E: int, k: int, L: int = 1, device="cuda", routed=False) -> torch.Tensor:
    n = int(lib().do_routed_workspace_size(T, E, k, L)) if routed else workspace_size(T, E, k, L)
    if n == 0:
        raise ValueError("invalid sizes")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def signatures(logits: torch.Tensor, k: int, bits=None, counts=None):
    """Step 1: bits [L,E,W] (int32 storage of uint32 words), counts [L,E] int32."""
    z = _as3d(logits)
    L, T, E = z.shape
    if bits is None:
        bits = torch.empty(L, E, words(T), dtype=torch.int32, device=z.device)
    if counts is None:
        counts = torch.empty(L, E, dtype=torch.int32, device=z.device)
    _check("do_signatures", lib().do_signatures(z.data_ptr(), T, E, k, L, bits.data_ptr(),
                                                counts.data_ptr(), _stream(z)))
    return bits, counts


def pairwise_hamming(bits: torch.Tensor, T: int, D=None, accumulate=False):
    """Step 2: D [L,E,E] int32 from bits [L,E,W]; with accumulate, D += it."""
    if bits.dim() == 2:
        bits = bits.unsqueeze(0)
    L, E, _ = bits.shape
    if D is None:
        if accumulate:
            raise ValueError("accumulate needs the D to add to")
        D = torch.empty(L, E, E, dtype=torch.int32, device=bits.device)
    name = "do_pairwise_hamming_accumulate" if accumulate else "do_pairwise_hamming"
    _check(name, getattr(lib(), name)(bits.data_ptr(), T, E, L, D.data_ptr(), _stream(bits)))
    return D


def loss_fwd_bwd(logits, bits, D, k, gate=GATE_SIGMOID_NORM, d_scale=1.0, grad_scale=1.0,
                 with_grad=True, with_origin=True, workspace=None, dlogits=None):
    """Step 3: (loss [L] f32, origin_do [L] i64 or None, dlogits [L,T,E] or None)."""
    z = _as3d(logits)
    L, T, E = z.shape
    if bits.dim() == 2:
        bits = bits.unsqueeze(0)
    if D.dim() == 2:
        D = D.unsqueeze(0)
    loss = torch.empty(L, dtype=torch.float32, device=z.device)
    origin = torch.empty(L, dtype=torch.int64, device=z.device) if with_origin else None
    if with_grad and dlogits is None:
        dlogits = torch.empty_like(z)
    if not with_grad:
        dlogits = None
    if workspace is None:
        workspace = new_workspace(T, E, k, L, z.device)
    _check("do_loss_fwd_bwd", lib().do_loss_fwd_bwd(
        z.data_ptr(), bits.data_ptr(), D.data_ptr(), T, E, k, L, gate, d_scale, grad_scale,
        loss.data_ptr(), _ptr(origin), _ptr(dlogits), workspace.data_ptr(), workspace.numel(),
        _stream(z)))
    return loss, origin, dlogits


class Buffers:
    """Device outputs and workspace of do_forward_backward for one shape."""

    def __init__(self, L, T, E, k, device="cuda", with_grad=True):
        self.shape = (L, T, E, k)
        self.bits = torch.empty(L, E, words(T), dtype=torch.int32, device=device)
        self.counts = torch.empty(L, E, dtype=torch.int32, device=device)
        self.D = torch.empty(L, E, E, dtype=torch.int32, device=device)
        self.loss = torch.empty(L, dtype=torch.float32, device=device)
        self.origin_do = torch.empty(L, dtype=torch.int64, device=device)
        self.dlogits = torch.empty(L, T, E, dtype=torch.float32, device=device) if with_grad else None
        # large enough for the routed call as well
        self.workspace = new_workspace(T, E, k, L, device, routed=True)


def forward_backward(logits, k, gate=GATE_SIGMOID_NORM, grad_scale=1.0, out: Buffers | None = None,
                     with_grad=True):
    """Steps 1-3 in one call; returns the Buffers holding every output."""
    z = _as3d(logits)
    L, T, E = z.shape
    if out is None:
        out = Buffers(L, T, E, k, z.device, with_grad)
    if out.shape != (L, T, E, k):
        raise ValueError("output buffers were made for another shape")
    dl = out.dlogits if with_grad else None
    _check("do_forward_backward", lib().do_forward_backward(
        z.data_ptr(), T, E, k, L, gate, grad_scale, out.bits.data_ptr(), out.counts.data_ptr(),
        out.D.data_ptr(), out.loss.data_ptr(), out.origin_do.data_ptr(), _ptr(dl),
        out.workspace.data_ptr(), out.workspace.numel(), _stream(z)))
    return out


class Routing:
    """Routing outputs (Sec. 3.1.1) for one shape: expert_ids [L,T,k] int32,
    combine [L,T,k] fp32, counts [L,E] int32, offsets [L,E+1] int32,
    rows [L,T*k] int32, pos [L,T,k] int32, and the do_routing workspace."""

    def __init__(self, L, T, E, k, device="cuda", with_dispatch=True):
        self.shape = (L, T, E, k)
        self.expert_ids = torch.empty(L, T, k, dtype=torch.int32, device=device)
        self.combine = torch.empty(L, T, k, dtype=torch.float32, device=device)
        self.counts = torch.empty(L, E, dtype=torch.int32, device=device)
        if with_dispatch:
            self.offsets = torch.empty(L, E + 1, dtype=torch.int32, device=device)
            self.rows = torch.empty(L, T * k, dtype=torch.int32, device=device)
            self.pos = torch.empty(L, T, k, dtype=torch.int32, device=device)
        else:
            self.offsets = self.rows = self.pos = None
        n = int(lib().do_routing_workspace_size(T, E, k, L))
        if n == 0:
            raise ValueError("invalid sizes")
        self.workspace = torch.zeros(n, dtype=torch.uint8, device=device)


def routing(logits, k, gate=GATE_SIGMOID_NORM, out: Routing | None = None):
    """do_routing: the chosen experts, their re-normalized combine weights and
    the expert-grouped dispatch order; returns the Routing holding them."""
    z = _as3d(logits)
    L, T, E = z.shape
    if out is None:
        out = Routing(L, T, E, k, z.device)
    if out.shape != (L, T, E, k):
        raise ValueError("routing buffers were made for another shape")
    _check("do_routing", lib().do_routing(
        z.data_ptr(), T, E, k, L, gate, out.expert_ids.data_ptr(), out.combine.data_ptr(),
        out.counts.data_ptr(), _ptr(out.offsets), _ptr(out.rows), _ptr(out.pos),
        out.workspace.data_ptr(), out.workspace.numel(), _stream(z)))
    return out


def route_backward(logits, expert_ids, grad_combine, gate=GATE_SIGMOID_NORM,
                   dlogits: torch.Tensor | None = None, accumulate=False,
                   status_flags: torch.Tensor | None = None):
    """do_route_backward: the gradient of the combine weights (grad_combine
    [L,T,k] or [T,k] fp32) to the logits [L,T,E], the selection expert_ids
    held fixed.  With accumulate, it is added to the chosen entries of the
    given dlogits; otherwise dlogits (made when None) is overwritten.  Returns
    dlogits."""
    z = _as3d(logits)
    L, T, E = z.shape
    ids = expert_ids.reshape(L, T, -1)
    g = grad_combine.reshape(L, T, -1)
    k = ids.shape[2]
    if ids.dtype != torch.int32 or g.dtype != torch.float32 or g.shape[2] != k:
        raise ValueError("expert_ids must be int32 and grad_combine float32 of the same [L,T,k]")
    if not (ids.is_cuda and g.is_cuda and ids.is_contiguous() and g.is_contiguous()):
        raise ValueError("expert_ids and grad_combine must be contiguous CUDA tensors")
    if dlogits is None:
        if accumulate:
            raise ValueError("accumulate needs the dlogits to add to")
        dlogits = torch.empty_like(z)
    if (dlogits.numel() != z.numel() or dlogits.dtype != torch.float32
            or not dlogits.is_contiguous() or dlogits.device != z.device):
        raise ValueError("dlogits must be a contiguous float32 tensor shaped like the logits")
    _check("do_route_backward", lib().do_route_backward(
        z.data_ptr(), ids.data_ptr(), g.data_ptr(), T, E, k, L, gate, int(bool(accumulate)),
        dlogits.data_ptr(), _ptr(status_flags), _stream(z)))
    return dlogits


def routed_forward(logits, k, gate=GATE_SIGMOID_NORM, out: Buffers | None = None,
                   route: Routing | None = None, with_routing=True):
    """do_routed_forward: steps 1-2 and (with_routing) the routing outputs;
    no loss, no gradient.  Returns (Buffers, Routing or None); out.workspace
    carries what routed_backward reads, so pass the same Buffers to it."""
    z = _as3d(logits)
    L, T, E = z.shape
    if out is None:
        out = Buffers(L, T, E, k, z.device, True)
    if with_routing and route is None:
        route = Routing(L, T, E, k, z.device)
    if not with_routing:
        route = None
    if out.shape != (L, T, E, k) or (route is not None and route.shape != (L, T, E, k)):
        raise ValueError("output buffers were made for another shape")
    r = route
    _check("do_routed_forward", lib().do_routed_forward(
        z.data_ptr(), T, E, k, L, gate, out.bits.data_ptr(), out.counts.data_ptr(),
        out.D.data_ptr(), out.origin_do.data_ptr(), _ptr(r.expert_ids if r else None),
        _ptr(r.combine if r else None), _ptr(r.offsets if r else None),
        _ptr(r.rows if r else None), _ptr(r.pos if r else None),
        out.workspace.data_ptr(), out.workspace.numel(), _stream(z)))
    return out, route


def routed_backward(logits, expert_ids, grad_combine, k, gate=GATE_SIGMOID_NORM, grad_scale=1.0,
                    out: Buffers | None = None, D: torch.Tensor | None = None, d_scale=1.0):
    """do_routed_backward: the DO-loss and its gradient plus the combine
    weights' gradient (grad_combine [L,T,k] fp32; expert_ids and grad_combine
    may both be None) in out.dlogits, after routed_forward filled `out`.  D
    (default out.D) with d_scale: a matrix summed over ranks or micro-batches
    (Eq. global_do).  Returns out."""
    z = _as3d(logits)
    L, T, E = z.shape
    if out is None or out.shape != (L, T, E, k) or out.dlogits is None:
        raise ValueError("routed_backward needs the Buffers of routed_forward (with dlogits)")
    if (expert_ids is None) != (grad_combine is None):
        raise ValueError("expert_ids and grad_combine go together")
    ids = g = None
    if expert_ids is not None:
        ids = expert_ids.reshape(L, T, k)
        g = grad_combine.reshape(L, T, k)
        if ids.dtype != torch.int32 or g.dtype != torch.float32:
            raise ValueError("expert_ids must be int32 and grad_combine float32")
        if not (ids.is_cuda and g.is_cuda and ids.is_contiguous() and g.is_contiguous()):
            raise ValueError("expert_ids and grad_combine must be contiguous CUDA tensors")
    Dm = out.D if D is None else D
    if Dm.shape != (L, E, E) or Dm.dtype != torch.int32 or not Dm.is_contiguous():
        raise ValueError("D must be a contiguous int32 [L,E,E] tensor")
    _check("do_routed_backward", lib().do_routed_backward(
        z.data_ptr(), T, E, k, L, gate, d_scale, grad_scale, out.bits.data_ptr(),
        out.counts.data_ptr(), Dm.data_ptr(), _ptr(ids), _ptr(g), out.loss.data_ptr(),
        out.dlogits.data_ptr(), out.workspace.data_ptr(), out.workspace.numel(), _stream(z)))
    return out


def forward_backward_routed(logits, k, gate=GATE_SIGMOID_NORM, grad_scale=1.0,
                            out: Buffers | None = None, route: Routing | None = None,
                            with_grad=True):
    """do_forward_backward_routed: steps 1-3 plus the routing outputs from the
    same selection pass.  Returns (Buffers, Routing); route.counts and
    route.workspace are not used (the counts are out.counts)."""
    z = _as3d(logits)
    L, T, E = z.shape
    if out is None:
        out = Buffers(L, T, E, k, z.device, with_grad)
    if route is None:
        route = Routing(L, T, E, k, z.device)
    if out.shape != (L, T, E, k) or route.shape != (L, T, E, k):
        raise ValueError("output buffers were made for another shape")
    dl = out.dlogits if with_grad else None
    _check("do_forward_backward_routed", lib().do_forward_backward_routed(
        z.data_ptr(), T, E, k, L, gate, grad_scale, out.bits.data_ptr(), out.counts.data_ptr(),
        out.D.data_ptr(), out.loss.data_ptr(), out.origin_do.data_ptr(), _ptr(dl),
        route.expert_ids.data_ptr(), route.combine.data_ptr(), _ptr(route.offsets),
        _ptr(route.rows), _ptr(route.pos), out.workspace.data_ptr(), out.workspace.numel(),
        _stream(z)))
    return out, route


def router_forward_backward(X: torch.Tensor, Wr: torch.Tensor, k, gate=GATE_SIGMOID_NORM,
                            grad_scale=1.0, out: Buffers | None = None,
                            logits: torch.Tensor | None = None):
    """do_router_forward_backward: logits = X Wr^T (bf16 X [L,T,H] or [T,H],
    Wr [L,E,H] or [E,H]) on the tensor cores, then steps 1-3.  Returns
    (logits [L,T,E] fp32, Buffers)."""
    if X.dim() == 2:
        X = X.unsqueeze(0)
    if Wr.dim() == 2:
        Wr = Wr.unsqueeze(0)
    if X.dtype != torch.bfloat16 or Wr.dtype != torch.bfloat16 or not (X.is_cuda and Wr.is_cuda):
        raise ValueError("X and Wr must be CUDA bfloat16 tensors")
    if not (X.is_contiguous() and Wr.is_contiguous()):
        raise ValueError("X and Wr must be contiguous")
    L, T, H = X.shape
    if Wr.shape[0] != L or Wr.shape[2] != H:
        raise ValueError("Wr must be [L, E, H] for X [L, T, H]")
    E = Wr.shape[1]
    if logits is None:
        logits = torch.empty(L, T, E, dtype=torch.float32, device=X.device)
    if out is None:
        out = Buffers(L, T, E, k, X.device)
    if out.shape != (L, T, E, k):
        raise ValueError("output buffers were made for another shape")
    _check("do_router_forward_backward", lib().do_router_forward_backward(
        X.data_ptr(), Wr.data_ptr(), T, H, E, k, L, gate, grad_scale, logits.data_ptr(),
        out.bits.data_ptr(), out.counts.data_ptr(), out.D.data_ptr(), out.loss.data_ptr(),
        out.origin_do.data_ptr(), _ptr(out.dlogits), out.workspace.data_ptr(),
        out.workspace.numel(), _stream(X)))
    return logits, out


def router_backward(X: torch.Tensor, Wr: torch.Tensor, dlogits: torch.Tensor, with_dx=True,
                    workspace: torch.Tensor | None = None):
    """do_router_backward: dW [L,E,H] fp32 and dX [L,T,H] bf16 (or None) of the
    router's linear map for dlogits [L,T,E] fp32."""
    if X.dim() == 2:
        X = X.unsqueeze(0)
    if Wr.dim() == 2:
        Wr = Wr.unsqueeze(0)
    dz = _as3d(dlogits)
    L, T, H = X.shape
    E = Wr.shape[1]
    if dz.shape != (L, T, E) or Wr.shape != (L, E, H):
        raise ValueError("shapes must be X [L,T,H], Wr [L,E,H], dlogits [L,T,E]")
    dW = torch.empty(L, E, H, dtype=torch.float32, device=X.device)
    dX = torch.empty(L, T, H, dtype=torch.bfloat16, device=X.device) if with_dx else None
    if workspace is None:
        workspace = torch.zeros(int(lib().do_router_backward_workspace_size(T, E, H, L)),
                                dtype=torch.uint8, device=X.device)
    _check("do_router_backward", lib().do_router_backward(
        X.data_ptr(), Wr.data_ptr(), dz.data_ptr(), T, H, E, L, dW.data_ptr(), _ptr(dX),
        workspace.data_ptr(), workspace.numel(), _stream(X)))
    return dW, dX


def maxvio(counts: torch.Tensor, expert_rank: torch.Tensor, R: int, with_rank_loads=False,
           status_flags: torch.Tensor | None = None):
    """do_maxvio: MaxVio (App. E) of each problem's counts [L,E] (device int32)
    for the expert-to-rank map expert_rank [E] (device int32).  Returns maxvio
    [L] float64 (and rank_loads [L,R] int64 when asked)."""
    if counts.dim() == 1:
        counts = counts.unsqueeze(0)
    L, E = counts.shape
    if counts.dtype != torch.int32 or expert_rank.dtype != torch.int32:
        raise ValueError("counts and expert_rank must be int32")
    if not (counts.is_cuda and expert_rank.is_cuda and counts.is_contiguous()
            and expert_rank.is_contiguous()) or expert_rank.numel() != E:
        raise ValueError("counts [L,E] and expert_rank [E] must be contiguous CUDA tensors")
    out = torch.empty(L, dtype=torch.float64, device=counts.device)
    loads = torch.empty(L, R, dtype=torch.int64, device=counts.device) if with_rank_loads else None
    _check("do_maxvio", lib().do_maxvio(counts.data_ptr(), expert_rank.data_ptr(), E, R, L,
                                        _ptr(loads), out.data_ptr(), _ptr(status_flags),
                                        _stream(counts)))
    return (out, loads) if with_rank_loads else out


def rem_allocate(loads, expert_tokens, expert_rank, D: int):
    """do_rem_allocate (host): REM global-batch replica allocation.  Returns
    (placements, loads_after): placements a list of (expert, sender, receiver,
    tokens) in the order made, loads_after a float64 array [R]."""
    import numpy as np

    Lr = np.ascontiguousarray(loads, dtype=np.float64)
    Te = np.ascontiguousarray(expert_tokens, dtype=np.float64)
    er = np.ascontiguousarray(expert_rank, dtype=np.int32)
    R, E = Lr.size, Te.size
    if er.size != E:
        raise ValueError("expert_rank must have one entry per expert")
    cap = max(1, R * D)
    pe, ps, pr = (np.zeros(cap, np.int32) for _ in range(3))
    pt = np.zeros(cap, np.float64)
    n = np.zeros(1, np.int32)
    out = np.zeros(R, np.float64)
    _check("do_rem_allocate", lib().do_rem_allocate(
        Lr.ctypes.data, Te.ctypes.data, er.ctypes.data, R, E, D, pe.ctypes.data, ps.ctypes.data,
        pr.ctypes.data, pt.ctypes.data, n.ctypes.data, out.ctypes.data))
    k = int(n[0])
    return [(int(pe[i]), int(ps[i]), int(pr[i]), float(pt[i])) for i in range(k)], out


def device_status(workspace: torch.Tensor) -> int:
    """Synchronizes the current stream and returns (and clears) the device status."""
    return int(lib().do_device_status(workspace.data_ptr(), _stream(workspace)))


def host_buffer_size(T, E, k, L=1) -> int:
    return int(lib().do_host_buffer_size(T, E, k, L))


def forward_backward_host(h_logits: torch.Tensor, k, gate=GATE_SIGMOID_NORM, grad_scale=1.0,
                          device_buffer: torch.Tensor | None = None, h_dlogits=None,
                          h_counts=None, h_D=None, h_loss=None):
    """Host arrays in, host arrays out (synchronous), through do_forward_backward_host."""
    z = h_logits.unsqueeze(0) if h_logits.dim() == 2 else h_logits
    if z.is_cuda or z.dtype != torch.float32 or not z.is_contiguous():
        raise ValueError("h_logits must be a contiguous CPU float32 tensor")
    L, T, E = z.shape
    if device_buffer is None:
        device_buffer = torch.zeros(host_buffer_size(T, E, k, L), dtype=torch.uint8, device="cuda")
    if h_loss is None:
        h_loss = torch.empty(L, dtype=torch.float32)
    _check("do_forward_backward_host", lib().do_forward_backward_host(
        z.data_ptr(), T, E, k, L, gate, grad_scale, h_loss.data_ptr(), _ptr(h_dlogits),
        _ptr(h_counts), _ptr(h_D), device_buffer.data_ptr(), device_buffer.numel(),
        torch.cuda.current_stream(device_buffer.device).cuda_stream))
    return h_loss


def forward_backward_host_async(h_logits: torch.Tensor, k, h_result: torch.Tensor,
                                device_buffer: torch.Tensor, gate=GATE_SIGMOID_NORM,
                                grad_scale=1.0, stream: torch.cuda.Stream | None = None):
    """do_forward_backward_host_async: enqueue the copy in, steps 1-3 and the
    copy of the losses and the status word into h_result (a pinned CPU tensor
    of at least 4 (L + 1) bytes) on `stream` (default: the current stream).
    Read the result with `host_result` once the stream has been synchronized."""
    z = h_logits.unsqueeze(0) if h_logits.dim() == 2 else h_logits
    if z.is_cuda or z.dtype != torch.float32 or not z.is_contiguous():
        raise ValueError("h_logits must be a contiguous CPU float32 tensor")
    L, T, E = z.shape
    if h_result.is_cuda or h_result.numel() * h_result.element_size() < 4 * (L + 1):
        raise ValueError("h_result must be a CPU tensor of at least 4 (L + 1) bytes")
    st = stream if stream is not None else torch.cuda.current_stream(device_buffer.device)
    _check("do_forward_backward_host_async", lib().do_forward_backward_host_async(
        z.data_ptr(), T, E, k, L, gate, grad_scale, h_result.data_ptr(), device_buffer.data_ptr(),
        device_buffer.numel(), st.cuda_stream))


def host_result(h_result: torch.Tensor, L: int):
    """(losses [L] float32, device status flags int) from an async call's result."""
    raw = h_result.view(torch.uint8)[: 4 * (L + 1)]
    loss = raw[: 4 * L].view(torch.float32).clone()
    flags = int(raw[4 * L: 4 * L + 4].view(torch.int32)[0])
    return loss, flags


def forward_backward_static(logits, k, out: Buffers, gate=GATE_SIGMOID_NORM, grad_scale=1.0,
                            status_flags: torch.Tensor | None = None):
    """do_forward_backward_static: steps 1-3 with the library's own fixed
    scratch array; out.workspace is not used.  status_flags: int32 [1] on the
    device, or None."""
    z = _as3d(logits)
    L, T, E = z.shape
    if out.shape != (L, T, E, k):
        raise ValueError("output buffers were made for another shape")
    _check("do_forward_backward_static", lib().do_forward_backward_static(
        z.data_ptr(), T, E, k, L, gate, grad_scale, out.bits.data_ptr(), out.counts.data_ptr(),
        out.D.data_ptr(), out.loss.data_ptr(), out.origin_do.data_ptr(), _ptr(out.dlogits),
        _ptr(status_flags), _stream(z)))
    return out


def selftest_wait_limit(workspace: torch.Tensor) -> None:
    """Launches the bounded-wait self-test on the current stream (see
    include/doloss.h); do_device_status afterwards reports the time-out."""
    _check("do_selftest_wait_limit",
           lib().do_selftest_wait_limit(workspace.data_ptr(), _stream(workspace)))


def all_reduce_distances(D: torch.Tensor, group=None):
    """Sums the local Hamming matrices of the data-parallel ranks in place and
    returns (D, d_scale), d_scale = 1 / (number of ranks): the summed matrix
    G^g = d_scale * sum_r D_r of Global-DO (Sec. 3.1.4, Eq. global_do).  D is
    int32 (the sum of per-rank distances stays exact); one rank or no
    initialised process group leaves D as it is with d_scale = 1."""
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()):
        return D, 1.0
    world = dist.get_world_size(group)
    if world > 1:
        dist.all_reduce(D, op=dist.ReduceOp.SUM, group=group)
    return D, 1.0 / world


def global_forward_backward(logits, k, gate=GATE_SIGMOID_NORM, grad_scale=1.0, group=None):
    """Global-DO on the local tokens of this rank: signatures and the local
    Hamming matrix, its sum over the ranks of `group`, then the loss and the
    gradient with d_scale = 1/ranks (m stays the local token count).
    Returns (loss [L], dlogits [L,T,E], D_global [L,E,E] int32, counts [L,E])."""
    z = _as3d(logits)
    # the forward half (fused selection and co-occurrence reduction), the sum
    # over the ranks, then the backward half with that matrix
    out, _ = routed_forward(z, k, gate, with_routing=False)
    D, d_scale = all_reduce_distances(out.D, group)
    routed_backward(z, None, None, k, gate, grad_scale, out=out, D=D, d_scale=d_scale)
    return out.loss, out.dlogits, D, out.counts


def window_forward_backward(logits_list, k, gate=GATE_SIGMOID_NORM, grad_scale=1.0, group=None):
    """Global-DO over a gradient-accumulation window (Sec. 3.1.4, Eq. global_do;
    App. batch ablation): the Hamming matrices of the window's micro-batches
    (each from its forward half) are summed, then summed over the ranks of
    `group`, and every micro-batch's loss and gradient use that matrix with
    d_scale = 1 / (ranks x micro-batches) and m = its own token count.
    logits_list: the window's micro-batches, each [L,T,E] or [T,E] on the GPU.
    Returns (losses: list of [L] fp32, dlogits: list of [L,T,E], D [L,E,E])."""
    zs = [_as3d(z) for z in logits_list]
    if not zs:
        raise ValueError("an empty window")
    L, _, E = zs[0].shape
    D = torch.zeros(L, E, E, dtype=torch.int32, device=zs[0].device)
    outs = []
    for z in zs:
        if z.shape[0] != L or z.shape[2] != E:
            raise ValueError("the window's micro-batches must share L and E")
        # the forward half of each micro-batch (its own buffers: the backward
        # half reads the selection it leaves), its matrix added to the window's
        out, _ = routed_forward(z, k, gate, with_routing=False)
        _check("do_accumulate_distances", lib().do_accumulate_distances(
            out.D.data_ptr(), E, L, D.data_ptr(), _stream(z)))
        outs.append(out)
    D, d_rank = all_reduce_distances(D, group)
    d_scale = d_rank / len(zs)
    for z, out in zip(zs, outs):
        routed_backward(z, None, None, k, gate, grad_scale, out=out, D=D, d_scale=d_scale)
    return [o.loss for o in outs], [o.dlogits for o in outs], D


class _DOLossFunction(torch.autograd.Function):
    """The DO-loss of one call as an autograd node: the forward runs steps 1-3
    (the gradient with grad_scale = 1 comes out of the same pass), and the
    backward returns it times the incoming gradient of each problem's loss."""

    @staticmethod
    def forward(ctx, logits, k, gate):
        squeeze = logits.dim() == 2
        out = forward_backward(logits.detach(), k, gate, 1.0)
        ctx.save_for_backward(out.dlogits)
        ctx.squeeze = squeeze
        return out.loss[0].clone() if squeeze else out.loss.clone()

    @staticmethod
    def backward(ctx, grad):
        (dz,) = ctx.saved_tensors
        dz = dz * grad.reshape(-1, 1, 1).to(dz.dtype)
        return (dz[0] if ctx.squeeze else dz), None, None


def do_loss(logits: torch.Tensor, k: int, gate=GATE_SIGMOID_NORM) -> torch.Tensor:
    """The DO-loss (Sec. 3.1.3, Eq. do_loss) of router logits [T,E] or [L,T,E]
    (fp32, CUDA) as a differentiable tensor: a scalar, or [L] per problem.
    Multiply by the loss weight and add to the training objective; the
    gradient reaches the logits through autograd."""
    return _DOLossFunction.apply(_as3d(logits) if logits.dim() == 3 else logits, k, gate)


class _RouteFunction(torch.autograd.Function):
    """The routing outputs of one call as an autograd node: the forward runs
    do_routing (ids, combine weights, dispatch order); the backward sends the
    incoming gradient of the combine weights to the logits through
    do_route_backward, the selection held fixed."""

    @staticmethod
    def forward(ctx, logits, k, gate):
        z = _as3d(logits.detach())
        route = routing(z, k, gate)
        ctx.save_for_backward(z, route.expert_ids)
        ctx.gate = gate
        ctx.squeeze = logits.dim() == 2
        ids, combine = route.expert_ids, route.combine
        if ctx.squeeze:
            ids, combine = ids[0], combine[0]
        ctx.mark_non_differentiable(ids)
        return ids, combine, route

    @staticmethod
    def backward(ctx, grad_ids, grad_combine, grad_route):
        z, ids = ctx.saved_tensors
        if grad_combine is None:
            return None, None, None
        g = grad_combine.reshape(ids.shape).to(torch.float32).contiguous()
        dz = route_backward(z, ids, g, ctx.gate)
        return (dz[0] if ctx.squeeze else dz), None, None


def route(logits: torch.Tensor, k: int, gate=GATE_SIGMOID_NORM):
    """Routing of router logits [T,E] or [L,T,E] (fp32, CUDA) for an MoE layer
    (Sec. 3.1.1): returns (expert_ids, combine, Routing) where combine, the
    re-normalized weights of the chosen experts, is differentiable -- its
    gradient reaches the logits through autograd with the choice of experts
    held fixed -- and the Routing also holds the counts and the dispatch
    order."""
    return _RouteFunction.apply(logits, k, gate)


def offdiag_variance(origin_do: torch.Tensor, T: int, E: int, k: int) -> torch.Tensor:
    """do_offdiag_variance: the variance of the off-diagonal entries of each
    problem's local Hamming matrix (App. C.1) from origin_do [L] int64 (CUDA),
    computed on the device; returns float64 [L]."""
    if origin_do.dtype != torch.int64 or not origin_do.is_cuda or not origin_do.is_contiguous():
        raise ValueError("origin_do must be a contiguous CUDA int64 tensor")
    L = origin_do.numel()
    var = torch.empty(L, dtype=torch.float64, device=origin_do.device)
    _check("do_offdiag_variance", lib().do_offdiag_variance(
        origin_do.data_ptr(), T, E, k, L, var.data_ptr(), _stream(origin_do)))
    return var
