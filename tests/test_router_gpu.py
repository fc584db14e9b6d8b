"""Router-side fusion (do_router_forward_backward): the logits of the router's
linear map on the tensor cores against the oracle, and the rest of the path
against the oracle and the plain fused path on those logits.

Logits: bf16 products are exact in fp32 and summed in fp32 over H terms, so
|z - z_ref| <= gamma * sum_h |x_h w_h| with gamma = 2 H 2^-24 (twice the
classic bound); z_ref is the oracle's fp64 sum.  The selection is taken on
the kernel's fp32 logits, so bits, counts, D and origin_do must equal the
oracle's on those logits exactly, and the loss and dlogits meet the path's
tolerances (and equal the plain path's bit for bit)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

pytestmark = pytest.mark.gpu
U32 = 2.0 ** -24


@pytest.fixture(scope="module")
def dl():
    import paper_2609_32398_gb300.doloss as m

    m.lib()
    return m


def bits16(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def check_logits(z, X, W, rows):
    """z [T,E] from the GPU, X [T,H], W [E,H] bf16: sampled rows against the oracle."""
    Xs = bits16(X[rows])
    Wb = bits16(W)
    ref = oracle.router_logits(Xs, Wb)
    absprod = np.abs(oracle.bf16_to_double(Xs)) @ np.abs(oracle.bf16_to_double(Wb)).T
    H = X.shape[1]
    err = np.abs(z[rows].double().cpu().numpy() - ref)
    assert (err <= 2 * H * U32 * absprod + 1e-30).all(), float((err / (absprod + 1e-30)).max())


@pytest.mark.parametrize("T,H,k,L,gate", [(4096 + 33, 256, 8, 1, 0), (1000, 64, 4, 2, 0),
                                           (300, 128, 1, 1, 1), (129, 2048, 2, 1, 0),
                                           (1, 64, 8, 1, 0)])
def test_router_path_matches_oracle(dl, T, H, k, L, gate):
    X, W = workloads.router_inputs(T, H, 128, L, seed=T + H + k, device="cuda")
    logits, out = dl.router_forward_backward(X, W, k, gate)
    st = dl.device_status(out.workspace)
    assert st == 0, dl.status_string(st)
    plain = dl.forward_backward(logits, k, gate)
    assert dl.device_status(plain.workspace) == 0
    for name in ("bits", "counts", "D", "loss", "origin_do", "dlogits"):
        assert torch.equal(getattr(out, name), getattr(plain, name)), name
    for l in range(L):
        check_logits(logits[l], X[l], W[l], np.arange(T))
        zl = logits[l].cpu().numpy()
        ref = oracle.forward_backward(zl, k, gate)
        assert np.array_equal(out.bits[l].cpu().numpy().view(np.uint32), ref["bits"])
        assert np.array_equal(out.counts[l].cpu().numpy(), ref["counts"])
        assert np.array_equal(out.D[l].cpu().numpy(), ref["D"])
        assert int(out.origin_do[l]) == ref["origin_do"]
        assert abs(float(out.loss[l]) - ref["loss"]) <= 1e-5 * abs(ref["loss"]) + 1e-12
        g = out.dlogits[l].double().cpu().numpy()
        assert np.abs(g - ref["dz"]).max() <= 1e-4 * np.abs(ref["dz"]).max()


def test_router_path_full_size(dl):
    """The benchmark's router layer: T = 65536 tokens, H = 2048, E = 128, k = 8."""
    T, H, k = 65536, 2048, 8
    X, W = workloads.router_inputs(T, H, 128, 1, seed=2, device="cuda")
    logits, out = dl.router_forward_backward(X, W, k, 0)
    assert dl.device_status(out.workspace) == 0
    rows = np.random.default_rng(0).choice(T, 512, replace=False)
    check_logits(logits[0], X[0], W[0], np.sort(rows))
    # every element against torch's fp32 product of the same bf16 values
    ref = X[0].float() @ W[0].float().T
    absprod = X[0].float().abs() @ W[0].float().abs().T
    assert ((logits[0] - ref).abs() <= 4 * H * U32 * absprod).all()
    plain = dl.forward_backward(logits, k, 0)
    for name in ("bits", "counts", "D", "loss", "origin_do", "dlogits"):
        assert torch.equal(getattr(out, name), getattr(plain, name)), name
    zl = logits[0].cpu().numpy()
    ref = oracle.forward_backward(zl, k, 0, with_grad=False)
    assert np.array_equal(out.D[0].cpu().numpy(), ref["D"])
    assert abs(float(out.loss[0]) - ref["loss"]) <= 1e-5 * abs(ref["loss"])


def test_router_path_is_reproducible(dl):
    X, W = workloads.router_inputs(20000, 512, 128, 1, seed=4, device="cuda")
    a_logits, a = dl.router_forward_backward(X, W, 8)
    b_logits, b = dl.router_forward_backward(X, W, 8)
    assert torch.equal(a_logits, b_logits)
    for name in ("bits", "D", "loss", "dlogits"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name


def check_router_grads(dW, dX, X, W, dz, cols=None, rows=None):
    """dW [E,H] fp32 and dX [T,H] bf16 against the oracle's fp64 gradients of the
    same bf16 X, W and the fp32 dz.  dz is rounded to bf16 (relative error at
    most 2^-9) and the products accumulate in fp32: per element the error is
    below (2^-8 + 2 n 2^-24) times the sum of |terms|, n the reduction length;
    dX is also rounded to bf16 on output (2^-8 of its value)."""
    T, H = X.shape
    E = W.shape[0]
    cols = np.arange(H) if cols is None else cols
    rows = np.arange(T) if rows is None else rows
    Xb, Wb = bits16(X), bits16(W)
    dzd = dz.double().cpu().numpy()
    Xs = np.ascontiguousarray(Xb[:, cols])
    Ws = np.ascontiguousarray(Wb[:, cols])
    dW_ref = oracle.router_grad(Xs, Ws, dzd)
    absW = np.abs(dzd).T @ np.abs(oracle.bf16_to_double(Xs))
    got = dW[:, cols].double().cpu().numpy()
    assert (np.abs(got - dW_ref) <= (2.0 ** -8 + 2 * T * U32) * absW + 1e-30).all()
    if dX is not None:
        Xr = np.ascontiguousarray(Xb[rows])
        _, dX_ref = oracle.router_grad(Xr, Wb, np.ascontiguousarray(dzd[rows]), with_dx=True)
        absX = np.abs(dzd[rows]) @ np.abs(oracle.bf16_to_double(Wb))
        gx = dX[rows].double().cpu().numpy()
        tol = 2.0 ** -8 * np.abs(dX_ref) + (2.0 ** -8 + 2 * E * U32) * absX + 1e-30
        assert (np.abs(gx - dX_ref) <= tol).all()


@pytest.mark.parametrize("T,H,L", [(4096 + 33, 256, 2), (300, 64, 1)])
def test_router_backward_matches_oracle(dl, T, H, L):
    X, W = workloads.router_inputs(T, H, 128, L, seed=T + 3 * H, device="cuda")
    logits, out = dl.router_forward_backward(X, W, 8, 0, grad_scale=1000.0)
    assert dl.device_status(out.workspace) == 0
    dW, dX = dl.router_backward(X, W, out.dlogits)
    for l in range(L):
        check_router_grads(dW[l], dX[l], X[l], W[l], out.dlogits[l])


def test_router_backward_full_size(dl):
    T, H = 65536, 2048
    X, W = workloads.router_inputs(T, H, 128, 1, seed=2, device="cuda")
    _, out = dl.router_forward_backward(X, W, 8, 0, grad_scale=1000.0)
    dW, dX = dl.router_backward(X, W, out.dlogits)
    rng = np.random.default_rng(1)
    check_router_grads(dW[0], dX[0], X[0], W[0], out.dlogits[0],
                       cols=np.sort(rng.choice(H, 48, replace=False)),
                       rows=np.sort(rng.choice(T, 256, replace=False)))


def test_router_cooc_in_global_memory_for_long_ranges(dl):
    """A CTA whose token range exceeds 65535 tokens adds its co-occurrence
    counts into its global triangle (L2 reductions) instead of 16-bit shared
    counters.  With one CTA per problem (as many problems as SMs) and
    T = 65536 + 32 that path runs; it must give the same signatures, counts,
    D, loss and gradient as the plain fused call on the router's logits."""
    L = torch.cuda.get_device_properties(0).multi_processor_count
    T, H = 65536 + 32, 64
    X, W = workloads.router_inputs(T, H, 128, L, seed=11, device="cuda")
    z, a = dl.router_forward_backward(X, W, 8)
    assert dl.device_status(a.workspace) == 0
    b = dl.forward_backward(z, 8, 0)
    assert dl.device_status(b.workspace) == 0
    for name in ("bits", "counts", "D", "loss", "origin_do", "dlogits"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
