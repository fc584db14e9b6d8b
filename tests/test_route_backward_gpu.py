"""Parity of do_route_backward (the gradient of the re-normalized combine
weights of Sec. 3.1.1 to the logits) with the oracle's entry-by-entry double
evaluation, on seeded logits and upstream gradients.

Tolerance, per entry of a chosen expert l of token t: the kernel evaluates
w_tl (g_tl - dot_t) (times 1 - s_tl for the sigmoid gate) in fp32 from k
gathered logits; each weight carries a few ulp, the two k-term sums of the
row k ulp each, so the error is below (4k + 32) 2^-24 times
scale_tl = w_tl (|g_tl| + sum_q |g_tq| w_tq) (times 1 - s_tl).  The entries of
the experts not chosen are exactly 0 (or untouched when accumulating)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dl():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import paper_2609_32398_gb300.doloss as m
    return m


def make_case(T, E, k, L, gate, seed, shift=0.0, ties=False):
    z = workloads.random_logits(T, E, seed=seed, L=L, ties=ties) + shift
    z = z.float().contiguous()
    ids = np.stack([oracle.route(z[l].numpy(), k, gate)[0] for l in range(L)]).astype(np.int32)
    g = torch.Generator().manual_seed(seed + 1)
    grad = torch.randn(L, T, k, generator=g, dtype=torch.float32)
    return z, ids, grad


def bound(zl, ids, g, gate):
    """(4k + 32) 2^-24 scale_tl on the chosen entries, as a dense [T,E] array."""
    k = ids.shape[1]
    _, w = oracle.route(zl, k, gate)
    gd = g.astype(np.float64)
    scale = w * (np.abs(gd) + (np.abs(gd) * w).sum(1, keepdims=True))
    if gate == oracle.GATE_SIGMOID_NORM:
        zc = np.take_along_axis(zl.astype(np.float64), ids.astype(np.int64), axis=1)
        scale = scale / (1.0 + np.exp(zc))
    out = np.zeros(zl.shape)
    np.put_along_axis(out, ids.astype(np.int64), scale, axis=1)
    return (4 * k + 32) * 2.0 ** -24 * out + 1e-37


def check(dz_gpu, z, ids, grad, gate):
    L = z.shape[0]
    for l in range(L):
        zl, il, gl = z[l].numpy(), ids[l], grad[l].numpy()
        ref = oracle.route_backward(zl, il, gl.astype(np.float64), gate)
        got = dz_gpu[l].double().cpu().numpy()
        err = np.abs(got - ref)
        tol = bound(zl, il, gl, gate)
        assert (err <= tol).all(), (l, float((err / tol).max()))
        chosen = np.zeros(zl.shape, bool)
        np.put_along_axis(chosen, il.astype(np.int64), True, axis=1)
        assert (got[~chosen] == 0.0).all()


@pytest.mark.parametrize("T,E,k,L,gate,ties", [
    (1, 8, 1, 1, 0, False),
    (1033, 8, 2, 2, 0, True),
    (1033, 33, 5, 2, 1, False),
    (4096 + 17, 128, 8, 1, 0, True),
    (4096 + 17, 128, 8, 1, 1, False),
    (500, 16, 16, 1, 0, False),          # k = E: every expert chosen
    (3000 + 7, 128, 1, 1, 1, False),     # one row per lane: 128 rows per warp pass
    (1000 + 3, 1024, 8, 1, 0, True),     # 4 KB rows
    (2000 + 1, 64, 4, 2, 0, False),
    (300, 1024, 64, 1, 0, False),        # k > 32: several choices per lane
    (300, 1024, 33, 2, 1, True),
])
def test_route_backward_matches_oracle(dl, T, E, k, L, gate, ties):
    z, ids, grad = make_case(T, E, k, L, gate, seed=T + E + k, ties=ties)
    dz = dl.route_backward(z.cuda(), torch.from_numpy(ids).cuda(), grad.cuda(), gate)
    torch.cuda.synchronize()
    check(dz, z, ids, grad, gate)


@pytest.mark.parametrize("accumulate", [False, True])
def test_unaligned_buffers(dl, accumulate):
    """Logits and dlogits 4-byte but not 16-byte aligned: the rows are zeroed
    with 4-byte stores instead of 16-byte ones; the values are the same."""
    T, E, k, gate = 4096 + 9, 128, 8, 0
    z, ids, grad = make_case(T, E, k, 1, gate, seed=31)
    zbuf = torch.empty(T * E + 1, device="cuda")
    zc = zbuf[1:].view(1, T, E)
    zc.copy_(z)
    dbuf = torch.zeros(T * E + 1, device="cuda")
    dz = dbuf[1:].view(1, T, E)
    assert zc.data_ptr() % 16 == 4 and dz.data_ptr() % 16 == 4
    dl.route_backward(zc, torch.from_numpy(ids).cuda(), grad.cuda(), gate, dlogits=dz,
                      accumulate=accumulate)
    check(dz, z, ids, grad, gate)
    aligned = dl.route_backward(z.cuda(), torch.from_numpy(ids).cuda(), grad.cuda(), gate)
    torch.cuda.synchronize()
    assert torch.equal(dz, aligned)   # the same arithmetic on both kernels


@pytest.mark.parametrize("shift", [-120.0, -30.0, 60.0])
@pytest.mark.parametrize("gate", [0, 1])
def test_route_backward_far_from_zero(dl, shift, gate):
    """Logits shifted far from 0: the sigmoid weights take the ratio form
    (no 0/0 when every chosen sigmoid underflows) and 1 - s stays exact in
    its own precision."""
    z, ids, grad = make_case(777, 64, 8, 1, gate, seed=9, shift=shift)
    dz = dl.route_backward(z.cuda(), torch.from_numpy(ids).cuda(), grad.cuda(), gate)
    check(dz, z, ids, grad, gate)


def test_route_backward_full_size_c3(dl):
    """The c3 routing workload at full size (T = 65536, E = 128, k = 8,
    sigmoid-norm) in the launch configuration the benchmark times, every
    entry against the oracle."""
    w = workloads.get("c3")
    z = workloads.logits(w, "cpu")
    ids = oracle.route(z[0].numpy(), w.k, w.gate)[0][None].astype(np.int32)
    grad = torch.randn(1, w.T, w.k, generator=torch.Generator().manual_seed(3))
    dz = dl.route_backward(z.cuda(), torch.from_numpy(ids).cuda(), grad.cuda(), w.gate)
    check(dz, z, ids, grad, w.gate)


@pytest.mark.parametrize("gate", [0, 1])
def test_accumulate_adds_to_the_chosen_entries_only(dl, gate):
    z, ids, grad = make_case(2048 + 5, 128, 8, 2, gate, seed=21)
    zc, ic, gc = z.cuda(), torch.from_numpy(ids).cuda(), grad.cuda()
    over = dl.route_backward(zc, ic, gc, gate)
    base = torch.randn(z.shape, generator=torch.Generator().manual_seed(4)).cuda()
    acc = dl.route_backward(zc, ic, gc, gate, dlogits=base.clone(), accumulate=True)
    torch.cuda.synchronize()
    # one RED per chosen entry: fl(base + d); elsewhere base + 0 = base
    assert torch.equal(acc, base + over)


def test_route_backward_is_reproducible(dl):
    z, ids, grad = make_case(8192, 128, 8, 1, 0, seed=5)
    zc, ic, gc = z.cuda(), torch.from_numpy(ids).cuda(), grad.cuda()
    a = dl.route_backward(zc, ic, gc, 0)
    b = dl.route_backward(zc, ic, gc, 0)
    c = dl.route_backward(zc, ic, gc, 0, dlogits=torch.zeros_like(zc), accumulate=True)
    torch.cuda.synchronize()
    assert torch.equal(a, b) and torch.equal(a, c)


def test_out_of_range_ids_are_flagged_and_left_out(dl):
    """An id outside [0, E) raises status bit 2 and is left out of its row
    (the kernel checks every id before using it); the other rows are as the
    oracle has them."""
    T, E, k = 256, 32, 4
    z, ids, grad = make_case(T, E, k, 1, 0, seed=13)
    bad = ids.copy()
    bad[0, 7, 2] = E
    bad[0, 100, 0] = -1
    flags = torch.zeros(1, dtype=torch.int32, device="cuda")
    dz = dl.route_backward(z.cuda(), torch.from_numpy(bad).cuda(), grad.cuda(), 0,
                           status_flags=flags)
    torch.cuda.synchronize()
    assert int(flags[0]) == 4
    keep = np.ones(T, bool)
    keep[[7, 100]] = False
    ref = oracle.route_backward(z[0].numpy(), ids[0], grad[0].numpy().astype(np.float64), 0)
    got = dz[0].double().cpu().numpy()
    tol = bound(z[0].numpy(), ids[0], grad[0].numpy(), 0)
    assert (np.abs(got - ref)[keep] <= tol[keep]).all()
    assert np.isfinite(got).all()


def test_do_loss_plus_routing_gradient_in_one_buffer(dl):
    """do_forward_backward writes the DO-loss gradient, do_route_backward adds
    the combine weights' gradient into the same buffer: the sum of the two
    oracle gradients, within the sum of the two tolerances."""
    w = workloads.get("c3", T=4096)
    z = workloads.logits(w, "cpu")
    zc = z.cuda()
    out = dl.forward_backward(zc, w.k, gate=w.gate)
    route = dl.routing(zc, w.k, w.gate)
    grad = torch.randn(1, w.T, w.k, generator=torch.Generator().manual_seed(8)).cuda()
    dl.route_backward(zc, route.expert_ids, grad, w.gate, dlogits=out.dlogits, accumulate=True)
    torch.cuda.synchronize()
    zl = z[0].numpy()
    ids = oracle.route(zl, w.k, w.gate)[0]
    assert np.array_equal(route.expert_ids[0].cpu().numpy(), ids)
    ref_do = oracle.forward_backward(zl, w.k, w.gate)["dz"]
    g64 = grad[0].double().cpu().numpy()
    ref_route = oracle.route_backward(zl, ids, g64, w.gate)
    got = out.dlogits[0].double().cpu().numpy()
    tol = 1e-4 * np.abs(ref_do).max() + bound(zl, ids, grad[0].cpu().numpy(), w.gate)
    assert (np.abs(got - (ref_do + ref_route)) <= tol).all()


@pytest.mark.parametrize("gate", [0, 1])
def test_autograd_route_with_the_do_loss(dl, gate):
    """dl.route as an autograd node: a loss built from the combine weights and
    the DO-loss together backpropagate to the logits as the oracle's two
    gradients summed (combine weights: the selection held fixed)."""
    T, E, k = 2048 + 3, 128, 8
    z_cpu = workloads.random_logits(T, E, seed=41)[0]
    z = z_cpu.cuda().requires_grad_(True)
    ids, combine, route = dl.route(z, k, gate)
    assert ids.shape == (T, k) and combine.shape == (T, k) and not ids.requires_grad
    u = torch.randn(T, k, generator=torch.Generator().manual_seed(2)).cuda()
    lam = 0.25
    objective = (combine * u).sum() + lam * dl.do_loss(z, k, gate)
    objective.backward()
    zl = z_cpu.numpy()
    ids_ref, _ = oracle.route(zl, k, gate)
    assert np.array_equal(ids.cpu().numpy(), ids_ref)
    want_route = oracle.route_backward(zl, ids_ref, u.double().cpu().numpy(), gate)
    want_do = lam * oracle.forward_backward(zl, k, gate)["dz"]
    tol = 1e-4 * np.abs(want_do).max() + bound(zl, ids_ref, u.cpu().numpy(), gate)
    got = z.grad.double().cpu().numpy()
    assert (np.abs(got - (want_route + want_do)) <= tol).all()


def test_route_backward_worked_example_on_the_gpu(dl):
    """The hand-worked tokens of tests/golden/route_backward_worked_n4_k2.json
    through do_route_backward (E = 4: the gather kernel's unaligned-width
    path), both gates."""
    import json
    import os
    from fractions import Fraction

    g = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                    "route_backward_worked_n4_k2.json")))
    sym = {"0": 0.0, "1": 1.0, "ln2": np.log(2.0), "-ln2": -np.log(2.0), "ln3": np.log(3.0),
           "-ln3": -np.log(3.0)}
    z = torch.tensor([[sym[v] for v in row] for row in g["logits_symbolic"]], dtype=torch.float32)
    ids = torch.tensor(g["expert_ids"], dtype=torch.int32)
    grad = torch.tensor(g["grad_combine"], dtype=torch.float32)

    def value(v):
        if v.lstrip("-") == "sig(-1)":
            x = 1.0 / (1.0 + np.e)
            return -x if v.startswith("-") else x
        return float(Fraction(v))
    for gate, key in ((0, "dlogits_sigmoid_norm"), (1, "dlogits_softmax")):
        dz = dl.route_backward(z.cuda(), ids.cuda(), grad.cuda(), gate)
        want = np.array([[value(v) for v in row] for row in g[key]])
        np.testing.assert_allclose(dz.double().cpu().numpy()[0], want, rtol=0, atol=1e-6)
