"""The routed step split into its forward half (do_routed_forward: steps 1-2
and the routing outputs) and its backward half (do_routed_backward: the
DO-loss, its gradient and the combine weights' gradient, Sec. 3.1.1), against
the oracle and against the one-call entry points.

Tolerances: bits, counts, D, origin_do and the routing ids bit-exact; the
loss within 1e-5 relative; dlogits within 1e-4 of the largest DO-gradient
entry (the path's gradient tolerance) plus the routing gradient's
per-entry bound (4k + 32) 2^-24 w (|g| + sum |g| w) (1 - s)."""
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


def route_bound(zl, ids, g, gate):
    k = ids.shape[1]
    _, w = oracle.route(zl, k, gate)
    gd = g.astype(np.float64)
    scale = w * (np.abs(gd) + (np.abs(gd) * w).sum(1, keepdims=True))
    if gate == oracle.GATE_SIGMOID_NORM:
        zc = np.take_along_axis(zl.astype(np.float64), ids.astype(np.int64), axis=1)
        scale = scale / (1.0 + np.exp(zc))
    out = np.zeros(zl.shape)
    np.put_along_axis(out, ids.astype(np.int64), scale, axis=1)
    return (4 * k + 32) * 2.0 ** -24 * out


def run_split(dl, z, k, gate, grad, grad_scale=1.0):
    out, route = dl.routed_forward(z, k, gate)
    dl.routed_backward(z, route.expert_ids, grad, k, gate, grad_scale, out=out)
    torch.cuda.synchronize()
    assert dl.device_status(out.workspace) == 0
    return out, route


@pytest.mark.parametrize("T,E,k,L,gate", [
    (4096 + 33, 128, 8, 1, 0),     # tensor-core loss kernel with the fused routing gradient
    (2048 + 7, 128, 4, 2, 0),
    (1000, 128, 1, 1, 0),
    (3000 + 5, 128, 8, 1, 1),      # softmax: the ALU loss kernel, then the routing kernel
    (4096 + 1, 64, 8, 1, 0),
    (1000 + 9, 33, 5, 2, 0),       # generic kernels
    (1, 8, 2, 1, 0),
])
def test_split_matches_oracle(dl, T, E, k, L, gate):
    z = workloads.random_logits(T, E, L=L, seed=T + E + k)
    grad = torch.randn(L, T, k, generator=torch.Generator().manual_seed(T))
    out, route = run_split(dl, z.cuda(), k, gate, grad.cuda(), grad_scale=0.5)
    for l in range(L):
        zl = z[l].numpy()
        ref = oracle.forward_backward(zl, k, gate)
        assert (out.bits[l].cpu().numpy().view(np.uint32) == ref["bits"]).all()
        assert (out.counts[l].cpu().numpy() == ref["counts"]).all()
        assert (out.D[l].cpu().numpy() == ref["D"]).all()
        assert int(out.origin_do[l]) == ref["origin_do"]
        ids, comb = oracle.route(zl, k, gate)
        assert (route.expert_ids[l].cpu().numpy() == ids).all()
        assert np.abs(route.combine[l].double().cpu().numpy() - comb).max() < 1e-5
        _, rows, _ = oracle.dispatch(ids, E)
        assert (route.rows[l].cpu().numpy() == rows).all()
        assert abs(float(out.loss[l]) - ref["loss"]) <= 1e-5 * abs(ref["loss"]) + 1e-30
        gl = grad[l].numpy()
        want = 0.5 * ref["dz"] + oracle.route_backward(zl, ids, gl.astype(np.float64), gate)
        tol = 1e-4 * 0.5 * np.abs(ref["dz"]).max() + route_bound(zl, ids, gl, gate)
        got = out.dlogits[l].double().cpu().numpy()
        assert (np.abs(got - want) <= tol).all(), float((np.abs(got - want) / tol).max())


def test_split_full_size_c3(dl):
    """The c3 workload at full size (T = 65536) on the fused kernel, every
    entry of dlogits against the oracle."""
    w = workloads.get("c3")
    z = workloads.logits(w, "cpu")
    grad = torch.randn(1, w.T, w.k, generator=torch.Generator().manual_seed(2))
    out, route = run_split(dl, z.cuda(), w.k, w.gate, grad.cuda())
    zl = z[0].numpy()
    ref = oracle.forward_backward(zl, w.k, w.gate)
    ids, _ = oracle.route(zl, w.k, w.gate)
    assert (route.expert_ids[0].cpu().numpy() == ids).all()
    assert (out.D[0].cpu().numpy() == ref["D"]).all()
    assert abs(float(out.loss[0]) - ref["loss"]) <= 1e-5 * abs(ref["loss"])
    gl = grad[0].numpy()
    want = ref["dz"] + oracle.route_backward(zl, ids, gl.astype(np.float64), w.gate)
    tol = 1e-4 * np.abs(ref["dz"]).max() + route_bound(zl, ids, gl, w.gate)
    assert (np.abs(out.dlogits[0].double().cpu().numpy() - want) <= tol).all()


@pytest.mark.parametrize("T,E,k,gate", [(4096 + 33, 128, 8, 0), (2048, 64, 4, 0), (999, 33, 3, 1)])
def test_zero_upstream_gradient_gives_the_plain_step(dl, T, E, k, gate):
    """With grad_combine = 0 the backward half returns exactly the loss and
    dlogits of do_forward_backward (the DO part is the same arithmetic)."""
    z = workloads.random_logits(T, E, seed=7).cuda()
    out, route = run_split(dl, z, k, gate, torch.zeros(1, T, k, device="cuda"))
    ref = dl.forward_backward(z, k, gate)
    torch.cuda.synchronize()
    assert torch.equal(out.loss, ref.loss)
    assert torch.equal(out.dlogits, ref.dlogits)
    assert torch.equal(out.D, ref.D) and torch.equal(out.origin_do, ref.origin_do)


@pytest.mark.parametrize("T,E,k,gate", [(4096 + 33, 128, 8, 0), (3000, 128, 8, 1), (999, 33, 3, 0)])
def test_split_against_the_one_call_entries(dl, T, E, k, gate):
    """Forward half twice (the counts accumulator is cleared within it), then
    the backward half twice: identical each time, and within the routing
    bound of do_forward_backward's dlogits plus do_route_backward's."""
    z = workloads.random_logits(T, E, seed=11).cuda()
    grad = torch.randn(1, T, k, device="cuda")
    out, route = dl.routed_forward(z, k, gate)
    out, route = dl.routed_forward(z, k, gate, out=out, route=route)
    dl.routed_backward(z, route.expert_ids, grad, k, gate, out=out)
    first = out.dlogits.clone()
    dl.routed_backward(z, route.expert_ids, grad, k, gate, out=out)
    ref = dl.forward_backward(z, k, gate)
    sep = dl.route_backward(z, route.expert_ids, grad, gate, dlogits=ref.dlogits.clone(),
                            accumulate=True)
    torch.cuda.synchronize()
    assert dl.device_status(out.workspace) == 0
    assert torch.equal(first, out.dlogits)
    assert torch.equal(out.counts, ref.counts) and torch.equal(out.D, ref.D)
    zl = z[0].cpu().numpy()
    ids = route.expert_ids[0].cpu().numpy()
    tol = 2 * route_bound(zl, ids, grad[0].cpu().numpy(), gate) + 1e-30
    assert (np.abs(out.dlogits[0].double().cpu().numpy() - sep[0].double().cpu().numpy())
            <= tol).all()


@pytest.mark.parametrize("T,E,k,gate", [(4096, 128, 8, 0), (777, 33, 3, 1)])
def test_bad_ids_are_reported(dl, T, E, k, gate):
    """An expert id outside [0, E) in the backward half is left out and makes
    do_device_status return DO_ERR_INVALID_ARG; the context stays usable."""
    z = workloads.random_logits(T, E, seed=3).cuda()
    out, route = dl.routed_forward(z, k, gate)
    ids = route.expert_ids.clone()
    ids[0, 5, 0] = E
    ids[0, 6, k - 1] = -7
    dl.routed_backward(z, ids, torch.ones(1, T, k, device="cuda"), k, gate, out=out)
    torch.cuda.synchronize()
    assert dl.device_status(out.workspace) == 1
    assert torch.isfinite(out.dlogits).all()
    dl.routed_backward(z, route.expert_ids, torch.ones(1, T, k, device="cuda"), k, gate, out=out)
    assert dl.device_status(out.workspace) == 0


def test_split_with_unaligned_routing_outputs_and_no_dispatch(dl):
    """expert_ids and combine 4- but not 16-byte aligned (the routing outputs
    then come from the generic selection beside the fused path's) and no
    dispatch arrays (the counts accumulator is then cleared by a memset):
    the same outputs as the aligned call (the weights to their tolerance),
    twice in a row."""
    T, E, k, gate = 4096 + 33, 128, 8, 0
    z = workloads.random_logits(T, E, seed=17, ties=True).cuda()
    grad = torch.randn(1, T, k, device="cuda")
    ref_out, ref_route = run_split(dl, z, k, gate, grad)
    out = dl.Buffers(1, T, E, k)
    route = dl.Routing(1, T, E, k, with_dispatch=False)
    ids_store = torch.empty(T * k + 1, dtype=torch.int32, device="cuda")
    comb_store = torch.empty(T * k + 1, dtype=torch.float32, device="cuda")
    route.expert_ids = ids_store[1:].view(1, T, k)
    route.combine = comb_store[1:].view(1, T, k)
    for _ in range(2):
        dl.routed_forward(z, k, gate, out=out, route=route)
        torch.cuda.synchronize()
        assert torch.equal(route.expert_ids, ref_route.expert_ids)
        # the generic selection kernel sums the weights in another order:
        # both are within 2(k + 12) 2^-24 of the exact ratio
        assert (route.combine - ref_route.combine).abs().max() <= 4 * (k + 12) * 2.0 ** -24
        assert torch.equal(out.counts, ref_out.counts) and torch.equal(out.D, ref_out.D)
        assert torch.equal(out.origin_do, ref_out.origin_do)
    ids_aligned = route.expert_ids.clone()
    dl.routed_backward(z, ids_aligned, grad, k, gate, out=out)
    torch.cuda.synchronize()
    assert dl.device_status(out.workspace) == 0
    assert torch.equal(out.loss, ref_out.loss)
    assert torch.equal(out.dlogits, ref_out.dlogits)


@pytest.mark.parametrize("T,E,k,gate,routed", [
    (4096 + 33, 128, 8, 0, True),     # ALU loss kernel with a summed D (no tensor-core image)
    (4096 + 33, 128, 8, 0, False),
    (2048, 64, 4, 1, True),
    (999, 33, 3, 0, True),            # generic kernels
])
def test_backward_half_with_a_summed_matrix(dl, T, E, k, gate, routed):
    """Global-DO (Sec. 3.1.4, Eq. global_do) through the halves: the forward
    half's local D plus another rank's, d_scale = 1/2, m = the local T; the
    loss and gradient as the oracle computes them with that matrix, plus the
    routing gradient when asked."""
    z = workloads.random_logits(T, E, seed=T + 5)
    z_other = workloads.random_logits(T + 100, E, seed=T + 6)
    out, route = dl.routed_forward(z.cuda(), k, gate, with_routing=routed)
    zl = z[0].numpy()
    f = oracle.select(zl, k)
    D_sum = oracle.hamming(f) + oracle.hamming(oracle.select(z_other[0].numpy(), k))
    Dg = torch.from_numpy(D_sum.astype(np.int32))[None].cuda()
    grad = torch.randn(1, T, k, generator=torch.Generator().manual_seed(1)).cuda()
    dl.routed_backward(z.cuda(), route.expert_ids if routed else None, grad if routed else None,
                       k, gate, 0.75, out=out, D=Dg, d_scale=0.5)
    torch.cuda.synchronize()
    assert dl.device_status(out.workspace) == 0
    want_loss = oracle.loss(D_sum, oracle.direction(zl, f, gate), T, k, 0.5)
    assert abs(float(out.loss[0]) - want_loss) <= 1e-5 * abs(want_loss)
    g_do = 0.75 * oracle.gate_backward(zl, oracle.dloss_dp(D_sum, f, T, k, d_scale=0.5), gate)
    tol = 1e-4 * np.abs(g_do).max()
    want = g_do
    if routed:
        ids, _ = oracle.route(zl, k, gate)
        gl = grad[0].cpu().numpy()
        want = want + oracle.route_backward(zl, ids, gl.astype(np.float64), gate)
        tol = tol + route_bound(zl, ids, gl, gate)
    assert (np.abs(out.dlogits[0].double().cpu().numpy() - want) <= tol).all()


def test_global_do_binding_at_one_rank_is_the_local_step(dl):
    """global_forward_backward through the halves with no process group:
    d_scale = 1, the tensor-core path, bit for bit do_forward_backward."""
    w = workloads.get("c3", T=8192)
    z = workloads.logits(w).cuda()
    loss, dz, D, counts = dl.global_forward_backward(z, w.k, w.gate, grad_scale=2.0)
    ref = dl.forward_backward(z, w.k, w.gate, grad_scale=2.0)
    torch.cuda.synchronize()
    assert torch.equal(D, ref.D) and torch.equal(counts, ref.counts)
    assert torch.equal(loss, ref.loss) and torch.equal(dz, ref.dlogits)
