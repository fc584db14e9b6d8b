"""Parity of the routing outputs (Sec. 3.1.1) of the CUDA path with the CPU
oracle, through the C ABI (do_routing and do_forward_backward_routed).

expert_ids, counts and the dispatch arrays (offsets, rows, pos) are exact
integers and must match bit for bit; the combine weights are fp32 and must
lie within COMBINE_ATOL(k) of the oracle's fp64 values.  Inputs are the seeded
workloads, drawn once and given byte for byte to both sides.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24   # fp32 unit roundoff


def combine_atol(k):
    """Each weight is u_q / sum u with u from one or three expf (at most 2 ulp
    each) and two or three roundings, and the sum of k terms: (k + 12) u bounds
    the error of a weight in (0, 1]; twice that is the test's tolerance."""
    return 2.0 * (k + 12) * U32


@pytest.fixture(scope="module")
def dl():
    import paper_2609_32398_gb300.doloss as m

    m.lib()
    return m


def check_layer(route, l, zl, k, gate, E):
    ids_ref, comb_ref = oracle.route(zl, k, gate)
    ids = route.expert_ids[l].cpu().numpy()
    assert np.array_equal(ids, ids_ref), "expert ids"
    comb = route.combine[l].double().cpu().numpy()
    err = np.abs(comb - comb_ref).max() if comb.size else 0.0
    assert err <= combine_atol(k), ("combine", err)
    offsets, rows, pos = oracle.dispatch(ids_ref, E)
    assert np.array_equal(route.counts[l].cpu().numpy(), np.diff(offsets)), "counts"
    if route.offsets is not None:
        assert np.array_equal(route.offsets[l].cpu().numpy(), offsets), "offsets"
        assert np.array_equal(route.rows[l].cpu().numpy(), rows), "rows"
        assert np.array_equal(route.pos[l].cpu().numpy(), pos), "pos"


def run_routing(dl, z_cpu, k, gate, **kw):
    z = z_cpu.to("cuda")
    L, T, E = z.shape
    route = dl.routing(z, k, gate, **kw)
    st = dl.device_status(route.workspace)
    assert st == 0, dl.status_string(st)
    return route


# fast kernel: E in {32, 64, 128}, k in {1, 2, 4, 8}; generic kernel otherwise
@pytest.mark.parametrize("T,E,k,L,gate,ties", [
    (4096 + 33, 128, 8, 1, 0, False),
    (4096 + 33, 128, 8, 2, 1, True),
    (1000, 64, 4, 3, 0, True),
    (300, 32, 2, 1, 1, False),
    (77, 128, 1, 2, 0, True),
    (1, 128, 8, 1, 0, False),
    (2500, 33, 5, 2, 0, True),       # generic
    (640, 256, 8, 1, 1, False),      # generic
    (97, 16, 16, 1, 0, True),        # k = E
    (500, 130, 100, 1, 0, True),     # one signature word per dispatch chunk
])
def test_routing_matches_oracle(dl, T, E, k, L, gate, ties):
    z = workloads.random_logits(T, E, L=L, seed=T + 7 * E + k, ties=ties)
    route = run_routing(dl, z, k, gate)
    for l in range(L):
        check_layer(route, l, z[l].numpy(), k, gate, E)


def test_routing_workloads_c2_c3(dl):
    for name in ("c2", "c3"):
        w = workloads.get(name)
        z = workloads.logits(w)
        route = run_routing(dl, z, w.k, w.gate)
        check_layer(route, 0, z[0].numpy(), w.k, w.gate, w.E)


@pytest.mark.parametrize("shift", [-120.0, -30.0, 60.0])
@pytest.mark.parametrize("gate", [0, 1])
def test_routing_far_from_zero(dl, shift, gate):
    """All chosen logits far below zero: the sigmoid-norm weights are ratios of
    tiny sigmoids, which the kernels take without forming them; far above
    zero every chosen sigmoid is near one."""
    z = workloads.random_logits(1000, 128, seed=5, ties=True) * 4.0 + shift
    route = run_routing(dl, z, 8, gate)
    check_layer(route, 0, z[0].numpy(), 8, gate, 128)


def test_unaligned_outputs_take_the_generic_kernel(dl):
    """expert_ids and combine 4- but not 16-byte aligned: same results."""
    T, E, k = 2000, 128, 8
    z = workloads.random_logits(T, E, seed=9, ties=True)
    route = dl.Routing(1, T, E, k)
    ids_store = torch.empty(T * k + 1, dtype=torch.int32, device="cuda")
    comb_store = torch.empty(T * k + 1, dtype=torch.float32, device="cuda")
    route.expert_ids = ids_store[1:].view(1, T, k)
    route.combine = comb_store[1:].view(1, T, k)
    assert route.expert_ids.data_ptr() % 16 != 0
    dl.routing(z.cuda(), k, 0, out=route)
    assert dl.device_status(route.workspace) == 0
    check_layer(route, 0, z[0].numpy(), k, 0, E)


def test_dispatch_arrays_are_optional(dl):
    T, E, k = 3000, 64, 8
    z = workloads.random_logits(T, E, seed=12)
    route = dl.Routing(1, T, E, k, with_dispatch=False)
    dl.routing(z.cuda(), k, 0, out=route)
    assert dl.device_status(route.workspace) == 0
    check_layer(route, 0, z[0].numpy(), k, 0, E)


@pytest.mark.parametrize("T,E,k,L,gate", [(65536, 128, 8, 1, 0), (4096 + 33, 128, 4, 2, 0),
                                           (2000, 64, 8, 1, 1), (1500, 33, 3, 1, 0)])
def test_routed_loss_is_the_plain_loss_plus_routing(dl, T, E, k, L, gate):
    """do_forward_backward_routed writes the same loss, gradient, signatures,
    counts and D as do_forward_backward (bit for bit) and the routing outputs
    of do_routing."""
    z = workloads.random_logits(T, E, L=L, seed=T + E, ties=True).cuda()
    plain = dl.forward_backward(z, k, gate)
    out, route = dl.forward_backward_routed(z, k, gate)
    assert dl.device_status(out.workspace) == 0
    assert dl.device_status(plain.workspace) == 0
    for name in ("bits", "counts", "D", "loss", "origin_do", "dlogits"):
        assert torch.equal(getattr(out, name), getattr(plain, name)), name
    alone = dl.routing(z, k, gate)
    assert dl.device_status(alone.workspace) == 0
    for name in ("expert_ids", "combine", "offsets", "rows", "pos"):
        assert torch.equal(getattr(route, name), getattr(alone, name)), name
    route.counts = out.counts
    zc = z.cpu()
    for l in range(L):
        check_layer(route, l, zc[l].numpy(), k, gate, E)


def test_routing_is_reproducible(dl):
    z = workloads.random_logits(20000, 128, seed=3, ties=True).cuda()
    a = dl.routing(z, 8, 0)
    b = dl.routing(z, 8, 0)
    for name in ("expert_ids", "combine", "counts", "offsets", "rows", "pos"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
