"""Full-size parity of the workloads that the benchmark does not time.

* collapse (E=128, k=8, T=262144, biased experts and exact ties): element by
  element against the oracle (its loss and gradient run in O(T E^2)).
* the long window (E=256, k=8, T=2^20): one layer, and all 48 layers in one
  launch.  Signatures, counts, D and origin_do exactly against the oracle's
  selection, packing and population-count Hamming matrix; the loss against
  the oracle's Eq. do_loss with its direction term C summed over token ranges
  in worker processes (oracle_pool); dlogits on whole 65536-token slices at
  the start, middle and end of the window through the oracle's per-range
  gradient with the full D.  In the 48-layer launch every layer is also held
  to Eq. zero_sum and the shape of D (symmetric, zero diagonal), and three
  layers (first, middle, last) to the oracle as above.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

pytestmark = pytest.mark.gpu

LOSS_RTOL = 1e-5
GRAD_TOL = 1e-4


@pytest.fixture(scope="module")
def dl():
    import paper_2609_32398_gb300.doloss as m

    m.lib()
    return m


def run(dl, z, k, gate):
    out = dl.forward_backward(z.cuda(), k, gate=gate)
    assert dl.device_status(out.workspace) == 0
    return out


def test_collapse_full_size_elementwise(dl):
    w = workloads.get("collapse")
    z = workloads.logits(w)
    out = run(dl, z, w.k, w.gate)
    ref = oracle.forward_backward(z[0].numpy(), w.k, w.gate)
    assert np.array_equal(out.bits[0].cpu().numpy().view(np.uint32), ref["bits"])
    assert np.array_equal(out.counts[0].cpu().numpy(), ref["counts"])
    assert np.array_equal(out.D[0].cpu().numpy(), ref["D"])
    assert int(out.origin_do[0]) == ref["origin_do"]
    assert float(out.loss[0]) == pytest.approx(ref["loss"], rel=LOSS_RTOL)
    g = out.dlogits[0].double().cpu().numpy()
    assert np.abs(g - ref["dz"]).max() / np.abs(ref["dz"]).max() <= GRAD_TOL


SLICE = 65536


def oracle_loss_full(z, f, D, k, gate):
    """Eq. do_loss by the oracle, C summed over token ranges in spawned workers."""
    from tests.oracle_pool import direction_parallel

    return oracle.loss(D, direction_parallel(z, f, gate), z.shape[0], k)


def check_layer_against_oracle(out, l, zn, k, gate):
    """Layer l of a fused call: exact integers, the loss, and dlogits on three
    whole slices of SLICE tokens."""
    T, E = zn.shape
    f = oracle.select(zn, k)
    bits = oracle.pack(f)
    D = oracle.hamming_bits(bits, T)
    assert np.array_equal(out.bits[l].cpu().numpy().view(np.uint32), bits), "bits"
    assert np.array_equal(out.counts[l].cpu().numpy(), oracle.counts(f)), "counts"
    assert np.array_equal(out.D[l].cpu().numpy(), D), "D"
    assert int(out.origin_do[l]) == oracle.origin_do(D), "origin_do"
    want = oracle_loss_full(zn, f, D, k, gate)
    assert abs(float(out.loss[l]) - want) <= LOSS_RTOL * abs(want), ("loss", float(out.loss[l]), want)
    for t0 in (0, T // 2 - SLICE // 2, T - SLICE):
        t1 = t0 + SLICE
        g = oracle.dloss_dp(D, f, T, k, t0=t0, t1=t1)
        dz = oracle.gate_backward(zn, g, gate, t0=t0, t1=t1)[t0:t1]
        err = np.abs(out.dlogits[l, t0:t1].double().cpu().numpy() - dz).max()
        assert err <= GRAD_TOL * np.abs(dz).max(), (l, t0, err)


def test_long_window_layer_full_size(dl):
    w = workloads.get("long", L=1)
    z = workloads.logits(w)
    out = run(dl, z, w.k, w.gate)
    check_layer_against_oracle(out, 0, z[0].numpy(), w.k, w.gate)


def test_long_window_all_layers_in_one_launch(dl):
    """The long-window recipe as specified: L = 48 layers of E=256, k=8,
    T=2^20 in one call (about 100 GB of device memory)."""
    w = workloads.get("long")
    T, E, k = w.T, w.E, w.k
    z = workloads.logits(w, device="cuda")
    out = run(dl, z, k, w.gate)
    torch.cuda.synchronize()
    # every layer: Eq. zero_sum (sum_i n_i = T k and sum_ij D_ij = 2 T k (E - k)),
    # D symmetric with a zero diagonal, the loss finite
    n_sum = out.counts.sum(dim=1, dtype=torch.int64).cpu()
    d_sum = out.D.sum(dim=(1, 2), dtype=torch.int64).cpu()
    assert (n_sum == T * k).all(), n_sum
    assert (d_sum == 2 * T * k * (E - k)).all(), d_sum
    assert torch.equal(out.D, out.D.transpose(1, 2))
    assert (out.D.diagonal(dim1=1, dim2=2) == 0).all()
    assert torch.isfinite(out.loss).all()
    for l in (0, w.L // 2 - 1, w.L - 1):
        check_layer_against_oracle(out, l, z[l].cpu().numpy(), k, w.gate)
