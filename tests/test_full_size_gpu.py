"""Full-size parity of the workloads that the benchmark does not time.

* collapse (E=128, k=8, T=262144, biased experts and exact ties): element by
  element against the oracle (its loss and gradient run in O(T E^2)).
* one layer of the long window (E=256, k=8, T=2^20, the generic kernels):
  signatures, counts, D and origin_do exactly against the oracle's selection,
  packing and population-count Hamming matrix; dlogits on sampled token ranges
  through the oracle's per-range gradient with the full D; the loss against
  the factored form w_it = f_it R_i - sum_{j in S_t} D_ij evaluated in numpy
  (the factored form is pinned to the literal double sum in the CPU tests).
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


def factored_loss(z, f, D, k, gate, chunk=8192):
    """(1/(T^2 k)) sum_t sum_i p_it w_it in float64, chunk by chunk."""
    T, E = z.shape
    R = D.sum(axis=1).astype(np.float64)
    acc = 0.0
    for t0 in range(0, T, chunk):
        zc = z[t0:t0 + chunk].astype(np.float64)
        fc = f[t0:t0 + chunk]
        if gate == workloads.GATE_SIGMOID_NORM:
            s = 1.0 / (1.0 + np.exp(-zc))
            p = s / s.sum(axis=1, keepdims=True)
        else:
            e = np.exp(zc - zc.max(axis=1, keepdims=True))
            p = e / e.sum(axis=1, keepdims=True)
        sel = np.argsort(1 - fc.astype(np.int16), axis=1, kind="stable")[:, :k]  # the k selected
        gathered = D[sel].sum(axis=1).astype(np.float64)           # sum_{j in S_t} D_j.
        wv = fc * R[None, :] - gathered
        acc += float((p * wv).sum())
    return acc / (float(T) * T * k)


def test_long_window_layer_full_size(dl):
    w = workloads.get("long", L=1)
    z = workloads.logits(w)
    T, E, k = w.T, w.E, w.k
    out = run(dl, z, k, w.gate)
    zn = z[0].numpy()
    f = oracle.select(zn, k)
    bits = oracle.pack(f)
    D = oracle.hamming_bits(bits, T)
    assert np.array_equal(out.bits[0].cpu().numpy().view(np.uint32), bits)
    assert np.array_equal(out.counts[0].cpu().numpy(), oracle.counts(f))
    assert np.array_equal(out.D[0].cpu().numpy(), D)
    assert int(out.origin_do[0]) == oracle.origin_do(D)
    ref_loss = factored_loss(zn, f, D, k, w.gate)
    assert float(out.loss[0]) == pytest.approx(ref_loss, rel=LOSS_RTOL)
    gpu_dz = out.dlogits[0]
    scale = None
    for t0 in (0, T // 2 - 37, T - 64):
        t1 = t0 + 64
        g = oracle.dloss_dp(D, f, T, k, t0=t0, t1=t1)
        dz = oracle.gate_backward(zn, g, w.gate, t0=t0, t1=t1)[t0:t1]
        scale = np.abs(dz).max() if scale is None else max(scale, np.abs(dz).max())
        err = np.abs(gpu_dz[t0:t1].double().cpu().numpy() - dz).max()
        assert err <= GRAD_TOL * np.abs(dz).max(), (t0, err)
