"""Pins of the routing-output oracle (Sec. 3.1.1) against what the paper and
the mathematics fix: a worked example derived by hand, library sorts, and
the identities that make the re-normalized weights independent of the dense
normaliser.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_z(T, E, seed, ties=False):
    z = workloads.random_logits(T, E, seed=seed, ties=ties)[0].numpy()
    return np.ascontiguousarray(z, np.float32)


def _sym(v):
    ln2, ln3 = np.log(2.0), np.log(3.0)
    table = {"0": 0.0, "1": 1.0, "ln2": ln2, "-ln2": -ln2, "ln3": ln3, "-ln3": -ln3}
    return table[v]


def test_route_worked_example():
    g = json.load(open(os.path.join(GOLDEN, "route_worked_n4_k2.json")))
    z = np.array([[_sym(v) for v in row] for row in g["logits_symbolic"]], np.float32)
    k = g["K"]
    for gate, key in ((oracle.GATE_SIGMOID_NORM, "combine_sigmoid_norm"),
                      (oracle.GATE_SOFTMAX, "combine_softmax")):
        ids, comb = oracle.route(z, k, gate)
        assert ids.tolist() == g["expert_ids"]
        want = np.array([[float(Fraction(x)) for x in row] for row in g[key]])
        # the logits are fp32 roundings of ln 2 and ln 3: agreement to their rounding
        np.testing.assert_allclose(comb, want, rtol=0, atol=1e-7)
    offsets, rows, pos = oracle.dispatch(np.array(g["expert_ids"], np.int32), g["n"])
    assert offsets.tolist() == g["expert_offsets"]
    assert rows.tolist() == g["dispatch_rows"]
    assert pos.tolist() == g["dispatch_pos"]


@pytest.mark.parametrize("E,k,ties", [(5, 1, False), (8, 2, True), (13, 4, True), (16, 16, False),
                                      (33, 8, True), (128, 8, True)])
def test_route_ids_are_a_stable_descending_sort(E, k, ties):
    """ids[t] = the first k entries of the logits sorted by value descending,
    equal values in index order (numpy's stable sort of -z)."""
    z = rand_z(157, E, seed=E * 7 + k, ties=ties)
    ids, _ = oracle.route(z, k)
    want = np.argsort(-z.astype(np.float64), axis=1, kind="stable")[:, :k]
    np.testing.assert_array_equal(ids, want)
    # the same set as the load bits f of Eq. 1
    f = oracle.select(z, k)
    onehot = np.zeros_like(f)
    np.put_along_axis(onehot, ids.astype(np.int64), 1, axis=1)
    np.testing.assert_array_equal(onehot, f)


@pytest.mark.parametrize("E,k", [(8, 2), (33, 5), (128, 8)])
def test_sigmoid_norm_weights_are_ratios_of_chosen_sigmoids(E, k):
    """p_i / sum_chosen p = s_i / sum_chosen s: the dense normaliser cancels."""
    z = rand_z(120, E, seed=E + 3 * k)
    ids, comb = oracle.route(z, k, oracle.GATE_SIGMOID_NORM)
    zc = torch.from_numpy(np.take_along_axis(z, ids.astype(np.int64), axis=1)).double()
    s = torch.sigmoid(zc)
    np.testing.assert_allclose(comb, (s / s.sum(1, keepdim=True)).numpy(), rtol=1e-13, atol=0)


@pytest.mark.parametrize("E,k", [(8, 2), (33, 5), (128, 8)])
def test_softmax_weights_are_the_softmax_of_the_chosen_logits(E, k):
    """softmax(z)_i / sum_chosen softmax(z) = softmax over the chosen logits."""
    z = rand_z(120, E, seed=5 * E + k)
    ids, comb = oracle.route(z, k, oracle.GATE_SOFTMAX)
    zc = torch.from_numpy(np.take_along_axis(z, ids.astype(np.int64), axis=1)).double()
    np.testing.assert_allclose(comb, torch.softmax(zc, dim=1).numpy(), rtol=1e-13, atol=1e-16)


@pytest.mark.parametrize("gate", [oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX])
def test_k_equal_e_keeps_the_dense_gate_and_k1_weighs_one(gate):
    z = rand_z(64, 16, seed=11)
    ids, comb = oracle.route(z, 16, gate)
    dense = np.take_along_axis(oracle.gate(z, gate), ids.astype(np.int64), axis=1)
    np.testing.assert_allclose(comb, dense, rtol=1e-14, atol=0)
    _, one = oracle.route(z, 1, gate)
    assert (one == 1.0).all()


@pytest.mark.parametrize("T,E,k", [(1, 4, 1), (97, 8, 2), (300, 33, 5), (1000, 128, 8)])
def test_dispatch_is_a_stable_sort_by_expert(T, E, k):
    ids, _ = oracle.route(rand_z(T, E, seed=T + E, ties=True), k)
    offsets, rows, pos = oracle.dispatch(ids, E)
    e_flat = ids.reshape(-1).astype(np.int64)
    t_flat = np.repeat(np.arange(T), k)
    order = np.lexsort((t_flat, e_flat))            # expert first, then token
    np.testing.assert_array_equal(rows, t_flat[order])
    inv = np.empty(T * k, np.int64)
    inv[order] = np.arange(T * k)
    np.testing.assert_array_equal(pos.reshape(-1), inv)
    np.testing.assert_array_equal(offsets, np.concatenate([[0], np.cumsum(np.bincount(e_flat, minlength=E))]))
    np.testing.assert_array_equal(np.diff(offsets), oracle.counts(oracle.select(rand_z(T, E, seed=T + E, ties=True), k)))
    assert offsets[-1] == T * k
    for e in range(E):
        seg = rows[offsets[e]:offsets[e + 1]]
        assert (np.diff(seg) > 0).all()             # each token once, ascending
        assert all(e in ids[t] for t in seg)


@pytest.mark.parametrize("gate", [oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX])
@pytest.mark.parametrize("E,k", [(8, 2), (33, 5), (128, 8)])
def test_route_backward_matches_autograd(gate, E, k):
    """The combine weights' gradient to the logits against torch float64
    autograd through the paper's definition (dense p, then re-normalized over
    the chosen experts), the selection held fixed."""
    T = 50
    z = rand_z(T, E, seed=E * 3 + k + gate)
    ids, _ = oracle.route(z, k, gate)
    g = np.random.default_rng(E + k).standard_normal((T, k))
    zt = torch.from_numpy(z.astype(np.float64)).requires_grad_(True)
    if gate == oracle.GATE_SOFTMAX:
        p = torch.softmax(zt, dim=1)
    else:
        s = torch.sigmoid(zt)
        p = s / s.sum(1, keepdim=True)
    pc = torch.gather(p, 1, torch.from_numpy(ids.astype(np.int64)))
    w = pc / pc.sum(1, keepdim=True)
    (w * torch.from_numpy(g)).sum().backward()
    dz = oracle.route_backward(z, ids, g, gate)
    np.testing.assert_allclose(dz, zt.grad.numpy(), rtol=1e-10, atol=1e-13)
    # the experts not chosen get nothing
    mask = np.ones_like(dz, dtype=bool)
    np.put_along_axis(mask, ids.astype(np.int64), False, axis=1)
    assert (dz[mask] == 0.0).all()


@pytest.mark.parametrize("c", [0.0, 3.0, 60.0, -60.0])
@pytest.mark.parametrize("gate", [oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX])
def test_route_backward_equal_chosen_logits_closed_form(c, gate):
    """All chosen logits equal to c (the rest far below): w = 1/k, so
    dz_l = (1/k) (g_l - mean g) for softmax and (1/k) sigmoid(-c) (g_l - mean g)
    for sigmoid-norm, at every size of c (1 - sigmoid(c) is tiny for c = 60)."""
    T, E, k = 20, 16, 5
    z = np.full((T, E), c - 200.0, np.float32)
    z[:, 3:3 + k] = c
    ids, _ = oracle.route(z, k, gate)
    assert (np.sort(ids, 1) == np.arange(3, 3 + k)).all()
    g = np.random.default_rng(1).standard_normal((T, k))
    dz = oracle.route_backward(z, ids, g, gate)
    factor = 1.0 if gate == oracle.GATE_SOFTMAX else 1.0 / (1.0 + np.exp(c))
    want = (g - g.mean(1, keepdims=True)) / k * factor
    np.testing.assert_allclose(np.take_along_axis(dz, ids.astype(np.int64), axis=1), want,
                               rtol=1e-12, atol=0)


def _value(v):
    if v.lstrip("-") == "sig(-1)":
        x = 1.0 / (1.0 + np.e)
        return -x if v.startswith("-") else x
    return float(Fraction(v))


def test_route_backward_worked_example():
    """The combine weights' gradient on the hand-worked tokens of the routing
    example (tests/golden/route_backward_worked_n4_k2.json)."""
    g = json.load(open(os.path.join(GOLDEN, "route_backward_worked_n4_k2.json")))
    z = np.array([[_sym(v) for v in row] for row in g["logits_symbolic"]], np.float32)
    ids = np.array(g["expert_ids"], np.int32)
    grad = np.array(g["grad_combine"], np.float64)
    for gate, key in ((oracle.GATE_SIGMOID_NORM, "dlogits_sigmoid_norm"),
                      (oracle.GATE_SOFTMAX, "dlogits_softmax")):
        got_ids, _ = oracle.route(z, g["K"], gate)
        assert got_ids.tolist() == g["expert_ids"]
        want = np.array([[_value(v) for v in row] for row in g[key]])
        dz = oracle.route_backward(z, ids, grad, gate)
        # the logits are fp32 roundings of ln 2 and ln 3: agreement to their rounding
        np.testing.assert_allclose(dz, want, rtol=0, atol=2e-7)
        assert (dz[want == 0] == 0).all()
