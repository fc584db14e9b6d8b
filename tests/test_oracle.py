"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every oracle function is checked here against something other than itself:
brute force on tiny inputs, library routines (torch.cdist, torch autograd),
the paper's closed forms (Eq. zero_sum, App. A, App. C.2, App. C.3), metric
axioms, finite differences, and the relation between the straight-through
gradient (Sec. 3.1.2) and the surrogate (Sec. 3.1.3).
"""
import itertools
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_z(T, E, seed, ties=False):
    z = workloads.random_logits(T, E, seed=seed, ties=ties)[0].numpy()
    return np.ascontiguousarray(z, np.float32)


# ---------------------------------------------------------------- selection

@pytest.mark.parametrize("E,k,ties", [(5, 1, False), (8, 2, True), (13, 4, True), (16, 16, False),
                                      (33, 8, True), (7, 6, True)])
def test_select_matches_bruteforce_sort(E, k, ties):
    z = rand_z(97, E, seed=E * 31 + k, ties=ties)
    f = oracle.select(z, k)
    for t in range(z.shape[0]):
        want = sorted(range(E), key=lambda i: (-float(z[t, i]), i))[:k]
        got = sorted(np.nonzero(f[t])[0].tolist())
        assert got == sorted(want), (t, z[t], got, want)
    assert (f.sum(1) == k).all()


def test_select_degenerate_rows():
    E, k = 12, 5
    z = np.zeros((3, E), np.float32)
    z[1, :] = -2.5                       # all equal -> lowest k indices
    z[2, :] = 0.0
    z[2, 3] = -0.0                       # -0 ties +0; index decides
    f = oracle.select(z, k)
    for t in range(3):
        assert f[t, :k].all() and not f[t, k:].any()
    assert oracle.select(rand_z(5, E, 3), E).all()            # k = E selects all


# ---------------------------------------------------------------- packing and counts

def test_pack_layout_and_padding():
    T, E = 70, 3                         # two full words and a ragged third
    f = np.zeros((T, E), np.uint8)
    f[0, 0] = f[31, 0] = f[32, 1] = f[69, 2] = 1
    bits = oracle.pack(f)
    assert bits.shape == (3, 3)
    assert bits[0, 0] == (1 | (1 << 31)) and bits[0, 1] == 0 and bits[0, 2] == 0
    assert bits[1, 1] == 1 and bits[2, 2] == (1 << (69 - 64))
    z = rand_z(T, 9, 4)
    fb = oracle.pack(oracle.select(z, 3))
    assert (fb[:, -1] >> (T % 32) == 0).all()                # pad bits are zero


def test_counts_sum_to_mk():
    z = rand_z(301, 17, 5)
    f = oracle.select(z, 6)
    n = oracle.counts(f)
    assert n.sum() == 301 * 6
    assert (n == f.sum(0)).all()


# ---------------------------------------------------------------- Hamming matrix

@pytest.mark.parametrize("T,E,k", [(64, 8, 2), (77, 16, 5), (200, 33, 8)])
def test_hamming_matches_cdist_and_bits(T, E, k):
    z = rand_z(T, E, seed=T + E, ties=True)
    f = oracle.select(z, k)
    D = oracle.hamming(f)
    F = torch.from_numpy(f.T.astype(np.float64))          # [E, T] signatures
    ref = torch.cdist(F, F, p=0).round().to(torch.int64).numpy()
    assert (D == ref).all()
    assert (oracle.hamming_bits(oracle.pack(f), T) == D).all()


def test_zero_sum_constraint():
    for (T, E, k) in [(100, 8, 2), (257, 32, 8), (64, 12, 12), (50, 9, 1)]:
        f = oracle.select(rand_z(T, E, seed=T * E), k)
        D = oracle.hamming(f)
        assert D.sum() == 2 * T * k * (E - k)                # Eq. zero_sum


def test_metric_axioms_and_cooccurrence_identity():
    T, E, k = 150, 14, 4
    f = oracle.select(rand_z(T, E, 11, ties=True), k)
    D = oracle.hamming(f).astype(np.int64)
    assert (np.diag(D) == 0).all() and (D == D.T).all()
    assert (D[:, :, None] <= D[:, None, :] + D.T[None, :, :]).all()   # D_ij <= D_il + D_lj
    n = oracle.counts(f).astype(np.int64)
    c = f.T.astype(np.int64) @ f.astype(np.int64)           # co-occurrence c_ij
    assert (D == n[:, None] + n[None, :] - 2 * c).all()     # App. C.3


def test_hamming_is_additive_over_token_shards():
    T, E, k = 300, 16, 4
    f = oracle.select(rand_z(T, E, 12), k)
    full = oracle.hamming(f)
    parts = oracle.hamming(f, 0, 111) + oracle.hamming(f, 111, 300)
    assert (full == parts).all()


# ---------------------------------------------------------------- worked example

def _equidistant_example():
    g = json.load(open(os.path.join(GOLDEN, "equidistant_n4_k2_m6.json")))
    z = np.zeros((g["m"], g["n"]), np.float32)
    for t, (a, b) in enumerate(g["subsets"]):
        z[t, a] = z[t, b] = 1.0
    return g, z


def test_worked_example_closed_forms():
    g, z = _equidistant_example()
    n, K, m = g["n"], g["K"], g["m"]
    f = oracle.select(z, K)
    cnt = oracle.counts(f)
    D = oracle.hamming(f)
    c = f.T.astype(np.int64) @ f.astype(np.int64)
    off = ~np.eye(n, dtype=bool)
    assert (cnt == g["counts_each"]).all() and g["counts_each"] == m * K // n
    assert (c[off] == g["cooccurrence_offdiag"]).all()
    assert g["cooccurrence_offdiag"] * n * (n - 1) == m * K * (K - 1)
    assert (D[off] == g["hamming_offdiag"]).all() and (np.diag(D) == 0).all()
    assert D.sum() == g["zero_sum_total"] == 2 * m * K * (n - K)
    assert g["d_star_all_pairs_mean"] * n * n == 2 * m * K * (n - K)


@pytest.mark.parametrize("gate", [oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX])
def test_worked_example_loss_from_appendix_a(gate):
    """At equidistance every off-diagonal G_ij equals d, so App. A's Step 2 gives
    sum_ij G_ij C_ij = d * m (n s_K - k) and L = d (n s_K - k) / (m k)."""
    g, z = _equidistant_example()
    n, K, m = g["n"], g["K"], g["m"]
    f = oracle.select(z, K)
    D = oracle.hamming(f)
    C = oracle.direction(z, f, gate)
    # p of a selected expert from the two-valued rows, in closed form
    if gate == oracle.GATE_SIGMOID_NORM:
        s1, s0 = 1.0 / (1.0 + np.exp(-1.0)), 0.5
    else:
        s1, s0 = np.e, 1.0
    p_sel = s1 / (K * s1 + (n - K) * s0)
    s_K = K * p_sel
    d = g["hamming_offdiag"]
    want = d * (n * s_K - K) / (m * K)
    assert oracle.loss(D, C, m, K) == pytest.approx(want, rel=1e-13)


# ---------------------------------------------------------------- gate and direction

def test_gate_invariants():
    z = rand_z(40, 10, 13)
    for gk in (oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX):
        p = oracle.gate(z, gk)
        np.testing.assert_allclose(p.sum(1), 1.0, rtol=0, atol=1e-14)
        order = np.argsort(z, axis=1, kind="stable")
        assert (np.diff(np.take_along_axis(p, order, 1), axis=1) >= 0).all()   # monotone in z
    zero = np.zeros((2, 7), np.float32)
    np.testing.assert_allclose(oracle.gate(zero, oracle.GATE_SIGMOID_NORM), 1 / 7, rtol=1e-15)
    shifted = oracle.gate(z + np.float32(3.0), oracle.GATE_SOFTMAX)
    np.testing.assert_allclose(shifted, oracle.gate(z, oracle.GATE_SOFTMAX), rtol=1e-5)
    torch_sm = torch.softmax(torch.from_numpy(z).double(), 1).numpy()
    np.testing.assert_allclose(oracle.gate(z, oracle.GATE_SOFTMAX), torch_sm, rtol=1e-13)


def test_sum_of_direction_terms_appendix_a():
    """App. A, Step 2: sum_ij C_ij = m (n s_K - k) with s_K the mean Top-K mass."""
    T, E, k = 120, 12, 3
    z = rand_z(T, E, 14)
    f = oracle.select(z, k)
    for gk in (oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX):
        C = oracle.direction(z, f, gk)
        p = oracle.gate(z, gk)
        s_K = (p * f).sum() / T
        assert C.sum() == pytest.approx(T * (E * s_K - k), rel=1e-12)
        assert np.abs(np.diag(C)).max() == 0.0               # C_ii = 0


def test_uniform_probabilities_give_zero_loss():
    """All-equal logits: p = 1/n and sum_ij G_ij C_ij telescopes to zero."""
    T, E, k = 64, 8, 3
    z = np.full((T, E), 0.25, np.float32)
    z[::3, :] = -1.0
    f = oracle.select(rand_z(T, E, 15), k)                   # any selection
    D = oracle.hamming(f)
    for gk in (oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX):
        C = oracle.direction(z, f, gk)
        assert abs(oracle.loss(D, C, T, k)) < 1e-12


# ---------------------------------------------------------------- gradient

def _torch_surrogate_loss(z, f, D, k, gk, d_scale=1.0):
    """Eq. do_loss built from torch ops with G and F as constants."""
    zt = torch.from_numpy(z).double().requires_grad_(True)
    if gk == oracle.GATE_SOFTMAX:
        p = torch.softmax(zt, 1)
    else:
        s = torch.sigmoid(zt)
        p = s / s.sum(1, keepdim=True)
    F = torch.from_numpy(f).double()                         # [T, E]
    G = torch.from_numpy(D).double() * d_scale
    T = z.shape[0]
    # C_ij = sum_t p_it f_it - sum_t p_it f_jt
    C = (p * F).sum(0)[:, None] - p.T @ F
    L = (G * C).sum() / (T * T * k)
    return zt, L


@pytest.mark.parametrize("gk", [oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX])
def test_gradient_matches_torch_autograd(gk):
    T, E, k = 90, 11, 3
    z = rand_z(T, E, 16, ties=True)
    f = oracle.select(z, k)
    D = oracle.hamming(f)
    zt, L = _torch_surrogate_loss(z, f, D, k, gk, d_scale=0.75)
    L.backward()
    g = oracle.dloss_dp(D, f, T, k, d_scale=0.75)
    dz = oracle.gate_backward(z, g, gk, grad_scale=2.5)
    np.testing.assert_allclose(dz, 2.5 * zt.grad.numpy(), rtol=1e-10, atol=1e-16)
    C = oracle.direction(z, f, gk)
    assert oracle.loss(D, C, T, k, d_scale=0.75) == pytest.approx(L.item(), rel=1e-12)


@pytest.mark.parametrize("zbig", [40.0, 60.0, -60.0])
def test_sigmoid_gate_backward_at_saturated_logits(zbig):
    """Sigmoid-norm gate backward where s is within 1e-17 of 1 (or of 0): the
    Jacobian factor s (1 - s) must come out as sigmoid(z) sigmoid(-z), not as
    the cancelled 1 - s.  Pinned to a 50-digit numerical derivative of
    p_i(z) = s_i / sum_j s_j (mpmath), independent of the oracle's formula."""
    mpmath = pytest.importorskip("mpmath")
    mp = mpmath.mp
    mp.dps = 50
    z = np.array([[zbig, 0.5, -1.0, 2.0]], np.float32)
    g = np.array([[1.5, -0.25, 0.75, 0.0]], np.float64)
    dz = oracle.gate_backward(z, g, oracle.GATE_SIGMOID_NORM, grad_scale=1.0)[0]

    def p_dot_g(zz):
        s = [1 / (1 + mpmath.exp(-v)) for v in zz]
        S = sum(s)
        return sum(mpmath.mpf(float(g[0, i])) * s[i] / S for i in range(4))

    zm = [mpmath.mpf(float(v)) for v in z[0]]
    for l in range(4):
        def along(h, l=l):
            zz = list(zm)
            zz[l] = zz[l] + h
            return p_dot_g(zz)
        want = float(mpmath.diff(along, 0))
        assert dz[l] == pytest.approx(want, rel=1e-12, abs=1e-300), (l, dz[l], want)
    assert dz[0] != 0.0


def test_straight_through_gradient_is_four_times_surrogate():
    """Sec. 3.1.2: with F_i -> P_i + sg[F_i - P_i], the origin loss keeps the value
    sum_{i!=j} ||F_i - F_j||^2 (Eq. origin_do) and its gradient in p_it is
    4 sum_j G_ij (f_it - f_jt), four times the surrogate's unnormalized one."""
    T, E, k = 40, 7, 2
    z = rand_z(T, E, 17)
    f = oracle.select(z, k)
    D = oracle.hamming(f)
    p = torch.from_numpy(oracle.gate(z)).requires_grad_(True)
    F = torch.from_numpy(f).double()
    Fste = p + (F - p).detach()                              # [T, E]
    diff = Fste.T[:, None, :] - Fste.T[None, :, :]           # [E, E, T]
    L_ste = (diff.abs().sum(-1) ** 2).sum()                  # i == j terms are zero
    L_ste.backward()
    assert L_ste.item() == pytest.approx(oracle.origin_do(D), rel=1e-12)
    g = oracle.dloss_dp(D, f, T, k) * (T * T * k)
    np.testing.assert_allclose(p.grad.numpy(), 4.0 * g, rtol=1e-12, atol=1e-12)


def test_origin_do_is_the_variance_of_distances():
    """App. C.1: under the fixed total, sum_{i!=j} G_ij^2 = n(n-1)(var + mean^2)."""
    T, E, k = 200, 10, 3
    f = oracle.select(rand_z(T, E, 18), k)
    D = oracle.hamming(f).astype(np.float64)
    off = D[~np.eye(E, dtype=bool)]
    mean = 2 * T * k * (E - k) / (E * (E - 1))
    assert off.mean() == pytest.approx(mean, rel=1e-14)
    assert oracle.origin_do(D.astype(np.int32)) == pytest.approx(E * (E - 1) * (off.var() + mean ** 2),
                                                                 rel=1e-12)


def test_gradient_matches_finite_differences():
    """Central differences of Eq. do_loss in z with the selection and G frozen."""
    T, E, k = 12, 6, 2
    z = rand_z(T, E, 19)
    f = oracle.select(z, k)
    D = oracle.hamming(f)
    for gk in (oracle.GATE_SIGMOID_NORM, oracle.GATE_SOFTMAX):
        dz = oracle.gate_backward(z, oracle.dloss_dp(D, f, T, k), gk)
        zd = z.astype(np.float64)
        for (t, l) in [(0, 0), (3, 2), (7, 5), (11, 1)]:
            h = 1e-3 * max(1.0, abs(zd[t, l]))
            vals = []
            for sgn in (+1, -1):
                zp = zd.copy()
                zp[t, l] += sgn * h
                # the oracle reads fp32 logits; evaluate the loss in double here
                # by perturbing through the direction term's definition
                zp32 = zp.astype(np.float32)
                hh = float(zp32[t, l] - np.float32(z[t, l]))
                vals.append((oracle.loss(D, oracle.direction(zp32, f, gk), T, k), hh))
            fd = (vals[0][0] - vals[1][0]) / (vals[0][1] - vals[1][1])
            assert fd == pytest.approx(dz[t, l], rel=2e-5, abs=1e-12)


# ---------------------------------------------------------------- collapse

def test_idle_experts_get_negative_gradient_appendix_c2():
    """App. C.2: for an idle expert i, G_ij = n_j and dL/dp_it is
    -1/(m^2 k) sum_{j in S_t} n_j < 0 on every token."""
    T, E, k = 128, 10, 2
    z = rand_z(T, E, 20)
    z[:, 7:] -= 50.0                                         # experts 7..9 never chosen
    f = oracle.select(z, k)
    n = oracle.counts(f)
    assert (n[7:] == 0).all()
    D = oracle.hamming(f)
    for i in range(7, 10):
        assert (D[i] == n).all()
    g = oracle.dloss_dp(D, f, T, k)
    want = -(f * n[None, :]).sum(1) / (T * T * k)
    for i in range(7, 10):
        np.testing.assert_allclose(g[:, i], want, rtol=1e-13)
        assert (g[:, i] < 0).all()


# ---------------------------------------------------------------- whole path

def test_forward_backward_is_the_composition_of_steps():
    T, E, k = 100, 16, 4
    z = rand_z(T, E, 21, ties=True)
    r = oracle.forward_backward(z, k, oracle.GATE_SIGMOID_NORM, d_scale=1.0, grad_scale=3.0)
    f = oracle.select(z, k)
    assert (r["bits"] == oracle.pack(f)).all()
    assert (r["counts"] == oracle.counts(f)).all()
    D = oracle.hamming(f)
    assert (r["D"] == D).all()
    C = oracle.direction(z, f)
    assert r["loss"] == pytest.approx(oracle.loss(D, C, T, k), rel=1e-14)
    assert r["origin_do"] == oracle.origin_do(D)
    dz = oracle.gate_backward(z, oracle.dloss_dp(D, f, T, k), grad_scale=3.0)
    np.testing.assert_allclose(r["dz"], dz, rtol=1e-14)


def test_global_do_scaling_is_linear_in_the_summed_matrix():
    """Eq. global_do: G^g = (1/|D|) sum_d G^d enters the loss linearly."""
    T, E, k = 80, 8, 2
    z = rand_z(T, E, 22)
    f = oracle.select(z, k)
    D1, D2 = oracle.hamming(f, 0, 40), oracle.hamming(f, 40, 80)
    C = oracle.direction(z, f)
    both = oracle.loss(D1 + D2, C, T, k, d_scale=0.5)
    assert both == pytest.approx(0.5 * (oracle.loss(D1, C, T, k) + oracle.loss(D2, C, T, k)), rel=1e-13)


def test_dense_p_reading_against_the_renormalized_one():
    """Sec. 3.1.1 gives p both dense and, after Top-K, re-normalized over the K
    chosen experts.  Mode 0 (dense) is the path's reading; checked here: it
    equals oracle.direction, and only it gives the idle experts of App. C.2 a
    gradient.  With re-normalized weights the experts outside a token's Top-K
    have p = 0 whatever their logits, and every idle expert's logit gradient
    (through the surrogate, G detached) vanishes; with the dense p it is
    negative (App. C.2: idle experts are pulled up)."""
    T, E, k = 60, 8, 2
    z = rand_z(T, E, 31)
    z[:, 6:] -= 6.0                                  # experts 6 and 7 never chosen
    f = oracle.select(z, k)
    assert not f[:, 6:].any()
    D = oracle.hamming(f)
    C0 = oracle.direction_mode(z, f, mode=0)
    np.testing.assert_allclose(C0, oracle.direction(z, f), rtol=1e-14, atol=1e-14)

    def loss_of(zz, mode):
        return oracle.loss(D, oracle.direction_mode(zz.astype(np.float32), f, mode=mode), T, k)

    for mode, sign in ((0, -1), (1, 0)):
        for i in (6, 7):
            h = 1e-2
            zp, zm = z.astype(np.float64).copy(), z.astype(np.float64).copy()
            zp[:, i] += h
            zm[:, i] -= h
            g = (loss_of(zp, mode) - loss_of(zm, mode)) / (2 * h)
            if sign == 0:
                assert abs(g) < 1e-12                # rounding of the cancelled normaliser only
            else:
                assert g < -1e-6
    # with re-normalized weights the chosen mass is one for every token
    # (App. A: s_K = 1), so sum C = m (n - k) exactly
    C1 = oracle.direction_mode(z, f, mode=1)
    assert C1.sum() == pytest.approx(T * (E - k), rel=1e-12)



def test_random_signatures_are_packed_selections():
    """The sweep generator's words unpack to a 0/1 matrix that the oracle packs
    back to the same words (bits past T zero), with about the asked density,
    and the oracle's word-wise distances equal its token-wise ones on them."""
    T, E, L = 1000 + 13, 9, 2
    bits = workloads.random_signatures(T, E, L, seed=4, density_log2=3)
    for l in range(L):
        f = np.zeros((T, E), np.uint8)
        for i in range(E):
            for t in range(T):
                f[t, i] = (int(bits[l, i, t // 32]) >> (t % 32)) & 1
        assert np.array_equal(oracle.pack(f), bits[l])
        assert abs(f.mean() - 1 / 8) < 0.02
        assert np.array_equal(oracle.hamming_bits(bits[l], T), oracle.hamming(f))
