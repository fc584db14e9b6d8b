"""CPU oracle for the consumers of the per-expert counts (test infrastructure
only): the MaxVio load-imbalance metric (App. E) and the Replica Expert
Mechanism's global-batch replica allocation (Sec. 3.2, Eq. benefit_score;
App. B.1, Algorithm rem_allocation).

Only the tests, the package smoke check and the benchmark's CPU-baseline leg
use it; the product path never imports it.  It shares no code with the CUDA
library.  Plain Python loops in double precision, the steps in the paper's
order.  Pins live in ``tests/test_oracle_rem.py``.

Readings where the paper is silent:
  * An expert e is sent from its home rank (the rank that holds its original
    parameters, ``expert_rank[e]``); a replica is never placed on the home
    rank, nor twice on one rank.
  * Loads and token volumes are real numbers (the controller works on moving
    averages); tau is fixed before the loop, as Algorithm rem_allocation
    computes it once, from the loads summed in rank order; the floor of the
    second case is taken as printed.
  * Ties: the least-loaded rank with the lowest index; among equal scores the
    lowest expert index.
  * A rank is full when it holds D replicas; the loop ends when every rank is
    full or the best score of the chosen receiver is not positive.
  * MaxVio of a batch without tokens (tau = 0) is 0.
"""
from __future__ import annotations

import math

import numpy as np


def rank_loads(counts, expert_rank, R):
    """L_r = sum of the token counts of the experts that reside on rank r (App. E)."""
    L = [0] * R
    for e, n in enumerate(counts):
        L[int(expert_rank[e])] += int(n)
    return L


def maxvio(loads):
    """App. E: MaxVio = max_r |L_r / tau - 1|, tau = (1/|R|) sum_r L_r.  A batch
    without tokens (tau = 0) has no violation: 0."""
    R = len(loads)
    tau = sum(float(x) for x in loads) / R
    if tau == 0.0:
        return 0.0
    return max(abs(float(x) / tau - 1.0) for x in loads)


def benefit_score(T_e, L_s, L_r, tau):
    """Eq. benefit_score: the tokens the receiving rank (load L_r) can take over
    from the sending rank (load L_s) for an expert with token volume T_e."""
    if L_r < tau and L_s > tau:
        return min(tau - L_r, T_e, L_s - tau)
    if L_r >= tau and L_s > L_r:
        return min(math.floor((L_s - L_r) / 2.0), T_e)
    return -1.0


def rem_allocate(loads, expert_tokens, expert_rank, D):
    """Algorithm rem_allocation.  Returns (placements, loads): placements is the
    list of (e, r_s, r_r, delta) in the order they were made; loads the updated
    load estimates."""
    L = [float(x) for x in loads]
    T = [float(x) for x in expert_tokens]
    R = len(L)
    total = 0.0
    for x in L:                 # the loads summed in rank order
        total += x
    tau = total / R
    placed = [[] for _ in range(R)]        # experts replicated on each rank
    A = []
    while True:
        open_ranks = [r for r in range(R) if len(placed[r]) < D]
        if not open_ranks:
            break
        r_r = min(open_ranks, key=lambda r: (L[r], r))
        best, best_e = None, None
        for e in range(len(T)):
            r_s = int(expert_rank[e])
            if r_s == r_r or e in placed[r_r]:
                continue
            s = benefit_score(T[e], L[r_s], L[r_r], tau)
            if best is None or s > best:
                best, best_e = s, e
        if best is None or best <= 0:
            break
        e, r_s = best_e, int(expert_rank[best_e])
        A.append((e, r_s, r_r, best))
        placed[r_r].append(e)
        L[r_r] += best
        L[r_s] -= best
        T[e] -= best
    return A, L


def maxvio_layers(counts_layers, expert_rank, R):
    """MaxVio of every layer's counts [L][E] for one expert-to-rank map."""
    return np.array([maxvio(rank_loads(c, expert_rank, R)) for c in counts_layers], np.float64)
