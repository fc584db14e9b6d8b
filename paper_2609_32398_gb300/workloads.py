"""Seeded synthetic router logits shaped like the paper's MoE layers.

This module only draws inputs; it holds none of the DO-loss arithmetic.  The
same logits bytes go to the CUDA path and to the CPU oracle, so parity never
depends on which device drew them.

The paper trains on a proprietary corpus (Sec. 4.3) and publishes no router
outputs, so these draws stand in for real routing:

* ``tiny``      E=8,   k=2, T=1024:   X[1024,64] fp32 ~N(0,1), W[64,8] ~N(0,0.02), z = XW; seed 0.
* ``c2``        E=64,  k=8, T=16384:  X[T,1024] bf16 ~N(0,1), W[1024,64] bf16 ~N(0,0.02),
                                       z = X W in fp32 (4 sequences x 4096); seed 1.
* ``c3``        E=128, k=8, T=65536:  X[T,2048] bf16 ~N(0,1), W[2048,128] bf16 ~N(0,0.02),
                                       z = X W in fp32 (16 x 4096; the 30BA3B router, Sec. 4.1); seed 2.
* ``collapse``  E=128, k=8, T=262144: z ~N(0,1), +3 on experts 0-15, -3 on experts 16-47,
                                       and 5% of rows (seeded) rounded to multiples of 0.5 so
                                       that rows carry exact ties, also at the k-th place; seed 3.
* ``long``      E=256, k=8, T=2^20, L=48 layers: z ~N(0,1) + b_l with a per-layer
                                       per-expert bias b_l ~N(0,0.5); layer l uses seed 4000+l.

``T`` and ``L`` may be overridden to draw the same recipe at a smaller size.
"""
from __future__ import annotations

from dataclasses import dataclass, replace

import numpy as np
import torch

GATE_SIGMOID_NORM = 0
GATE_SOFTMAX = 1


@dataclass(frozen=True)
class Workload:
    name: str
    E: int
    k: int
    T: int
    L: int
    gate: int
    seed: int
    hidden: int = 0  # router input width for the X W recipes, 0 for direct draws

    def describe(self) -> str:
        return f"{self.name}: E={self.E} k={self.k} T={self.T} L={self.L}"


WORKLOADS = {
    "tiny": Workload("tiny", 8, 2, 1024, 1, GATE_SOFTMAX, 0, hidden=64),
    "c2": Workload("c2", 64, 8, 16384, 1, GATE_SIGMOID_NORM, 1, hidden=1024),
    "c3": Workload("c3", 128, 8, 65536, 1, GATE_SIGMOID_NORM, 2, hidden=2048),
    "collapse": Workload("collapse", 128, 8, 262144, 1, GATE_SIGMOID_NORM, 3),
    "long": Workload("long", 256, 8, 1 << 20, 48, GATE_SIGMOID_NORM, 4000),
}


def get(name: str, T: int | None = None, L: int | None = None) -> Workload:
    w = WORKLOADS[name]
    if T is not None:
        w = replace(w, T=int(T))
    if L is not None:
        w = replace(w, L=int(L))
    return w


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _router_logits(w: Workload, device, out: torch.Tensor) -> None:
    g = _gen(device, w.seed)
    x_dtype = torch.float32 if w.name == "tiny" else torch.bfloat16
    W = (torch.randn(w.hidden, w.E, generator=g, device=device) * 0.02).to(x_dtype)
    rows = 8192
    for t0 in range(0, w.T, rows):
        t1 = min(w.T, t0 + rows)
        X = torch.randn(t1 - t0, w.hidden, generator=g, device=device).to(x_dtype)
        out[t0:t1] = X.float() @ W.float()


def _collapse_logits(w: Workload, device, out: torch.Tensor) -> None:
    g = _gen(device, w.seed)
    out.copy_(torch.randn(w.T, w.E, generator=g, device=device))
    bias = torch.zeros(w.E, device=device)
    bias[0:16] = 3.0
    bias[16:48] = -3.0
    out += bias
    n_tie = max(1, (w.T * 5) // 100)
    rows = torch.randperm(w.T, generator=g, device=device)[:n_tie]
    out[rows] = torch.round(out[rows] * 2.0) / 2.0


def _long_layer(w: Workload, layer: int, device, out: torch.Tensor) -> None:
    g = _gen(device, w.seed + layer)
    bias = torch.randn(w.E, generator=g, device=device) * 0.5
    out.copy_(torch.randn(w.T, w.E, generator=g, device=device))
    out += bias


def logits(w: Workload, device="cpu", out: torch.Tensor | None = None) -> torch.Tensor:
    """Draw fp32 logits [L, T, E] (row-major, token-major) for workload ``w``."""
    if out is None:
        out = torch.empty(w.L, w.T, w.E, dtype=torch.float32, device=device)
    device = out.device
    with torch.no_grad():
        for layer in range(w.L):
            if w.hidden:
                lw = replace(w, seed=w.seed + 7919 * layer)
                _router_logits(lw, device, out[layer])
            elif w.name == "collapse":
                _collapse_logits(replace(w, seed=w.seed + 7919 * layer), device, out[layer])
            else:
                _long_layer(w, layer, device, out[layer])
    return out


def random_logits(T: int, E: int, L: int = 1, seed: int = 0, device="cpu",
                  ties: bool = False) -> torch.Tensor:
    """Plain N(0,1) logits for property sweeps; ``ties`` rounds them to multiples
    of 0.5 so that equal values are common inside a row."""
    g = _gen(device, seed)
    z = torch.randn(L, T, E, generator=g, device=device)
    if ties:
        z = torch.round(z * 2.0) / 2.0
    return z


def random_signatures(T: int, E: int, L: int = 1, seed: int = 0, density_log2: int = 1):
    """Load signatures [L, E, W] uint32 (numpy) for the pairwise-distance sweeps:
    each bit is 1 with probability 2^-density_log2 (the AND of that many
    uniform words; 4 gives k/E = 8/128), token t of an expert at bit t % 32 of
    word t // 32, and the bits past T in the last word zero."""
    W = (T + 31) // 32
    g = np.random.default_rng(seed)
    bits = np.full((L, E, W), 0xFFFFFFFF, np.uint32)
    for _ in range(max(1, density_log2)):
        bits &= g.integers(0, 1 << 32, size=(L, E, W), dtype=np.uint64).astype(np.uint32)
    if T % 32:
        bits[..., W - 1] &= np.uint32((1 << (T % 32)) - 1)
    return bits


def router_inputs(T: int, H: int, E: int = 128, L: int = 1, seed: int = 0, device="cpu"):
    """Router inputs in the c3 recipe's distribution: hidden states X [L,T,H]
    ~N(0,1) and router weights W [L,E,H] ~N(0,0.02), both rounded to bf16."""
    g = _gen(device, seed)
    X = torch.randn(L, T, H, generator=g, device=device).to(torch.bfloat16)
    W = (torch.randn(L, E, H, generator=g, device=device) * 0.02).to(torch.bfloat16)
    return X, W
