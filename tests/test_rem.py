"""The library's counts consumers against the oracle: do_rem_allocate (a host
function, so it runs without a GPU) and do_maxvio (a device kernel).

Both evaluate the same double-precision formulas in the same order as the
oracle, so placements, loads and MaxVio values must agree exactly."""
import json
import os

import numpy as np
import pytest
import torch

from oracle import rem

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def dl():
    from paper_2609_32398_gb300 import build, doloss

    build.build()
    return doloss


def test_rem_allocate_worked_examples(dl):
    for ex in json.load(open(os.path.join(GOLDEN, "rem_worked_examples.json")))["examples"]:
        A, L = dl.rem_allocate(ex["loads"], ex["expert_tokens"], ex["expert_rank"], ex["D"])
        assert [list(a) for a in A] == ex["placements"]
        assert L.tolist() == ex["loads_after"]


@pytest.mark.parametrize("seed", range(12))
def test_rem_allocate_matches_oracle(dl, seed):
    rng = np.random.default_rng(100 + seed)
    R, E, D = int(rng.integers(2, 17)), int(rng.integers(2, 130)), int(rng.integers(0, 4))
    home = rng.integers(0, R, E)
    tokens = rng.gamma(0.6, 800.0, E)
    if seed % 2 == 0:
        tokens = tokens.round()                             # token counts
    loads = rem.rank_loads(tokens, home, R) if seed % 3 else rng.uniform(0, 5000, R)
    A_ref, L_ref = rem.rem_allocate(loads, tokens, home, D)
    A, L = dl.rem_allocate(loads, tokens, home, D)
    assert A == [(int(e), int(s), int(r), float(d)) for e, s, r, d in A_ref]
    assert L.tolist() == L_ref


def test_rem_allocate_rejects_bad_input(dl):
    with pytest.raises(dl.DoLossError):
        dl.rem_allocate([1.0, 2.0], [1.0, 2.0], [0, 2], 1)    # rank outside [0, R)
    with pytest.raises(dl.DoLossError):
        dl.rem_allocate([1.0, 2.0], [1.0, 2.0], [0, 1], -1)   # negative slot count
    A, L = dl.rem_allocate([5.0, 1.0], [5.0, 1.0], [0, 1], 0)  # no slots: nothing placed
    assert A == [] and L.tolist() == [5.0, 1.0]


@pytest.mark.gpu
def test_maxvio_matches_oracle(dl):
    from paper_2609_32398_gb300 import workloads

    rng = np.random.default_rng(7)
    w = workloads.get("c3", T=16384)
    z = workloads.logits(w, "cuda")
    out = dl.forward_backward(z, w.k, w.gate)
    counts = torch.cat([out.counts, torch.from_numpy(rng.integers(0, 5000, (3, w.E))).int().cuda(),
                        torch.zeros(1, w.E, dtype=torch.int32, device="cuda")])
    for R in (1, 8, 13, 128, 4096):
        home = torch.from_numpy(rng.integers(0, R, w.E).astype(np.int32)).cuda()
        mv, loads = dl.maxvio(counts, home, R, with_rank_loads=True)
        c = counts.cpu().numpy()
        h = home.cpu().numpy()
        for l in range(c.shape[0]):
            ref_loads = rem.rank_loads(c[l], h, R)
            assert loads[l].cpu().tolist() == ref_loads
            assert float(mv[l]) == rem.maxvio(ref_loads)
    assert float(mv[-1]) == 0.0                              # no tokens


@pytest.mark.gpu
def test_maxvio_flags_an_expert_rank_out_of_range(dl):
    counts = torch.ones(2, 16, dtype=torch.int32, device="cuda")
    home = torch.arange(16, dtype=torch.int32, device="cuda") % 4
    home[5] = 9
    flags = torch.zeros(1, dtype=torch.int32, device="cuda")
    mv = dl.maxvio(counts, home, 4, status_flags=flags)
    assert int(flags) == 4
    # the expert on the unknown rank is left out: rank loads 4, 3, 4, 4
    assert float(mv[0]) == rem.maxvio([4, 3, 4, 4])
