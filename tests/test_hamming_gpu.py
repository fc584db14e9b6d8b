"""The split Hamming entry points, do_pairwise_hamming and
do_pairwise_hamming_accumulate (Sec. 3.1.3, Eq. gij_cij), against the oracle's
XOR-popcount matrix, bit for bit.

The shapes cover a signature shorter than one 128-word stage, a ragged last
stage, W not a multiple of 4 (4-byte copies), a signature array that is not
16-byte aligned, expert counts that cut the 16-expert blocks, every split of
the words over a cluster (1 to 8 CTAs, with a ragged last range), the c2, c3
and long-window layer sizes, many layers, and E = 1024.  D starts filled with
a sentinel, so every entry must be written (once per unordered pair, zero on
the diagonal); with accumulate the result adds to what D held."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dl():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    import paper_2609_32398_gb300.doloss as dl

    dl.lib()
    return dl


def check(dl, bits_np, T, offset=False, accumulate=False):
    L, E, W = bits_np.shape
    b = torch.from_numpy(bits_np.view(np.int32)).cuda()
    if offset:  # the same words one 4-byte slot into a larger buffer
        buf = torch.zeros(b.numel() + 1, dtype=torch.int32, device="cuda")
        buf[1:] = b.reshape(-1)
        b = buf[1:].view(L, E, W)
        assert b.data_ptr() % 16 != 0
    g = np.random.default_rng(T + E)
    base = g.integers(0, 1 << 20, size=(L, E, E)).astype(np.int32)
    D = torch.from_numpy(base).cuda() if accumulate else \
        torch.full((L, E, E), -7, dtype=torch.int32, device="cuda")
    dl.pairwise_hamming(b, T, D=D, accumulate=accumulate)
    got = D.cpu().numpy()
    for l in range(L):
        ref = oracle.hamming_bits(bits_np[l], T)
        if accumulate:
            ref = ref + base[l]  # the diagonal keeps what it held
        assert np.array_equal(got[l], ref), f"layer {l}"


@pytest.mark.parametrize(
    "T,E,L,density",
    [(1, 1, 1, 1), (31, 5, 2, 1), (32 * 129, 3, 1, 1), (4096 + 7, 37, 3, 2), (16384, 128, 1, 4),
     (16384, 64, 1, 4), (65536, 128, 1, 4), (65536 * 4 + 32, 16, 1, 1), (65536 * 4 + 64, 17, 2, 2),
     (300, 1024, 1, 4), (2049, 96, 5, 3), (1 << 20, 256, 1, 5), (5000, 200, 2, 1),
     (128 * 64, 48, 65, 2), (65536, 64, 8, 4), (1 << 17, 128, 9, 4)])
def test_matches_oracle(dl, T, E, L, density):
    bits = workloads.random_signatures(T, E, L, seed=T * 3 + E, density_log2=density)
    check(dl, bits, T)


@pytest.mark.parametrize("T,E,L", [(5000, 200, 2), (4096 * 3, 128, 1), (33, 16, 3)])
def test_unaligned_signatures(dl, T, E, L):
    bits = workloads.random_signatures(T, E, L, seed=T + 5, density_log2=2)
    check(dl, bits, T, offset=True)


@pytest.mark.parametrize("T,E,L", [(65536, 128, 1), (3000, 64, 2), (100, 7, 1), (1 << 18, 32, 1)])
def test_accumulate_adds_to_the_running_sum(dl, T, E, L):
    bits = workloads.random_signatures(T, E, L, seed=T + 11, density_log2=3)
    check(dl, bits, T, accumulate=True)


def test_signatures_of_the_c3_workload(dl):
    """The matrix of the c3 selection, from the signatures kernel's own bits."""
    w = workloads.get("c3")
    z = workloads.logits(w).cuda()
    bits, _ = dl.signatures(z, w.k)
    D = dl.pairwise_hamming(bits, w.T)
    torch.cuda.synchronize()
    ref = oracle.hamming_bits(bits[0].cpu().numpy().view(np.uint32), w.T)
    assert np.array_equal(D[0].cpu().numpy(), ref)
    # Eq. zero_sum: every token adds k (E - k) to the upper triangle
    assert int(np.triu(ref.astype(np.int64), 1).sum()) == w.T * w.k * (w.E - w.k)
