"""do_forward_backward_static: the fused path with the library's fixed scratch
array gives the results of do_forward_backward, call after call, and rejects
sizes whose workspace exceeds the array before launching anything."""
import ctypes

import pytest
import torch

from paper_2609_32398_gb300 import workloads

pytestmark = pytest.mark.gpu

LOSS_RTOL = 1e-5
GRAD_TOL = 1e-5


@pytest.fixture(scope="module")
def dl():
    import paper_2609_32398_gb300.doloss as m

    m.lib()
    return m


@pytest.mark.parametrize("T,E,k,L,gate", [(8192 + 17, 128, 8, 1, 0), (3000, 96, 3, 2, 1),
                                          (65536, 128, 8, 1, 0)])
def test_static_scratch_matches_workspace_path(dl, T, E, k, L, gate):
    z = workloads.random_logits(T, E, L=L, seed=T + E).cuda()
    ref = dl.forward_backward(z, k, gate, grad_scale=1.5)
    assert dl.device_status(ref.workspace) == 0
    flags = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    outs = [dl.Buffers(L, T, E, k, "cuda") for _ in range(2)]
    for i in range(2):  # two consecutive calls on the same scratch
        out = outs[i]
        torch.cuda.synchronize()
        free0, allocated0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
        dl.forward_backward_static(z, k, out, gate, grad_scale=1.5, status_flags=flags)
        torch.cuda.synchronize()
        if i > 0:  # the first call in the process may load the module's code
            assert torch.cuda.mem_get_info()[0] == free0, "device memory was allocated"
        assert torch.cuda.memory_allocated() == allocated0
        assert int(flags[0]) == 0
        for name in ("bits", "counts", "D", "origin_do"):
            assert torch.equal(getattr(out, name), getattr(ref, name)), name
        for l in range(L):
            assert float(out.loss[l]) == pytest.approx(float(ref.loss[l]), rel=LOSS_RTOL)
            err = (out.dlogits[l] - ref.dlogits[l]).abs().max() / ref.dlogits[l].abs().max()
            assert float(err) <= GRAD_TOL


def largest_static_T(dl, E, k, L=1):
    lo, hi = 1, 1 << 24
    while lo < hi:
        mid = (lo + hi + 1) // 2
        if dl.workspace_size(mid, E, k, L) <= (16 << 20):
            lo = mid
        else:
            hi = mid - 1
    return lo


def test_static_scratch_rejects_oversized_problems(dl):
    E, k = 128, 8
    T = largest_static_T(dl, E, k) + 1
    assert 900_000 < T < 1_000_000
    assert dl.workspace_size(T, E, k, 1) > (16 << 20)
    small = torch.zeros(64, device="cuda")
    p = ctypes.c_void_p(small.data_ptr())   # never dereferenced: the size check fails first
    st = dl.lib().do_forward_backward_static(p, T, E, k, 1, 0, 1.0, p, p, p, p, None, None, None,
                                             None)
    assert st == 6, dl.status_string(st)    # DO_ERR_WORKSPACE
