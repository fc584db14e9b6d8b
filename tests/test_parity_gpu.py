"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Bits, counts, the Hamming matrix and origin_do must be bit-exact; the loss
within 1e-5 relative; dlogits within 1e-4 of the oracle's largest entry
(max-abs normalised).  Inputs are the seeded workloads, drawn once and given
byte for byte to both sides.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_32398_gb300 import workloads

pytestmark = pytest.mark.gpu

LOSS_RTOL = 1e-5
GRAD_TOL = 1e-4
U32 = 2.0 ** -24   # fp32 unit roundoff


def zero_loss_tolerance(z, f, D, k, gate, d_scale=1.0):
    """For cases whose exact loss is zero by construction (uniform p, or a
    Hamming matrix of zeros), where a relative bound is meaningless: the fp32
    accumulation bound of the kernel.  Each token's sum_i p_it w_it is summed in
    fp32 over E terms, so its error is below E u sum_i |p_it w_it|; over all
    tokens that is E u M with M = sum_t sum_i p_it |dL/dp_it|."""
    T, E = z.shape
    M = float((oracle.gate(z, gate) * np.abs(oracle.dloss_dp(D, f, T, k, d_scale))).sum())
    return E * U32 * M


@pytest.fixture(scope="module")
def dl():
    import paper_2609_32398_gb300.doloss as m

    m.lib()
    return m


def gpu_run(dl, z_cpu, k, gate, grad_scale=1.0):
    z = z_cpu.to("cuda")
    out = dl.forward_backward(z, k, gate=gate, grad_scale=grad_scale)
    st = dl.device_status(out.workspace)
    assert st == 0, dl.status_string(st)
    return out


def assert_layer(out, l, zl, k, gate, grad_scale=1.0, zero_loss=False):
    """Layer l of a fused call against the oracle.  The loss must be within
    1e-5 of the oracle's, relative; only a case whose exact loss is zero by
    construction (zero_loss=True, named by the caller) is held to the fp32
    accumulation bound instead."""
    ref = oracle.forward_backward(zl, k, gate, grad_scale=grad_scale)
    bits = out.bits[l].cpu().numpy().view(np.uint32)
    assert np.array_equal(bits, ref["bits"]), "signatures"
    assert np.array_equal(out.counts[l].cpu().numpy(), ref["counts"]), "counts"
    assert np.array_equal(out.D[l].cpu().numpy(), ref["D"]), "Hamming matrix"
    assert int(out.origin_do[l]) == ref["origin_do"], "origin_do"
    loss = float(out.loss[l])
    if zero_loss:
        tol = zero_loss_tolerance(zl, oracle.select(zl, k), ref["D"], k, gate)
        assert abs(ref["loss"]) <= tol, "the case is not a zero-loss one"
    else:
        tol = LOSS_RTOL * abs(ref["loss"])
    assert abs(loss - ref["loss"]) <= tol, ("loss", loss, ref["loss"], tol)
    g = out.dlogits[l].double().cpu().numpy()
    scale = np.abs(ref["dz"]).max()
    err = np.abs(g - ref["dz"]).max() / scale if scale > 0 else np.abs(g).max()
    assert err <= GRAD_TOL, f"dlogits error {err:.3e}"


@pytest.mark.parametrize("gate", [workloads.GATE_SOFTMAX, workloads.GATE_SIGMOID_NORM])
def test_tiny_full_size(dl, gate):
    w = workloads.get("tiny")
    z = workloads.logits(w)
    out = gpu_run(dl, z, w.k, gate)
    assert_layer(out, 0, z[0].numpy(), w.k, gate)


@pytest.mark.parametrize("name,T,L", [("c2", None, None), ("c3", 8192 + 19, None),
                                      ("collapse", 16384 + 5, None), ("long", 4096 + 7, 3)])
def test_workload_recipes_reduced(dl, name, T, L):
    w = workloads.get(name, T=T, L=L)
    z = workloads.logits(w)
    out = gpu_run(dl, z, w.k, w.gate, grad_scale=1e-5 if name == "c3" else 1.0)
    for l in range(w.L):
        assert_layer(out, l, z[l].numpy(), w.k, w.gate, grad_scale=1e-5 if name == "c3" else 1.0)


def test_c3_full_size_elementwise(dl):
    """E=128, k=8, T=65536 -- the benchmark workload -- element by element."""
    w = workloads.get("c3")
    z = workloads.logits(w)
    out = gpu_run(dl, z, w.k, w.gate)
    assert_layer(out, 0, z[0].numpy(), w.k, w.gate)


@pytest.mark.parametrize(
    "T,E,k,L,gate,ties",
    [(1, 1, 1, 1, 0, False), (1, 5, 3, 2, 1, False), (31, 8, 8, 1, 0, True), (33, 33, 1, 1, 0, True),
     (100, 100, 7, 2, 1, True), (777, 64, 64, 1, 0, False), (1000, 200, 16, 1, 0, True),
     (513, 256, 8, 2, 0, True), (300, 1024, 8, 1, 0, False), (64, 37, 36, 1, 1, True),
     (2049, 96, 5, 1, 0, False)])
def test_edge_shapes(dl, T, E, k, L, gate, ties):
    z = workloads.random_logits(T, E, L=L, seed=T * 7 + E, ties=ties)
    out = gpu_run(dl, z, k, gate, grad_scale=0.5)
    for l in range(L):
        assert_layer(out, l, z[l].numpy(), k, gate, grad_scale=0.5)


def test_all_equal_logits_select_lowest_indices(dl):
    T, E, k = 96, 40, 6
    z = torch.full((1, T, E), 0.75)
    out = gpu_run(dl, z, k, 0)
    f = np.zeros((T, E), np.uint8)
    f[:, :k] = 1
    assert np.array_equal(out.bits[0].cpu().numpy().view(np.uint32), oracle.pack(f))
    assert float(out.loss[0]) == pytest.approx(0.0, abs=1e-7)    # p uniform -> L = 0
    assert_layer(out, 0, z[0].numpy(), k, 0, zero_loss=True)


def test_split_api_matches_fused_and_is_deterministic(dl):
    w = workloads.get("c2", T=5000)
    z = workloads.logits(w).cuda()
    fused = dl.forward_backward(z, w.k, w.gate)
    bits, counts = dl.signatures(z, w.k)
    D = dl.pairwise_hamming(bits, w.T)
    loss, origin, dz = dl.loss_fwd_bwd(z, bits, D, w.k, w.gate)
    again = dl.forward_backward(z, w.k, w.gate)
    torch.cuda.synchronize()
    for a, b in [(fused.bits, bits), (fused.counts, counts), (fused.D, D), (fused.loss, loss),
                 (fused.origin_do, origin), (fused.dlogits, dz), (fused.dlogits, again.dlogits),
                 (fused.loss, again.loss)]:
        assert torch.equal(a, b)


@pytest.mark.parametrize("T,E,k,L", [(97, 8, 2, 1), (500, 33, 5, 2), (4096 + 7, 128, 8, 3)])
def test_offdiag_variance_from_origin_do(dl, T, E, k, L):
    """do_offdiag_variance: Eq. origin_do with Eq. zero_sum gives the variance
    of the off-diagonal distances without reading D; numpy's variance of the
    oracle matrix's entries pins it."""
    z = workloads.random_logits(T, E, L=L, seed=T + E)
    out = gpu_run(dl, z, k, 0)
    var = dl.offdiag_variance(out.origin_do, T, E, k).cpu().numpy()
    for l in range(L):
        D = oracle.hamming(oracle.select(z[l].numpy(), k))
        off = D[~np.eye(E, dtype=bool)].astype(np.float64)
        assert var[l] == pytest.approx(off.var(), rel=1e-12, abs=1e-9)


def test_global_do_summed_matrix_with_d_scale(dl):
    """Eq. global_do: two replicas' Hamming matrices summed, scaled by 1/2, applied
    to one replica's local direction term."""
    T, E, k = 3000, 64, 4
    z = workloads.random_logits(2 * T, E, seed=99).reshape(2, T, E)
    zc = z.cuda()
    b0, _ = dl.signatures(zc[0], k)
    b1, _ = dl.signatures(zc[1], k)
    Dsum = dl.pairwise_hamming(b0, T) + dl.pairwise_hamming(b1, T)
    loss, _, dz = dl.loss_fwd_bwd(zc[0], b0, Dsum, k, 0, d_scale=0.5, grad_scale=2.0)
    torch.cuda.synchronize()
    z0 = z[0].numpy()
    f0 = oracle.select(z0, k)
    D = oracle.hamming(f0) + oracle.hamming(oracle.select(z[1].numpy(), k))
    assert np.array_equal(Dsum[0].cpu().numpy(), D)
    ref = oracle.loss(D, oracle.direction(z0, f0), T, k, d_scale=0.5)
    assert float(loss[0]) == pytest.approx(ref, rel=LOSS_RTOL)
    rdz = oracle.gate_backward(z0, oracle.dloss_dp(D, f0, T, k, d_scale=0.5), grad_scale=2.0)
    err = np.abs(dz[0].double().cpu().numpy() - rdz).max() / np.abs(rdz).max()
    assert err <= GRAD_TOL


def test_row_sum_overflow_is_reported(dl):
    T, E, k = 64, 8, 2
    z = workloads.random_logits(T, E, seed=5).cuda()
    bits, _ = dl.signatures(z, k)
    D = torch.full((1, E, E), 1 << 29, dtype=torch.int32, device="cuda")
    ws = dl.new_workspace(T, E, k)
    dl.loss_fwd_bwd(z, bits, D, k, 0, workspace=ws)
    assert dl.device_status(ws) == 5          # DO_ERR_OVERFLOW
    assert dl.device_status(ws) == 0          # cleared after reading


def test_host_entry_point_matches_device_path(dl):
    w = workloads.get("c2", T=4000)
    z = workloads.logits(w)
    hz = z.pin_memory()
    h_dz = torch.empty_like(hz).pin_memory()
    h_counts = torch.empty(1, w.E, dtype=torch.int32)
    h_D = torch.empty(1, w.E, w.E, dtype=torch.int32)
    h_loss = dl.forward_backward_host(hz, w.k, w.gate, h_dlogits=h_dz, h_counts=h_counts, h_D=h_D)
    dev = gpu_run(dl, z, w.k, w.gate)
    assert torch.equal(h_loss, dev.loss.cpu())
    assert torch.equal(h_dz, dev.dlogits.cpu())
    assert torch.equal(h_counts, dev.counts.cpu())
    assert torch.equal(h_D, dev.D.cpu())
    # loss only: the gradient is still computed (in the device buffer), not copied
    dbuf = torch.zeros(dl.host_buffer_size(w.T, w.E, w.k, 1), dtype=torch.uint8, device="cuda")
    h_loss2 = dl.forward_backward_host(hz, w.k, w.gate, device_buffer=dbuf)
    assert torch.equal(h_loss2, dev.loss.cpu())


@pytest.mark.parametrize(
    "T,E,k,L,gate,ties",
    [(1, 128, 8, 1, 0, False), (31, 32, 1, 2, 1, True), (97, 64, 2, 3, 0, True),
     (1000, 128, 4, 2, 1, False), (4096 + 33, 128, 8, 2, 0, True), (777, 32, 8, 1, 0, False),
     (3000, 64, 8, 1, 1, True), (2048, 128, 1, 1, 0, True), (3000 + 5, 256, 8, 2, 0, True),
     (777, 256, 1, 1, 1, False), (4096, 256, 4, 3, 0, True), (1000, 256, 2, 1, 0, False)])
def test_fast_path_shapes(dl, T, E, k, L, gate, ties):
    z = workloads.random_logits(T, E, L=L, seed=T + 13 * E + k, ties=ties)
    out = gpu_run(dl, z, k, gate, grad_scale=3.0)
    for l in range(L):
        assert_layer(out, l, z[l].numpy(), k, gate, grad_scale=3.0)


def test_fast_and_generic_paths_agree(dl):
    """A 4-byte-offset view of the same logits takes the generic kernels."""
    T, E, k = 3000 + 7, 128, 8
    z = workloads.random_logits(T, E, seed=77, ties=True).cuda()
    buf = torch.empty(T * E + 1, device="cuda")
    buf[1:] = z.reshape(-1)
    zoff = buf[1:].view(1, T, E)
    assert zoff.data_ptr() % 16 != 0
    fast = dl.forward_backward(z, k, 0)
    gen = dl.forward_backward(zoff, k, 0)
    torch.cuda.synchronize()
    for name in ("bits", "counts", "D", "origin_do"):
        assert torch.equal(getattr(fast, name), getattr(gen, name)), name
    assert float(fast.loss[0]) == pytest.approx(float(gen.loss[0]), rel=1e-5)
    err = (fast.dlogits - gen.dlogits).abs().max() / gen.dlogits.abs().max()
    assert float(err) <= 1e-5


@pytest.mark.parametrize("E,k,gate", [(128, 8, 0), (64, 2, 1), (32, 4, 0)])
def test_split_entry_points_fast_path(dl, E, k, gate):
    T, L = 2500, 2
    z = workloads.random_logits(T, E, L=L, seed=E + k).cuda()
    bits, counts = dl.signatures(z, k)
    D = dl.pairwise_hamming(bits, T)
    loss, origin, dz = dl.loss_fwd_bwd(z, bits, D, k, gate, grad_scale=0.25)
    torch.cuda.synchronize()
    zc = z.cpu()
    for l in range(L):
        ref = oracle.forward_backward(zc[l].numpy(), k, gate, grad_scale=0.25)
        assert np.array_equal(bits[l].cpu().numpy().view(np.uint32), ref["bits"])
        assert np.array_equal(counts[l].cpu().numpy(), ref["counts"])
        assert np.array_equal(D[l].cpu().numpy(), ref["D"])
        assert int(origin[l]) == ref["origin_do"]
        assert float(loss[l]) == pytest.approx(ref["loss"], rel=LOSS_RTOL)
        err = np.abs(dz[l].double().cpu().numpy() - ref["dz"]).max() / np.abs(ref["dz"]).max()
        assert err <= GRAD_TOL


def test_repeated_calls_reuse_workspace(dl):
    """The done counters and partial slots are reused call after call."""
    w = workloads.get("c3", T=8192)
    z = workloads.logits(w).cuda()
    out = dl.Buffers(1, w.T, w.E, w.k, "cuda")
    first = None
    for _ in range(5):
        dl.forward_backward(z, w.k, w.gate, out=out)
        torch.cuda.synchronize()
        cur = (out.loss.clone(), out.dlogits.clone(), out.D.clone())
        if first is None:
            first = cur
        assert all(torch.equal(a, b) for a, b in zip(first, cur))
    assert dl.device_status(out.workspace) == 0


@pytest.mark.parametrize("T,k,L", [(65536, 8, 1), (4096 + 33, 4, 2), (300, 1, 1), (1000, 2, 3),
                                   (66052, 8, 1), (128 * 5 + 1, 8, 2)])
def test_tcgen05_and_alu_loss_kernels_agree(dl, T, k, L):
    """The fused call's gradient pass at E = 128 (V = F D' on the tensor cores)
    against the split entry points, whose loss kernel gathers rows of D on the
    ALU, and both against the oracle at small T."""
    z = workloads.random_logits(T, 128, L=L, seed=T + k, ties=T < 2000)
    out = gpu_run(dl, z, k, workloads.GATE_SIGMOID_NORM, grad_scale=2.0)
    zc = z.cuda()
    bits, counts = dl.signatures(zc, k)
    D = dl.pairwise_hamming(bits, T)
    loss, origin, dz = dl.loss_fwd_bwd(zc, bits, D, k, workloads.GATE_SIGMOID_NORM,
                                       grad_scale=2.0)
    torch.cuda.synchronize()
    for a, b, name in ((out.bits, bits, "bits"), (out.counts, counts, "counts"), (out.D, D, "D"),
                       (out.origin_do, origin, "origin_do")):
        assert torch.equal(a, b), name
    for l in range(L):
        if T <= 8192:
            assert_layer(out, l, z[l].numpy(), k, workloads.GATE_SIGMOID_NORM, grad_scale=2.0)
        assert float(out.loss[l]) == pytest.approx(float(loss[l]), rel=1e-5)
        err = (out.dlogits[l] - dz[l]).abs().max() / dz[l].abs().max()
        assert float(err) <= 1e-5


def test_bounded_wait_reports_timeout_and_context_survives(dl):
    """A device wait that nothing completes gives up, reports DO_ERR_TIMEOUT and
    leaves the context usable (no trap, no fault, no hang)."""
    w = workloads.get("c2", T=2048)
    z = workloads.logits(w).cuda()
    out = dl.Buffers(1, w.T, w.E, w.k, "cuda")
    dl.selftest_wait_limit(out.workspace)
    assert dl.device_status(out.workspace) == 4          # DO_ERR_TIMEOUT
    assert dl.device_status(out.workspace) == 0          # cleared after reading
    dl.forward_backward(z, w.k, w.gate, out=out)
    assert dl.device_status(out.workspace) == 0
    ref = oracle.forward_backward(z[0].cpu().numpy(), w.k, w.gate)
    assert np.array_equal(out.D[0].cpu().numpy(), ref["D"])


@pytest.mark.parametrize("T,E,k,gate", [(65536, 128, 8, 0), (1000, 33, 3, 1)])
def test_async_host_entry_matches_the_synchronous_one(dl, T, E, k, gate):
    """do_forward_backward_host_async: the same loss as the synchronous host
    entry point (fused and generic paths), with the status word behind it;
    two calls in flight on two streams and two device buffers."""
    z = workloads.random_logits(T, E, seed=T + E)[0].contiguous().pin_memory()
    want = dl.forward_backward_host(z, k, gate).clone()
    bufs = [torch.zeros(dl.host_buffer_size(T, E, k, 1), dtype=torch.uint8, device="cuda")
            for _ in range(2)]
    res = [torch.zeros(8, dtype=torch.int32).pin_memory() for _ in range(2)]
    streams = [torch.cuda.Stream() for _ in range(2)]
    for i in range(4):
        dl.forward_backward_host_async(z, k, res[i % 2], bufs[i % 2], gate, stream=streams[i % 2])
    torch.cuda.synchronize()
    for r in res:
        loss, flags = dl.host_result(r, 1)
        assert flags == 0
        assert torch.equal(loss, want)


def test_autograd_wrapper_gives_the_path_gradient(dl):
    """do_loss as an autograd node: the loss of do_forward_backward, and the
    gradient times the incoming gradient (here the loss weight 0.3, and one
    weight per layer for a batched call)."""
    z = workloads.random_logits(4096 + 33, 128, L=2, seed=21).cuda()
    ref = dl.forward_backward(z, 8, 0)
    x = z.clone().requires_grad_(True)
    loss = dl.do_loss(x, 8)
    assert torch.equal(loss, ref.loss)
    (loss * torch.tensor([0.3, 2.0], device="cuda")).sum().backward()
    assert torch.allclose(x.grad[0], 0.3 * ref.dlogits[0], rtol=1e-6, atol=0)
    assert torch.allclose(x.grad[1], 2.0 * ref.dlogits[1], rtol=1e-6, atol=0)
    y = z[0].clone().requires_grad_(True)
    l1 = dl.do_loss(y, 8)
    assert l1.dim() == 0 and float(l1.detach()) == float(ref.loss[0])
    (0.3 * l1).backward()
    assert torch.allclose(y.grad, 0.3 * ref.dlogits[0], rtol=1e-6, atol=0)


def test_first_size_past_the_tensor_core_limit(dl):
    """T = 66053 at E = 128: (E - 1) T reaches 2^23, where the two-piece fp16
    split of D' stops being exact, so the fused path takes the ALU gradient
    pass; it must still match the oracle."""
    T, E, k = 66053, 128, 8
    z = workloads.random_logits(T, E, seed=66053)
    out = gpu_run(dl, z, k, 0)
    assert_layer(out, 0, z[0].numpy(), k, 0)


@pytest.mark.parametrize("T,E,k", [(32, 32, 2), (1, 8, 2)])
def test_largest_batch_of_problems(dl, T, E, k):
    """L = 65535 problems in one call (the grid's y/z limit): the fast kernels
    (E = 32) and the generic ones (E = 8), sampled layers against the oracle."""
    L = 65535
    z = workloads.random_logits(T, E, L=L, seed=L + E)
    out = gpu_run(dl, z, k, 0)
    for l in np.random.default_rng(E).choice(L, 40, replace=False).tolist() + [0, L - 1]:
        assert_layer(out, l, z[l].numpy(), k, 0)
