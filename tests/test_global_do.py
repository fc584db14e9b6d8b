"""Global-DO (Sec. 3.1.4, Eq. global_do): the Hamming matrices of the data-parallel
ranks are summed and scaled by 1/ranks before the loss.

CPU: two gloo ranks each hold half of the tokens; their oracle matrices, summed
by the binding's collective helper, equal the oracle matrix of all the tokens
(distances add over token shards) with d_scale = 1/2, and each rank's loss with
the summed matrix matches the oracle's loss of its shard under that matrix.
GPU: with one rank the helper reduces to the local path."""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world)})
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import oracle
    from paper_2609_32398_gb300 import doloss, workloads

    dist.init_process_group("gloo")
    w = workloads.get("c2", T=2048)
    z = workloads.logits(w)[0].numpy()
    shard = z[rank * 1024:(rank + 1) * 1024]
    f = oracle.select(shard, w.k)
    D_local = torch.from_numpy(oracle.hamming(f).astype(np.int32))
    D_sum, d_scale = doloss.all_reduce_distances(D_local.clone())
    C = oracle.direction(shard, f, w.gate)
    loss = oracle.loss(D_sum.numpy(), C, shard.shape[0], w.k, d_scale)
    out[rank] = (D_sum.numpy(), d_scale, loss)
    dist.destroy_process_group()


def test_two_ranks_sum_distances_on_cpu():
    import oracle
    from paper_2609_32398_gb300 import workloads

    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    out = manager.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
    assert all(p.exitcode == 0 for p in procs)
    w = workloads.get("c2", T=2048)
    z = workloads.logits(w)[0].numpy()
    D_all = oracle.hamming(oracle.select(z, w.k))
    for r in range(2):
        D_sum, d_scale, loss = out[r]
        assert np.array_equal(D_sum, D_all)
        assert d_scale == 0.5
        shard = z[r * 1024:(r + 1) * 1024]
        f = oracle.select(shard, w.k)
        ref = oracle.loss(D_all, oracle.direction(shard, f, w.gate), 1024, w.k, 0.5)
        assert loss == pytest.approx(ref, rel=1e-12)


@pytest.mark.gpu
def test_single_rank_global_do_equals_local_path():
    import paper_2609_32398_gb300.doloss as dl
    from paper_2609_32398_gb300 import workloads

    w = workloads.get("c2", T=4096)
    z = workloads.logits(w).cuda()
    loss, dz, D, counts = dl.global_forward_backward(z, w.k, w.gate, grad_scale=2.0)
    ref = dl.forward_backward(z, w.k, w.gate, grad_scale=2.0)
    torch.cuda.synchronize()
    assert torch.equal(D, ref.D) and torch.equal(counts, ref.counts)
    assert float(loss[0]) == pytest.approx(float(ref.loss[0]), rel=1e-5)
    err = (dz - ref.dlogits).abs().max() / ref.dlogits.abs().max()
    assert float(err) <= 1e-5


@pytest.mark.gpu
def test_accumulation_window_matches_oracle():
    """A window of three micro-batches (ragged sizes): D is the sum of their
    Hamming matrices, and each micro-batch's loss and gradient are Eq. global_do
    with that matrix, d_scale = 1/3 and m its own token count."""
    import oracle
    import paper_2609_32398_gb300.doloss as dl
    from paper_2609_32398_gb300 import workloads

    k, E = 8, 128
    zs = [workloads.random_logits(T, E, seed=T) for T in (4096, 1000 + 33, 2048)]
    losses, grads, D = dl.window_forward_backward([z.cuda() for z in zs], k)
    D_ref = sum(oracle.hamming(oracle.select(z[0].numpy(), k)) for z in zs)
    assert np.array_equal(D[0].cpu().numpy(), D_ref)
    for z, loss, dz in zip(zs, losses, grads):
        zl = z[0].numpy()
        f = oracle.select(zl, k)
        T = zl.shape[0]
        want = oracle.loss(D_ref, oracle.direction(zl, f), T, k, d_scale=1.0 / 3)
        assert abs(float(loss[0]) - want) <= 1e-5 * abs(want)
        g = oracle.gate_backward(zl, oracle.dloss_dp(D_ref, f, T, k, d_scale=1.0 / 3))
        assert np.abs(dz[0].double().cpu().numpy() - g).max() <= 1e-4 * np.abs(g).max()


@pytest.mark.gpu
@pytest.mark.parametrize("E,L,offset", [(128, 1, 0), (33, 3, 1), (256, 2, 0)])
def test_accumulate_distances_is_the_integer_sum(E, L, offset):
    """do_accumulate_distances adds [L,E,E] int32 matrices exactly, on the
    16-byte path and (one-element offset) the scalar one."""
    import paper_2609_32398_gb300.doloss as dl

    g = torch.Generator().manual_seed(E + L)
    a = torch.randint(0, 1 << 20, (L * E * E + offset,), generator=g, dtype=torch.int32).cuda()
    b = torch.randint(0, 1 << 20, (L * E * E + offset,), generator=g, dtype=torch.int32).cuda()
    want = (a.long() + b.long())[offset:]
    st = dl.lib().do_accumulate_distances(a[offset:].data_ptr(), E, L, b[offset:].data_ptr(),
                                          torch.cuda.current_stream().cuda_stream)
    assert st == 0
    torch.cuda.synchronize()
    assert torch.equal(b[offset:].long(), want)


def _gpu_rank_main(rank, world, port, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world)})
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    from paper_2609_32398_gb300 import doloss, workloads

    torch.cuda.set_device(0)
    dist.init_process_group("gloo")
    w = workloads.get("c3", T=8192)
    z = workloads.logits(w)[0]
    shard = z[rank * 4096:(rank + 1) * 4096].contiguous().cuda()
    loss, dz, D, counts = doloss.global_forward_backward(shard, w.k, w.gate, grad_scale=1.0)
    torch.cuda.synchronize()
    out[rank] = (float(loss[0]), dz[0].cpu().numpy(), D[0].cpu().numpy(), counts[0].cpu().numpy())
    dist.destroy_process_group()


@pytest.mark.gpu
def test_two_gloo_ranks_on_the_gpu_path():
    """Global-DO through the GPU halves with a real process group: two ranks
    (processes on one GPU; the only exchange is gloo's host all-reduce of D,
    none of the kernels waits on another rank) each hold half of the c3
    tokens.  The summed D is the oracle's matrix of all tokens, and each
    rank's loss and gradient are the oracle's for its shard with d_scale = 1/2
    (the ALU loss kernel)."""
    import oracle
    from paper_2609_32398_gb300 import workloads

    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    out = manager.dict()
    port = _free_port()
    procs = [ctx.Process(target=_gpu_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
    assert all(p.exitcode == 0 for p in procs)
    w = workloads.get("c3", T=8192)
    z = workloads.logits(w)[0].numpy()
    D_all = oracle.hamming(oracle.select(z, w.k))
    for r in range(2):
        loss, dz, D, counts = out[r]
        assert np.array_equal(D, D_all)
        shard = z[r * 4096:(r + 1) * 4096]
        f = oracle.select(shard, w.k)
        assert np.array_equal(counts, oracle.counts(f))
        want = oracle.loss(D_all, oracle.direction(shard, f, w.gate), 4096, w.k, 0.5)
        assert abs(loss - want) <= 1e-5 * abs(want)
        g = oracle.gate_backward(shard, oracle.dloss_dp(D_all, f, 4096, w.k, d_scale=0.5), w.gate)
        assert np.abs(dz - g).max() <= 1e-4 * np.abs(g).max()


@pytest.mark.gpu
def test_window_of_one_micro_batch_is_the_local_step():
    """A window of one micro-batch on one rank has d_scale = 1: the backward
    half takes the tensor-core kernel and returns do_forward_backward's loss
    and dlogits bit for bit."""
    import paper_2609_32398_gb300.doloss as dl
    from paper_2609_32398_gb300 import workloads

    w = workloads.get("c3", T=4096 + 17)
    z = workloads.logits(w).cuda()
    losses, grads, D = dl.window_forward_backward([z], w.k, w.gate, grad_scale=1.5)
    ref = dl.forward_backward(z, w.k, w.gate, grad_scale=1.5)
    torch.cuda.synchronize()
    assert torch.equal(D, ref.D)
    assert torch.equal(losses[0], ref.loss) and torch.equal(grads[0], ref.dlogits)


@pytest.mark.gpu
@pytest.mark.parametrize("with_route", [False, True])
def test_summed_matrix_beyond_the_fp16_image_takes_the_alu_kernel(with_route):
    """Eq. global_do with a given matrix at E = 128, two problems in one call:
    problem 0's matrix (three local matrices' sum) fits the two fp16 pieces of
    the tensor-core kernel's image of D', problem 1's (a 256-fold sum, row sums
    above 2^23) does not and goes to the ALU kernel.  Both problems' loss and
    gradient equal the oracle's for their matrix, with d_scale = 1/3, with and
    without the combine weights' gradient added in the same call."""
    import oracle
    import paper_2609_32398_gb300.doloss as dl
    from paper_2609_32398_gb300 import workloads

    k, E, T, L = 8, 128, 4096 + 64, 2
    z = workloads.random_logits(T, E, L=L, seed=321)
    zc = z.cuda()
    out, route = dl.routed_forward(zc, k, 0, with_routing=with_route)
    torch.cuda.synchronize()
    D_loc = [oracle.hamming(oracle.select(z[l].numpy(), k)) for l in range(L)]
    mult = (3, 256)
    D_sum = np.stack([D_loc[l].astype(np.int64) * mult[l] for l in range(L)])
    assert D_sum[1].sum(axis=1).max() >= 1 << 23 > D_sum[0].sum(axis=1).max()
    Dg = torch.from_numpy(D_sum.astype(np.int32)).cuda()
    gq = None
    if with_route:
        gq = torch.randn(L, T, k, generator=torch.Generator().manual_seed(9)).cuda()
    dl.routed_backward(zc, route.expert_ids if with_route else None, gq, k, 0, 1.5, out=out, D=Dg,
                       d_scale=1.0 / 3)
    torch.cuda.synchronize()
    for l in range(L):
        zl = z[l].numpy()
        f = oracle.select(zl, k)
        want = oracle.loss(D_sum[l], oracle.direction(zl, f), T, k, d_scale=1.0 / 3)
        assert abs(float(out.loss[l]) - want) <= 1e-5 * abs(want), l
        g = oracle.gate_backward(zl, oracle.dloss_dp(D_sum[l], f, T, k, d_scale=1.0 / 3),
                                 grad_scale=1.5)
        if with_route:
            g = g + oracle.route_backward(zl, route.expert_ids[l].cpu().numpy(),
                                          gq[l].double().cpu().numpy())
        err = np.abs(out.dlogits[l].double().cpu().numpy() - g).max() / np.abs(g).max()
        assert err <= 1e-4, (l, err)
    assert dl.device_status(out.workspace) == 0
