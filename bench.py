"""Benchmark of the DO-loss forward+backward path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

A step is one do_forward_backward call (Top-K signatures, Hamming matrix,
loss and dlogits) over the E=128, k=8, T=65536 router-logit workload (the
30BA3B-shaped layer).  Inputs are resident in HBM when the timed region
starts; consecutive steps rotate over 8 buffer sets (about 520 MiB, four times
the L2) so no step reads what the previous one left in L2.  Rank 0 prints one
JSON line.  With N > 1 (torchrun, one process per GPU) every rank runs an
independent replica: the path has no exchange step on one window, so the job
is weak-scaled replicas and the value is the tokens of all ranks over the
slowest rank's time.

--impl reference times the CPU oracle (the only reference this method has:
the paper publishes no code) on the host cores, on a bounded token sample of
the same workload per step.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import platform
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "c3"
METRIC = "DO-loss fwd+bwd routed tokens/s at E=128,k=8; % of GB300 HBM roofline"
UNIT = "tokens/s"
N_SETS = 8
NOMINAL_HBM_GBS = 8000.0  # GB300 HBM3e, nominal (context for the measured-peak fraction)
KERNELS_PER_STEP = 3  # signatures (+ co-occurrence), co-occurrence reduce (D), loss + gradient


def algorithmic_bytes(T, E, L=1):
    """Bytes the path must move once: logits read and dlogits written (4TE
    each), signatures written and read back (2 x 4EW), the Hamming matrix
    written and read (2 x 4E^2) and the counts (4E) -- per problem."""
    W = (T + 31) // 32
    return L * (8 * T * E + 8 * E * W + 8 * E * E + 4 * E)


def stage_bytes(T, E, L=1):
    W = (T + 31) // 32
    return {
        "signatures": L * (4 * T * E + 4 * E * W + 4 * E),
        "pairwise_hamming": L * (4 * E * W + 4 * E * E),
        "loss_fwd_bwd": L * (4 * T * E + 4 * E * W + 4 * E * E + 4 * T * E),
    }


def routing_bytes(T, E, k, L=1):
    """Bytes the routing outputs must move once: logits read (4TE), expert ids,
    combine weights, dispatch rows and positions written (4Tk each), counts
    and offsets (4E + 4(E+1)) -- per problem."""
    return L * (4 * T * E + 16 * T * k + 8 * E + 4)


def route_backward_bytes(T, E, k, L=1, accumulate=False):
    """Bytes of the combine weights' backward: expert ids, their gradient and
    the k chosen logits read (4Tk each); then either every dlogits entry
    written (4TE) or the k chosen entries read and written in place (8Tk)."""
    return L * (12 * T * k + (8 * T * k if accumulate else 4 * T * E))


def routed_backward_bytes(T, E, k, L=1):
    """Bytes of the backward half of the routed step: logits read and dlogits
    written (4TE each), the ids and the upstream gradient (4Tk each), the
    selected indices (Tk bytes) and the fp16 image of D' (4E^2)."""
    return L * (8 * T * E + 9 * T * k + 4 * E * E)


ROUTER_HIDDEN = 2048  # the 30BA3B router's input width (hidden size, Sec. 4.1)


def router_bytes(T, E, H, L=1):
    """Bytes of the router-fused step: X and W read (2TH + 2EH bf16), the
    logits written and read back once (8TE), dlogits written (4TE), and the
    signature, Hamming-matrix and count traffic of the DO-loss path."""
    W = (T + 31) // 32
    return L * (2 * T * H + 2 * E * H + 12 * T * E + 8 * E * W + 8 * E * E + 4 * E)


def host_cpu():
    """The host's CPU model and logical core count (context for the oracle
    baseline, which uses one core)."""
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() in ("Model name", "BIOS Model name") and ":" in line:
                model = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    return {"model": model or platform.machine(), "logical_cores": os.cpu_count()}


def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return None


# The sources each timed unit's kernels are compiled from (its launcher and
# argument checks included); a traffic record holds only while they are
# unchanged.
UNIT_SOURCES = {
    "do_forward_backward": ["sig_fast.cuh", "sig_fast.cu", "cooc_reduce.cu", "loss_mma.cu",
                            "loss.cu", "tma.cuh", "tma_host.cu", "dol_internal.cuh", "api.cu"],
    "do_routing": ["sig_fast.cuh", "route.cu", "signatures.cu", "tma.cuh", "tma_host.cu",
                   "dol_internal.cuh", "api.cu"],
    "do_route_backward": ["route_bwd.cu", "dol_internal.cuh", "api.cu"],
    "do_routed_backward": ["loss_mma.cu", "route_bwd.cu", "tma.cuh", "tma_host.cu",
                           "dol_internal.cuh", "api.cu"],
    "do_router_forward_backward": ["router.cu", "sig_fast.cuh", "cooc_reduce.cu", "loss_mma.cu",
                                   "loss.cu", "tma.cuh", "tma_host.cu", "dol_internal.cuh",
                                   "api.cu"],
}


def kernel_source_hash(unit="do_forward_backward"):
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_32398_gb300", "csrc")
    for f in sorted(UNIT_SOURCES[unit]):
        h.update(f.encode())
        h.update(open(os.path.join(csrc, f), "rb").read())
    return h.hexdigest()[:12]


def profiled_traffic(unit):
    """DRAM bytes (read + write) per launch of `unit` from the committed ncu
    summary, if it was captured on the current kernel sources (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.md")
    if not os.path.exists(path):
        return None
    src = kernel_source_hash(unit)
    for line in open(path):
        m = re.match(r"\|\s*([\w.]+)\s*\|\s*([0-9a-f]{12})\s*\|\s*(\d+)\s*\|", line)
        if m and m.group(1) == unit and m.group(2) == src:
            return int(m.group(3))
    return None


class ClockSampler:
    """nvidia-smi samples (every 200 ms) of SM clock and throttle reasons."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup(backend=None):
    """Rank, world size and local rank from the torchrun environment; joins the
    process group when world > 1 (NCCL on GPUs, gloo otherwise)."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist

        if backend is None:
            backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend)
    return rank, world, local


def reduce_max(x: float, world: int, device) -> float:
    """The largest x over all ranks (x itself on one rank)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def graph_ms_per_call(fn, reps: int) -> float:
    """Device time of one call of fn(r): reps calls captured in one CUDA graph
    (after one eager call that sets up any per-device state), the replay timed
    with CUDA events on the launching stream."""
    import torch

    fn(0)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for r in range(reps):
            fn(r)
    g.replay()
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record()
    g.replay()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / reps


def replica_throughput(units_per_rank: float, seconds: float, world: int, device) -> tuple:
    """Whole-job rate of `world` independent replicas: the units of all ranks
    over the slowest rank's time.  Returns (rate, slowest seconds)."""
    slowest = reduce_max(seconds, world, device)
    return world * units_per_rank / slowest, slowest


def barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def oracle_throughput(z_np, k, gate, budget_s, max_tokens=None):
    """Oracle forward+backward over leading token samples of z until `budget_s`
    seconds have been spent; returns (tokens/s, tokens, seconds, runs)."""
    import oracle

    T = z_np.shape[0]
    n = T if max_tokens is None else min(T, max_tokens)
    tokens, spent, runs = 0, 0.0, 0
    while runs == 0 or spent < budget_s:
        t0 = time.perf_counter()
        oracle.forward_backward(z_np[:n], k, gate)
        spent += time.perf_counter() - t0
        tokens += n
        runs += 1
    return tokens / spent, tokens, spent, runs


def run_reference(args, rank, world):
    """The reference arm: the CPU oracle as it stands, on the host cores."""
    import numpy as np

    from paper_2609_32398_gb300 import workloads

    if rank != 0:
        return
    w = workloads.get(WORKLOAD)
    import oracle

    oracle.build()
    z = np.ascontiguousarray(workloads.logits(w, "cpu")[0].numpy())
    # Calibrate a per-step token sample so that warmup + steps take about two minutes.
    t0 = time.perf_counter()
    oracle.forward_backward(z[:2048], w.k, w.gate)
    per_tok = (time.perf_counter() - t0) / 2048
    steps = args.steps + args.warmup
    sample = int(max(256, min(w.T, 120.0 / max(1, steps) / per_tok)))
    sample -= sample % 32 if sample > 32 else 0
    for i in range(args.warmup):
        oracle.forward_backward(z[:sample], w.k, w.gate)
    t0 = time.perf_counter()
    for i in range(args.steps):
        oracle.forward_backward(z[:sample], w.k, w.gate)
    dt = time.perf_counter() - t0
    value = sample * args.steps / dt
    desc = (f"leading {sample} of the {w.T} tokens of the E=128 k=8 workload per step, "
            f"single-threaded C oracle in double precision")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_dict(w),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": desc,
                         "host": host_cpu()},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# The other workloads of the path (the 4.8BA0.5B-shaped layer, the collapse
# regime and the 30BA3B-depth long window, 48 layers in one call), each timed
# through do_forward_backward with enough rotating buffer sets that the sets
# exceed L2 twice over (the larger ones exceed it on their own).
OTHER_WORKLOADS = {"c2": 500, "collapse": 200, "long": 3}  # calls timed
L2_BYTES = 129 * 2**20


def time_workload(dl, torch, workloads, name, reps, dev):
    """Microseconds per do_forward_backward call on the workload `name`."""
    w = workloads.get(name)
    per_set = 8 * w.T * w.E * w.L
    n_sets = max(1, -(-2 * L2_BYTES // per_set))
    base = workloads.logits(w, dev)
    sets = [(base if s == 0 else base + 0.0, dl.Buffers(w.L, w.T, w.E, w.k, dev))
            for s in range(n_sets)]

    def call(i):
        z, out = sets[i % n_sets]
        dl.forward_backward(z, w.k, w.gate, 1.0, out=out)

    for i in range(max(3, n_sets)):
        call(i)
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record()
    for i in range(reps):
        call(i)
    ev1.record()
    torch.cuda.synchronize()
    us = ev0.elapsed_time(ev1) * 1e3 / reps
    st = dl.device_status(sets[0][1].workspace)
    if st != 0:
        raise RuntimeError(f"device status after the {name} runs: {dl.status_string(st)}")
    del sets, base
    torch.cuda.empty_cache()
    return w, us, n_sets


def config_dict(w):
    return {"workload": f"3B-active-shaped router layer: E={w.E} k={w.k} T={w.T} L={w.L}",
            "E": w.E, "k": w.k, "T": w.T, "L": w.L, "gate": "sigmoid_norm",
            "l2": f"{N_SETS} rotating buffer sets (~{N_SETS * algorithmic_bytes(w.T, w.E) // 2**20} MiB) > L2",
            "parallelism": "replicas"}


def run_ours(args, rank, world, local):
    import numpy as np
    import torch

    import paper_2609_32398_gb300.doloss as dl
    from paper_2609_32398_gb300 import workloads

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dl.lib()
    w = workloads.get(WORKLOAD)
    T, E, k, L = w.T, w.E, w.k, w.L
    base = workloads.logits(w, dev)
    sets = []
    for s in range(N_SETS):
        z = base if s == 0 else (base + 0.0)   # same values, distinct HBM buffers
        sets.append((z, dl.Buffers(L, T, E, k, dev)))
    stream = torch.cuda.current_stream(dev)

    def step(i):
        z, out = sets[i % N_SETS]
        dl.forward_backward(z, k, w.gate, 1.0, out=out)

    warm = max(3, args.warmup)
    if args.quick:
        # profiling mode: a few plain calls of one entry point, nothing else
        # (used under ncu)
        if args.quick_path == "loss":
            call, ws = step, sets[0][1].workspace
        elif args.quick_path == "router":
            X, Wr = workloads.router_inputs(T, ROUTER_HIDDEN, E, L, seed=w.seed, device=dev)
            zr = torch.empty(L, T, E, dtype=torch.float32, device=dev)

            def call(i):
                dl.router_forward_backward(X, Wr, k, w.gate, 1.0, out=sets[0][1], logits=zr)
            ws = sets[0][1].workspace
        elif args.quick_path == "split":
            route = dl.Routing(L, T, E, k, dev)
            gq = torch.randn(L, T, k, device=dev)

            def call(i):
                dl.routed_forward(sets[i % N_SETS][0], k, w.gate, out=sets[i % N_SETS][1],
                                  route=route)
                dl.routed_backward(sets[i % N_SETS][0], route.expert_ids, gq, k, w.gate, 1.0,
                                   out=sets[i % N_SETS][1])
            ws = sets[0][1].workspace
        elif args.quick_path == "hamming":
            bits0, _ = dl.signatures(sets[0][0], k)
            Dh = torch.empty(L, E, E, dtype=torch.int32, device=dev)

            def call(i):
                dl.pairwise_hamming(bits0, T, Dh)
            ws = sets[0][1].workspace
        elif args.quick_path == "route_bwd":
            route = dl.routing(sets[0][0], k, w.gate)
            gq = torch.randn(L, T, k, device=dev)

            def call(i):
                dl.route_backward(sets[i % N_SETS][0], route.expert_ids, gq, w.gate,
                                  dlogits=sets[i % N_SETS][1].dlogits)
            ws = route.workspace
        else:
            route = dl.Routing(L, T, E, k, dev)
            if args.quick_path == "routing":
                def call(i):
                    dl.routing(sets[i % N_SETS][0], k, w.gate, out=route)
                ws = route.workspace
            else:
                def call(i):
                    dl.forward_backward_routed(sets[i % N_SETS][0], k, w.gate, 1.0,
                                               out=sets[i % N_SETS][1], route=route)
                ws = sets[0][1].workspace
        for i in range(warm + args.steps):
            call(i)
        torch.cuda.synchronize()
        st = dl.device_status(ws)
        print(json.dumps({"quick": True, "path": args.quick_path, "steps": warm + args.steps,
                          "status": st}), flush=True)
        return
    sampler = ClockSampler(local)
    sampler.start()
    for i in range(warm):
        step(i)
    torch.cuda.synchronize()
    # untimed soak so the clocks reach their loaded state and get sampled
    t_soak = time.perf_counter()
    i = 0
    while time.perf_counter() - t_soak < 1.0:
        step(i)
        i += 1
        if i % 256 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()

    # The K timed steps are captured in one CUDA graph (the calls a training
    # step makes, with the host's per-launch cost out of the device timeline)
    # and replayed once untimed before the timed replay.
    timing = "cuda_graph"
    g_steps = torch.cuda.CUDAGraph()
    try:
        with torch.cuda.graph(g_steps):
            for i in range(args.steps):
                step(i)
        g_steps.replay()
        torch.cuda.synchronize()
    except RuntimeError as ex:
        g_steps = None
        timing = f"eager loop (graph capture failed: {str(ex)[:80]})"
        torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    if g_steps is not None:
        g_steps.replay()
    else:
        for i in range(args.steps):
            step(i)
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clocks = sampler.stop()
    ms = ev0.elapsed_time(ev1)
    # the same steps as a Python loop of calls, for comparison
    ev0.record(stream)
    for i in range(args.steps):
        step(i)
    ev1.record(stream)
    torch.cuda.synchronize()
    eager_ms = ev0.elapsed_time(ev1) / args.steps
    value, seconds = replica_throughput(T * L * args.steps, ms * 1e-3, world, dev)
    ms_per_step = seconds * 1e3 / args.steps

    st = dl.device_status(sets[0][1].workspace)
    if st != 0:
        raise RuntimeError(f"device status after the timed region: {dl.status_string(st)}")

    # Per-stage durations through the split entry points: each stage's calls
    # (reps of them over the rotating sets, inputs left by the stage before)
    # captured in one CUDA graph, the replay timed with events, so that the
    # host's launch overhead between calls is not counted as device time.
    reps = max(20, min(args.steps, 2000))
    for r in range(N_SETS):
        z, out = sets[r]
        dl.signatures(z, k, out.bits, out.counts)
        dl.pairwise_hamming(out.bits, T, out.D)
    torch.cuda.synchronize()
    stage_calls = {
        "signatures": lambda r: dl.signatures(sets[r % N_SETS][0], k, sets[r % N_SETS][1].bits,
                                              sets[r % N_SETS][1].counts),
        "pairwise_hamming": lambda r: dl.pairwise_hamming(sets[r % N_SETS][1].bits, T,
                                                          sets[r % N_SETS][1].D),
        "loss_fwd_bwd": lambda r: dl.loss_fwd_bwd(
            sets[r % N_SETS][0], sets[r % N_SETS][1].bits, sets[r % N_SETS][1].D, k, w.gate,
            workspace=sets[r % N_SETS][1].workspace, dlogits=sets[r % N_SETS][1].dlogits),
    }
    stage_ms = {name: graph_ms_per_call(fn, reps) for name, fn in stage_calls.items()}
    # Routing outputs (Sec. 3.1.1): do_routing alone, and the DO-loss step that
    # also writes them from the same selection pass.
    routes = [dl.Routing(L, T, E, k, dev) for _ in range(N_SETS)]
    for r in range(2 * N_SETS):
        dl.routing(sets[r % N_SETS][0], k, w.gate, out=routes[r % N_SETS])
        dl.forward_backward_routed(sets[r % N_SETS][0], k, w.gate, 1.0, out=sets[r % N_SETS][1],
                                   route=routes[r % N_SETS])
    torch.cuda.synchronize()

    # Device time per call: reps calls in one CUDA graph (a Python loop of
    # several launches per call is limited by the host's launch rate).
    def time_calls(fn):
        return graph_ms_per_call(fn, reps)

    route_ms = time_calls(lambda r: dl.routing(sets[r % N_SETS][0], k, w.gate, out=routes[r % N_SETS]))
    routed_ms = time_calls(lambda r: dl.forward_backward_routed(
        sets[r % N_SETS][0], k, w.gate, 1.0, out=sets[r % N_SETS][1], route=routes[r % N_SETS]))
    plain_ms = time_calls(lambda r: dl.forward_backward(sets[r % N_SETS][0], k, w.gate, 1.0,
                                                        out=sets[r % N_SETS][1]))
    # The combine weights' backward to the logits: written over a dlogits
    # buffer, and added into the DO-loss step's dlogits (the training use).
    gqs = [torch.randn(L, T, k, device=dev, generator=torch.Generator(dev).manual_seed(r))
           for r in range(N_SETS)]
    rb_flags = torch.zeros(1, dtype=torch.int32, device=dev)
    rbwd_ms = time_calls(lambda r: dl.route_backward(
        sets[r % N_SETS][0], routes[r % N_SETS].expert_ids, gqs[r % N_SETS], w.gate,
        dlogits=sets[r % N_SETS][1].dlogits, status_flags=rb_flags))
    rbwd_acc_ms = time_calls(lambda r: dl.route_backward(
        sets[r % N_SETS][0], routes[r % N_SETS].expert_ids, gqs[r % N_SETS], w.gate,
        dlogits=sets[r % N_SETS][1].dlogits, accumulate=True, status_flags=rb_flags))
    if int(rb_flags[0]) != 0:
        raise RuntimeError("do_route_backward flagged an expert id out of range")
    # A training step's routed DO-loss split where the step splits: the forward
    # half (routing outputs, D) and the backward half (loss, DO gradient and
    # the combine weights' gradient in one kernel), against the one-call routed
    # step followed by the separate routing-gradient kernel.
    for r in range(2 * N_SETS):
        dl.routed_forward(sets[r % N_SETS][0], k, w.gate, out=sets[r % N_SETS][1],
                          route=routes[r % N_SETS])
        dl.routed_backward(sets[r % N_SETS][0], routes[r % N_SETS].expert_ids, gqs[r % N_SETS], k,
                           w.gate, 1.0, out=sets[r % N_SETS][1])
    torch.cuda.synchronize()
    split_fwd_ms = time_calls(lambda r: dl.routed_forward(
        sets[r % N_SETS][0], k, w.gate, out=sets[r % N_SETS][1], route=routes[r % N_SETS]))

    def split_step(r):
        dl.routed_forward(sets[r % N_SETS][0], k, w.gate, out=sets[r % N_SETS][1],
                          route=routes[r % N_SETS])
        dl.routed_backward(sets[r % N_SETS][0], routes[r % N_SETS].expert_ids, gqs[r % N_SETS], k,
                           w.gate, 1.0, out=sets[r % N_SETS][1])
    split_ms = time_calls(split_step)
    split_bwd_ms = time_calls(lambda r: dl.routed_backward(
        sets[r % N_SETS][0], routes[r % N_SETS].expert_ids, gqs[r % N_SETS], k, w.gate, 1.0,
        out=sets[r % N_SETS][1]))

    # Global-DO's per-rank step (Sec. 3.1.4, Eq. global_do) through the halves:
    # the local D (standing in for the matrix summed over the ranks, whose
    # exchange is a 64 KB all-reduce between the halves) with d_scale = 1/2,
    # which takes the ALU loss kernel; against the three split entry points.
    def global_step(r):
        dl.routed_forward(sets[r % N_SETS][0], k, w.gate, out=sets[r % N_SETS][1],
                          with_routing=False)
        dl.routed_backward(sets[r % N_SETS][0], None, None, k, w.gate, 1.0,
                           out=sets[r % N_SETS][1], d_scale=0.5)
    global_ms = time_calls(global_step)

    def one_call_step(r):
        dl.forward_backward_routed(sets[r % N_SETS][0], k, w.gate, 1.0, out=sets[r % N_SETS][1],
                                   route=routes[r % N_SETS])
        dl.route_backward(sets[r % N_SETS][0], routes[r % N_SETS].expert_ids, gqs[r % N_SETS],
                          w.gate, dlogits=sets[r % N_SETS][1].dlogits, accumulate=True)
    one_call_ms = time_calls(one_call_step)
    for r in range(N_SETS):
        st = dl.device_status(sets[r][1].workspace)
        if st != 0:
            raise RuntimeError(f"device status after the split runs: {dl.status_string(st)}")
    # Context for the fractions at this size: a plain device copy of one
    # logits-sized buffer into another, in the same rotation of input sets
    # (the measured peak comes from gigabyte-sized copies).
    copy_ms = time_calls(lambda r: sets[r % N_SETS][1].dlogits.copy_(sets[r % N_SETS][0]))
    for r in range(N_SETS):
        for ws in (routes[r].workspace, sets[r][1].workspace):
            st = dl.device_status(ws)
            if st != 0:
                raise RuntimeError(f"device status after the routing runs: {dl.status_string(st)}")
    # Consumers of the counts (App. E, Sec. 3.2): MaxVio on the device for this
    # layer and for a 48-layer stack of E = 256 experts (8 ranks each), and the
    # host REM replica allocation for 8 ranks with 2 replica slots each.
    R_ep = 8
    er1 = (torch.arange(E, device=dev, dtype=torch.int32) // (E // R_ep)).contiguous()
    c1 = sets[0][1].counts
    E48, L48 = 256, 48
    c48 = torch.randint(0, 2 * 65536 * 8 // E48, (L48, E48), device=dev, dtype=torch.int32,
                        generator=torch.Generator(dev).manual_seed(5))
    er48 = (torch.arange(E48, device=dev, dtype=torch.int32) // (E48 // R_ep)).contiguous()
    mv_out = torch.empty(L48, dtype=torch.float64, device=dev)
    lib = dl.lib()

    def maxvio_call(cnt, er, E_, L_):
        # the C entry point with preallocated outputs: launches back to back
        st_ = lib.do_maxvio(cnt.data_ptr(), er.data_ptr(), E_, R_ep, L_, None, mv_out.data_ptr(),
                            None, torch.cuda.current_stream().cuda_stream)
        if st_ != 0:
            raise RuntimeError(dl.status_string(st_))
    mv1_ms = time_calls(lambda r: maxvio_call(c1, er1, E, L))
    mv48_ms = time_calls(lambda r: maxvio_call(c48, er48, E48, L48))
    mv1, rank_loads = dl.maxvio(c1, er1, R_ep, with_rank_loads=True)
    loads_h = rank_loads[0].double().cpu().numpy()
    tokens_h = c1[0].double().cpu().numpy()
    er_h = er1.cpu().numpy()
    dl.rem_allocate(loads_h, tokens_h, er_h, 2)
    n_rem = 200
    t0 = time.perf_counter()
    for _ in range(n_rem):
        dl.rem_allocate(loads_h, tokens_h, er_h, 2)
    rem_us = (time.perf_counter() - t0) / n_rem * 1e6
    # Router-side fusion: the router's linear map on the tensor cores with the
    # signature step in its epilogue, then the rest of the path.  X (256 MiB of
    # bf16 at H = 2048) is larger than L2 by itself.  Beside it, for context:
    # cuBLAS's bf16 product (bf16 out) followed by the fused path on logits.
    X, Wr = workloads.router_inputs(T, ROUTER_HIDDEN, E, L, seed=w.seed, device=dev)
    zr = torch.empty(L, T, E, dtype=torch.float32, device=dev)
    rout = sets[0][1]
    for _ in range(3):
        dl.router_forward_backward(X, Wr, k, w.gate, 1.0, out=rout, logits=zr)
    torch.cuda.synchronize()
    router_reps = max(20, min(args.steps, 500))
    ra_, rb_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ra_.record(stream)
    for _ in range(router_reps):
        dl.router_forward_backward(X, Wr, k, w.gate, 1.0, out=rout, logits=zr)
    rb_.record(stream)
    torch.cuda.synchronize()
    router_ms = ra_.elapsed_time(rb_) / router_reps
    st = dl.device_status(rout.workspace)
    if st != 0:
        raise RuntimeError(f"device status after the router runs: {dl.status_string(st)}")
    # the router's backward (dz -> bf16, dW and dX on the tensor cores in our kernels)
    rbw = torch.empty(int(dl.lib().do_router_backward_workspace_size(T, E, ROUTER_HIDDEN, L)),
                      dtype=torch.uint8, device=dev)
    for _ in range(3):
        dl.router_backward(X, Wr, rout.dlogits, workspace=rbw)
    ra_.record(stream)
    for _ in range(router_reps):
        dl.router_backward(X, Wr, rout.dlogits, workspace=rbw)
    rb_.record(stream)
    torch.cuda.synchronize()
    router_bwd_ms = ra_.elapsed_time(rb_) / router_reps
    del rbw
    for _ in range(3):
        torch.matmul(X[0], Wr[0].T)
    ra_.record(stream)
    for _ in range(router_reps):
        torch.matmul(X[0], Wr[0].T)
    rb_.record(stream)
    torch.cuda.synchronize()
    cublas_ms = ra_.elapsed_time(rb_) / router_reps
    del X, Wr, zr

    peaks = measured_peaks()
    peak = peaks["hbm_gbs"] if peaks else 6800.0
    others = {}
    for name, reps_w in OTHER_WORKLOADS.items():
        ow, us, n_sets = time_workload(dl, torch, workloads, name, reps_w, dev)
        ab = algorithmic_bytes(ow.T, ow.E, ow.L)
        others[name] = {
            "workload": ow.describe(), "us_per_call": us,
            "tokens_per_s": ow.T * ow.L / (us * 1e-6),
            "roofline": {"bound": "hbm", "achieved": ab / (us * 1e-6) / 1e9, "peak": peak,
                         "unit": "GB/s", "frac": ab / (us * 1e-6) / 1e9 / peak,
                         "peak_source": "of measured" if peaks else "of fallback",
                         "algorithmic_bytes": ab},
            "buffer_sets": n_sets, "calls": reps_w}
    peak_src = "of measured" if peaks else "of fallback"
    # The unit of the roofline is one do_forward_backward launch sequence (three
    # dependent kernels chained by programmatic dependent launch), timed by the
    # events around the timed region on the launching stream.
    achieved = algorithmic_bytes(T, E, L) / (ms_per_step * 1e-3) / 1e9
    split_gbs = {k_: stage_bytes(T, E, L)[k_] / (v * 1e-3) / 1e9 for k_, v in stage_ms.items()}

    # End to end through the host entry point: pinned logits in, the loss out
    # (the step's result; the gradient is computed every step and stays on
    # the device, where the router's backward pass would consume it).  The
    # same call with the gradient copied out as well is reported beside it.
    e2e = None
    if rank == 0 or world > 1:
        hz = base.cpu().pin_memory()
        hdz = torch.empty_like(hz).pin_memory()
        hloss = torch.empty(L, dtype=torch.float32).pin_memory()
        dbuf = torch.zeros(dl.host_buffer_size(T, E, k, L), dtype=torch.uint8, device=dev)
        n_e2e = max(3, min(args.steps, 50))

        def timed(h_dlogits):
            for _ in range(3):
                dl.forward_backward_host(hz, k, w.gate, device_buffer=dbuf, h_dlogits=h_dlogits,
                                         h_loss=hloss)
            barrier(world)
            t0 = time.perf_counter()
            for _ in range(n_e2e):
                dl.forward_backward_host(hz, k, w.gate, device_buffer=dbuf, h_dlogits=h_dlogits,
                                         h_loss=hloss)
            return replica_throughput(T * L, (time.perf_counter() - t0) / n_e2e, world, dev)

        rate, dt = timed(None)
        rate_grad, dt_grad = timed(hdz)
        # The same work as a pipeline: do_forward_backward_host_async on two
        # device buffers and two streams, so that a step's copy in overlaps the
        # previous step's kernels; every step copies its logits in and its
        # losses and status word out.
        bufs = [dbuf, torch.zeros_like(dbuf)]
        res = [torch.zeros(L + 1, dtype=torch.int32).pin_memory() for _ in range(2)]
        strs = [torch.cuda.Stream(dev) for _ in range(2)]

        def pipelined(n):
            for i in range(n):
                dl.forward_backward_host_async(hz, k, res[i % 2], bufs[i % 2], w.gate,
                                               stream=strs[i % 2])
            torch.cuda.synchronize()

        n_pipe = max(8, min(args.steps, 200))
        pipelined(4)
        barrier(world)
        t0 = time.perf_counter()
        pipelined(n_pipe)
        rate_pipe, dt_pipe = replica_throughput(T * L, (time.perf_counter() - t0) / n_pipe, world, dev)
        for r_ in res:
            _, flags = dl.host_result(r_, L)
            if flags != 0:
                raise RuntimeError(f"device status flags {flags} in the pipelined host calls")
        e2e = {"value": rate_pipe, "unit": UNIT, "h2d_bytes_per_step": 4 * T * E * L,
               "d2h_bytes_per_step": 4 * L + 4, "ms_per_step": dt_pipe * 1e3,
               "read_back": "the losses and the device status word; dlogits are computed every "
                            "step and kept in device memory (with_dlogits_to_host copies them "
                            "out as well)",
               "api": "do_forward_backward_host_async, two device buffers and two streams",
               "synchronous_calls": {"value": rate, "d2h_bytes_per_step": 4 * L + 4,
                                     "ms_per_step": dt * 1e3,
                                     "api": "do_forward_backward_host, one call at a time"},
               "with_dlogits_to_host": {"value": rate_grad,
                                        "d2h_bytes_per_step": 4 * T * E * L + 4 * L,
                                        "ms_per_step": dt_grad * 1e3}}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        zc = np.ascontiguousarray(base[0].cpu().numpy())
        rate, ntok, spent, runs = oracle_throughput(zc, k, w.gate, budget_s=10.0)
        cpu = {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": f"{runs} oracle run(s) over all {T} tokens of the same workload "
                         f"({spent:.1f} s, single-threaded C, double precision)",
               "host": host_cpu()}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": warm, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": config_dict(w),
            "roofline": {"bound": "hbm", "kernel": "do_forward_backward",
                         "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "peak_source": peak_src,
                         "algorithmic_bytes": algorithmic_bytes(T, E, L),
                         "traffic": profiled_traffic("do_forward_backward"),
                         "traffic_over_algorithmic": (
                             profiled_traffic("do_forward_backward") / algorithmic_bytes(T, E, L)
                             if profiled_traffic("do_forward_backward") else None),
                         "frac_of_nominal_8000_GBs": achieved / NOMINAL_HBM_GBS},
            "assignments_per_s": value * k,
            "timing": timing,
            "eager_loop": {"what": "the same steps as a Python loop of do_forward_backward calls",
                           "us_per_step": eager_ms * 1e3,
                           "tokens_per_s": T * L / (eager_ms * 1e-3)},
            "split_entry_points": {"us": {k_: v * 1e3 for k_, v in stage_ms.items()},
                                   "GB/s": split_gbs},
            "size_matched_copy": {
                "what": "torch copy_ of one [L,T,E] fp32 buffer into another, same rotation",
                "bytes": 8 * T * E * L, "us": copy_ms * 1e3,
                "GB/s": 8 * T * E * L / (copy_ms * 1e-3) / 1e9},
            "routing": {
                "entry": "do_routing (selection with ids and combine weights, dispatch order)",
                "us_per_call": route_ms * 1e3, "tokens_per_s": T * L / (route_ms * 1e-3),
                "roofline": {"bound": "hbm", "kernel": "do_routing",
                             "achieved": routing_bytes(T, E, k, L) / (route_ms * 1e-3) / 1e9,
                             "peak": peak, "unit": "GB/s",
                             "frac": routing_bytes(T, E, k, L) / (route_ms * 1e-3) / 1e9 / peak,
                             "peak_source": peak_src,
                             "algorithmic_bytes": routing_bytes(T, E, k, L),
                             "traffic": profiled_traffic("do_routing")},
                "fused": {"entry": "do_forward_backward_routed",
                          "us_per_call": routed_ms * 1e3,
                          "us_per_call_without_routing": plain_ms * 1e3},
                "backward": {
                    "entry": "do_route_backward (combine weights' gradient to the logits)",
                    "us_per_call": rbwd_ms * 1e3,
                    "us_per_call_accumulate": rbwd_acc_ms * 1e3,
                    "roofline": {"bound": "hbm", "kernel": "route_backward_kernel",
                                 "achieved": route_backward_bytes(T, E, k, L) / (rbwd_ms * 1e-3) / 1e9,
                                 "peak": peak, "unit": "GB/s",
                                 "frac": route_backward_bytes(T, E, k, L) / (rbwd_ms * 1e-3) / 1e9
                                 / peak,
                                 "peak_source": peak_src,
                                 "algorithmic_bytes": route_backward_bytes(T, E, k, L),
                                 "algorithmic_bytes_accumulate":
                                     route_backward_bytes(T, E, k, L, accumulate=True),
                                 "traffic": profiled_traffic("do_route_backward")}},
                "global_do_step": {
                    "entries": "do_routed_forward (no routing outputs) then do_routed_backward "
                               "with a summed D and d_scale = 1/2",
                    "us_per_step": global_ms * 1e3,
                    "vs": "do_signatures + do_pairwise_hamming + do_loss_fwd_bwd",
                    "vs_us_per_step": sum(stage_ms.values()) * 1e3},
                "training_split": {
                    "entries": "do_routed_forward then do_routed_backward (routing gradient in "
                               "the loss kernel's epilogue)",
                    "us_per_step": split_ms * 1e3, "forward_us": split_fwd_ms * 1e3,
                    "backward_us": split_bwd_ms * 1e3,
                    "backward_roofline": {
                        "bound": "hbm", "kernel": "loss_mma_kernel<8, true>",
                        "achieved": routed_backward_bytes(T, E, k, L) / (split_bwd_ms * 1e-3) / 1e9,
                        "peak": peak, "unit": "GB/s",
                        "frac": routed_backward_bytes(T, E, k, L) / (split_bwd_ms * 1e-3) / 1e9
                        / peak, "peak_source": peak_src,
                        "algorithmic_bytes": routed_backward_bytes(T, E, k, L),
                        "traffic": profiled_traffic("do_routed_backward")},
                    "vs": "do_forward_backward_routed then do_route_backward (accumulate)",
                    "vs_us_per_step": one_call_ms * 1e3},
                "reps": reps},
            "counts_consumers": {
                "maxvio_us_per_call": {"E128_L1_R8": mv1_ms * 1e3, "E256_L48_R8": mv48_ms * 1e3},
                "maxvio_c3": float(mv1[0]),
                "rem_allocate_host_us_per_call": {"E128_R8_D2": rem_us},
                "bound": "launch latency (a few KB per call)"},
            "router_fused": {
                "entry": "do_router_forward_backward (logits = X W^T on tcgen05 with the signature "
                         "step in the GEMM epilogue, then the D reduction and the loss)",
                "hidden": ROUTER_HIDDEN, "x_dtype": "bf16",
                "us_per_call": router_ms * 1e3, "tokens_per_s": T * L / (router_ms * 1e-3),
                "roofline": {"bound": "hbm", "kernel": "do_router_forward_backward",
                             "achieved": router_bytes(T, E, ROUTER_HIDDEN, L) / (router_ms * 1e-3) / 1e9,
                             "peak": peak, "unit": "GB/s",
                             "frac": router_bytes(T, E, ROUTER_HIDDEN, L) / (router_ms * 1e-3) / 1e9 / peak,
                             "peak_source": peak_src,
                             "algorithmic_bytes": router_bytes(T, E, ROUTER_HIDDEN, L),
                             "traffic": profiled_traffic("do_router_forward_backward")},
                "context_unfused_us": {"cublas_bf16_matmul": cublas_ms * 1e3,
                                       "do_forward_backward": plain_ms * 1e3},
                "backward": {"entry": "do_router_backward (dz rounded to bf16; dW fp32 and dX "
                                      "bf16 by tcgen05 kernels)",
                             "us_per_call": router_bwd_ms * 1e3,
                             "bytes": 2 * T * L * ROUTER_HIDDEN * 2 + 4 * T * E * L + 4 * T * E * L
                             + 2 * E * ROUTER_HIDDEN * L + 4 * E * ROUTER_HIDDEN * L},
                "reps": router_reps},
            "other_workloads": others,
            "clocks": clocks, "e2e": e2e, "gpu_launches": KERNELS_PER_STEP * args.steps,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)


def main():
    if len(sys.argv) == 3 and sys.argv[1] == "--source-hash":
        print(kernel_source_hash(sys.argv[2]))
        return
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--quick", action="store_true",
                    help="run warmup+steps plain steps and exit (for profilers)")
    ap.add_argument("--quick-path", choices=["loss", "routing", "routed", "router", "route_bwd",
                                             "split", "hamming"],
                    default="loss",
                    help="entry point of --quick: do_forward_backward, do_routing, "
                         "do_forward_backward_routed, do_router_forward_backward, "
                         "do_route_backward, do_routed_forward + do_routed_backward or "
                         "do_pairwise_hamming")
    args = ap.parse_args()
    if args.impl == "reference":
        rank = int(os.environ.get("RANK", "0"))
        world = int(os.environ.get("WORLD_SIZE", str(args.gpus)))
        run_reference(args, rank, world)
        return
    rank, world, local = dist_setup()
    try:
        run_ours(args, rank, world, local)
    finally:
        if world > 1:
            import torch.distributed as dist

            dist.destroy_process_group()


if __name__ == "__main__":
    main()
