#!/usr/bin/env python
"""Benchmark of the LiLiCorr per-block draft-selection path (one process per GPU).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Default workload: single requests (batch 1, L = 16 slots, V = 151936 bf16 logits,
K = 8, d = 256, H = 4096), 1000 distinct blocks drawn from seeds 1..1000 and
resident in HBM (4.9 GB of logits, larger than L2, so no L2 flush is needed).
One step selects all 1000 blocks one after another, each a complete batch-1
call of lilicorr_select_block; the calls are captured 25 to a CUDA graph and the
graphs replayed. ``--workload serving_b32`` etc. time batched calls instead.

Prints one JSON line (rank 0): device-timed throughput (``value``), the same
metric end to end through pinned host buffers (``e2e``), the top-K kernel's
roofline measured live with CUDA events, SM clocks sampled during the timed
region, ``by_workload`` (the batched workloads, each entropy tier on its own:
call time, the top-K pass's bandwidth and the end-to-end roofline fraction), and
the CPU oracle timed on all host cores on a bounded sample (``cpu_baseline``).
``--impl reference`` times the CPU oracle itself as the reference arm.
"""
from __future__ import annotations

import os

for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")          # one BLAS thread per oracle worker process

import argparse
import json
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = "draft blocks selected/sec at 1 GB300"
UNIT = "blocks/s"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--workload", default="single_request", choices=workloads.WORKLOAD_ORDER)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--blocks", type=int, default=None, help="blocks per step (batch-1 workload)")
    p.add_argument("--batches", type=int, default=None,
                   help="distinct batches per step (batched workloads; default: up to 8, "
                        "about 1.6 GB of logits)")
    p.add_argument("--e2e-host-blocks", type=int, default=64)
    p.add_argument("--copy-streams", type=int, default=2,
                   help="streams the end-to-end host-to-device copies are spread over")
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    p.add_argument("--no-by-workload", dest="by_workload", action="store_false",
                   help="skip the batched workloads' section of the default run")
    p.add_argument("--no-extras", action="store_true",
                   help="time the selection only (no Viterbi, diagnostics, walk, vocabulary-shard "
                        "or LM-head sections): for short profiling runs")
    p.add_argument("--no-cpu-baseline", action="store_true")
    return p.parse_args()


# --------------------------------------------------------------------------- distributed
def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, x: float) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples of this GPU's SM clock and throttle reasons, every 200 ms."""
    FIELDS = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self):
        self.proc = None
        self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.uuid = str(torch.cuda.get_device_properties(torch.cuda.current_device()).uuid)
        except Exception:
            self.uuid = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait()
        self.out.flush()
        rows = []
        for line in open(self.out.name):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            if self.uuid and self.uuid not in f[0] and f[0] not in self.uuid:
                continue
            rows.append(f)
        os.unlink(self.out.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def profiled_traffic(kernel_src: str, workload: str):
    """DRAM bytes per launch of the top-K kernel from the committed ncu summary
    (profiles/topk_lse_kernel.<workload>.md), or None when that summary is missing or was
    taken on a different revision of the kernel source."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"topk_lse_kernel.{workload}.md")
    src = os.path.join(ROOT, "paper_2608_20530_gb300", "csrc", kernel_src)
    try:
        text = open(path).read()
        digest = hashlib.sha256(open(src, "rb").read()).hexdigest()
    except OSError:
        return None
    vals = {}
    for line in text.splitlines():
        if ":" in line and line.startswith("- "):
            k, v = line[2:].split(":", 1)
            vals[k.strip()] = v.strip().strip("`")
    if vals.get("kernel source sha256") != digest:
        return None
    try:
        return float(vals["dram bytes per launch"])
    except (KeyError, ValueError):
        return None


def peaks():
    try:
        return json.load(open(PEAKS_FILE)), "measured"
    except Exception:
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


# --------------------------------------------------------------------------- CPU oracle leg
def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


_ORACLE_JOB = {}      # the workload and weights the forked workers select with


def _oracle_noop(_):
    return os.getpid()


def _oracle_block(seed):
    """One whole block through the oracle, as it stands (runs in a pool worker)."""
    import oracle
    wl, W = _ORACLE_JOB["wl"], _ORACLE_JOB["W"]
    inp = workloads.sequence_inputs(wl, seed)
    emb = lambda ids: workloads.embed_rows(wl.V, wl.H, wl.dtype, ids)
    oracle.select_sequence(inp["logits"], inp["hidden"], inp["target"], emb, W, wl.K)
    return 1


class OraclePool:
    """The oracle on every host core: one worker process per core, one BLAS thread each.

    The workers are forked at construction, before this process touches the GPU (a child
    forked after CUDA initialisation can hang), after the embedding table is built, so
    they share its pages instead of each regenerating it."""

    def __init__(self, wl, W):
        import concurrent.futures as cf
        import multiprocessing as mp
        _ORACLE_JOB.update(wl=wl, W=W)
        workloads.embed_table(wl.V, wl.H, wl.dtype)        # cached in this process
        self.cores = host_cores()
        self.ex = cf.ProcessPoolExecutor(self.cores, mp_context=mp.get_context("fork"))
        list(self.ex.map(_oracle_noop, range(self.cores)))   # fork every worker now

    def run(self, seeds):
        """Select the blocks ``seeds`` on all workers; returns the wall time."""
        t0 = time.perf_counter()
        n = sum(self.ex.map(_oracle_block, seeds))
        assert n == len(seeds)
        return time.perf_counter() - t0

    def rate(self, seeds, seconds: float):
        """Blocks/s over waves of one block per worker until ``seconds`` have passed."""
        done, dt, i = 0, 0.0, 0
        while dt < seconds and i < len(seeds):
            wave = seeds[i:i + self.cores]
            dt += self.run(wave)
            done += len(wave)
            i += len(wave)
        return done / dt, done, dt

    def close(self):
        self.ex.shutdown()


def workload_config(wl, nblk: int, world: int) -> dict:
    """The ``config`` object of both arms' JSON lines (the same workload description)."""
    es = 2 if wl.dtype == "bf16" else 4
    batch1 = wl.blocks > 1
    B = 1 if batch1 else wl.B
    gb = nblk * B * wl.L * wl.V * es / 1e9
    return {"workload": wl.name, "B": B, "L": wl.L, "V": wl.V, "K": wl.K, "d": wl.d, "D": wl.D,
            "H": wl.H, "blocks_per_step": nblk,
            "l2": "inputs larger than L2 (no flush): %.2f GB of logits in %d distinct resident %s"
                  % (gb, nblk, "blocks" if batch1 else "batches"),
            "graphs": f"{GRAPH_CALLS} select_block calls per CUDA graph, replayed",
            "parallelism": f"dp{world}"}


def default_blocks(wl, args) -> int:
    if wl.blocks > 1:
        return args.blocks or wl.blocks
    es = 2 if wl.dtype == "bf16" else 4
    return args.batches or max(1, min(8, int(1.6e9 // (wl.B * wl.L * wl.V * es))))


def run_reference(args, world, rank, pool):
    """Reference arm: the CPU oracle on all host cores (one block per worker per step)."""
    if rank != 0:
        return
    wl = workloads.WORKLOADS[args.workload]
    seeds = wl.block_seeds() if wl.blocks > 1 else wl.seeds()
    C = pool.cores
    wave = lambda i: [seeds[(i * C + j) % len(seeds)] for j in range(C)]
    for i in range(args.warmup):
        pool.run(wave(i))
    dt = sum(pool.run(wave(args.warmup + i)) for i in range(args.steps))
    v = args.steps * C / dt
    sample = (f"{args.steps} steps of {C} sequences of the {wl.name} workload, one per "
              f"worker process (fp64 NumPy, 1 BLAS thread each)")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(wl, default_blocks(wl, args), world),
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": C, "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# --------------------------------------------------------------------------- GPU arm
GRAPH_CALLS = 25          # select_block calls captured per CUDA graph (batch-1 workload)
NOMINAL_HBM_GBS = 7900.0  # GB300 HBM3e, nominal


def upload(a: np.ndarray, dtype: str, dev) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(a))
    return (t.to(torch.bfloat16) if dtype == "bf16" else t).to(dev)


def gen_blocks(wl, seeds, dev, chunk=50):
    """Batch-1 blocks [n, 1, L, V] etc., generated in chunks straight into device memory."""
    n = len(seeds)
    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    logits = torch.empty((n, 1, wl.L, wl.V), dtype=tdt, device=dev)
    hidden = torch.empty((n, 1, wl.L, wl.H), dtype=tdt, device=dev)
    target = torch.empty((n, 1, wl.n_tgt, wl.H), dtype=tdt, device=dev)
    planted = np.zeros((n, 1, wl.L), np.int32)
    for i in range(0, n, chunk):
        inp = workloads.batch_inputs(wl, seeds[i:i + chunk])
        m = inp["logits"].shape[0]
        logits[i:i + m, 0] = upload(inp["logits"], wl.dtype, dev)
        hidden[i:i + m, 0] = upload(inp["hidden"], wl.dtype, dev)
        target[i:i + m, 0] = upload(inp["target"], wl.dtype, dev)
        if inp["planted"] is not None:
            planted[i:i + m, 0] = inp["planted"]
    return logits, hidden, target, planted


def gen_batches(wl, nb, tier, rank, dev):
    """nb distinct batches [nb, B, L, V] etc.; batch 0 of rank 0 is the workload's own."""
    tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    B = wl.B
    logits = torch.empty((nb, B, wl.L, wl.V), dtype=tdt, device=dev)
    hidden = torch.empty((nb, B, wl.L, wl.H), dtype=tdt, device=dev)
    target = torch.empty((nb, B, wl.n_tgt, wl.H), dtype=tdt, device=dev)
    for j in range(nb):
        inp = workloads.batch_inputs(wl, [s + rank * 100000 + j * 1000003 for s in wl.seeds(tier)],
                                     tier)
        logits[j] = upload(inp["logits"], wl.dtype, dev)
        hidden[j] = upload(inp["hidden"], wl.dtype, dev)
        target[j] = upload(inp["target"], wl.dtype, dev)
        del inp
    return logits, hidden, target


def graph_of(fns):
    """One CUDA graph replaying the calls ``fns`` in order."""
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for f in fns:
            f()
    return g


def time_replays(graphs, stream, reps: int, warm: int = 2) -> float:
    """ms per replay of the graph list, CUDA events on the launching stream."""
    for _ in range(warm):
        for g in graphs:
            g.replay()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        for g in graphs:
            g.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


def head_weight_bytes(wl) -> int:
    """Bytes of the head's weights read once per call (bf16), excluding the [V, .] table
    and the embedding projection that the folded table replaces."""
    es = 2 if wl.dtype == "bf16" else 4
    n = sum(int(np.prod(sh)) for name, sh in workloads.head_param_shapes(
        wl.H, wl.D, wl.d, wl.F, wl.n_heads, wl.L, wl.K, wl.n_layers)
        if name not in ("emb_w", "emb_b"))
    return n * es


def algorithmic(wl, B: int):
    """Algorithmic bytes and flops of one select_block call over B sequences."""
    es = 2 if wl.dtype == "bf16" else 4
    N = B * wl.L * wl.K
    D, H, L, K = wl.D, wl.H, wl.L, wl.K
    logit_bytes = B * L * wl.V * es
    nbytes = (logit_bytes + B * L * H * es + B * wl.n_tgt * H * es + N * D * 4
              + head_weight_bytes(wl) + B * L * 4)
    flops = (2 * B * L * H * D + 2 * B * H * D + 44 * N * D * D + 8 * B * (L * K) ** 2 * D
             + 2 * wl.d * B * ((L - 1) * K * K + K))
    return logit_bytes, nbytes, flops


def roofline_fracs(wl, B, us_call, us_topk, pk):
    hbm = float(pk.get("hbm_gbs", FALLBACK_HBM_GBS))
    tf = float(pk.get("bf16_tflops_sustained", pk.get("bf16_tflops", 1700.0)))
    logit_bytes, nbytes, flops = algorithmic(wl, B)
    t_bytes = nbytes / (hbm * 1e9) * 1e6
    t_flops = flops / (tf * 1e12) * 1e6
    topk_gbs = logit_bytes / (us_topk * 1e-6) / 1e9
    return {
        "topk_us": round(us_topk, 2), "topk_gbs": round(topk_gbs, 1),
        "topk_frac": round(topk_gbs / hbm, 4), "topk_frac_nominal": round(topk_gbs / NOMINAL_HBM_GBS, 4),
        "alg_bytes_per_call": nbytes, "alg_gflop_per_call": round(flops / 1e9, 2),
        "floor_us": {"hbm": round(t_bytes, 2), "tensor": round(t_flops, 2)},
        "e2e_frac": round(max(t_bytes, t_flops) / us_call, 4),
        "e2e_frac_bytes_over_hbm": round(t_bytes / us_call, 4),
    }


def bench_batched(ll, name, tier, dev, stream, E, pk, rank, copy_streams, d2h_stream, min_bytes=6e8,
                  reps=5):
    """One batched workload (one tier) through select_block: device-timed calls over
    distinct resident batches (inputs larger than L2), the top-K pass alone, and the
    same calls end to end from pinned host buffers."""
    wl = workloads.WORKLOADS[name]
    es = 2 if wl.dtype == "bf16" else 4
    B = wl.B
    nb = max(1, int(np.ceil(min_bytes / (B * wl.L * wl.V * es))))
    W = workloads.head_weights(wl)
    head = ll.Head.from_workload(wl, W, E)
    logits, hidden, target = gen_batches(wl, nb, tier, rank, dev)
    ws = head.workspace(B)
    tokens = torch.empty((nb, B, wl.L), dtype=torch.int32, device=dev)
    n0 = ll.launch_count()
    ll.select_block(head, logits[0], hidden[0], target[0], ws=ws, tokens=tokens[0])
    launches = ll.launch_count() - n0
    torch.cuda.synchronize()
    if ws.status() != 0:
        raise RuntimeError(f"{name}: device status set")
    calls = [lambda j=j: ll.select_block(head, logits[j], hidden[j], target[j], ws=ws,
                                         tokens=tokens[j]) for j in range(nb)]
    g = graph_of(calls)
    us_call = time_replays([g], stream, reps) * 1e3 / nb
    rows = B * wl.L
    tk_ws = ll.Workspace(ll.lib().lilicorr_topk_lse_workspace_bytes(rows, wl.V, wl.K))
    flat = logits.view(nb, rows, wl.V)
    ll.topk_lse(flat[0], wl.K, ws=tk_ws)
    tg = graph_of([lambda j=j: ll.topk_lse(flat[j], wl.K, ws=tk_ws) for j in range(nb)] * 2)
    us_topk = time_replays([tg], stream, reps) * 1e3 / (2 * nb)
    # end to end: each call copies its batch from pinned host memory and its tokens back,
    # the next call's copies overlapping this call's compute
    h_in = [logits.cpu().pin_memory(), hidden.cpu().pin_memory(), target.cpu().pin_memory()]
    h_tok = torch.empty((nb, B, wl.L), dtype=torch.int32).pin_memory()
    d_in = [[torch.empty_like(t[0]) for t in (logits, hidden, target)] for _ in range(2)]
    d_tok = [torch.empty((B, wl.L), dtype=torch.int32, device=dev) for _ in range(2)]
    n_e2e = max(nb, 4)
    eg = pipelined_e2e_graph(
        lambda x, tok: ll.select_block(head, x[0], x[1], x[2], ws=ws, tokens=tok),
        h_in, d_in, h_tok, d_tok, [j % nb for j in range(n_e2e)], copy_streams, d2h_stream)
    us_e2e = time_replays([eg], stream, max(2, reps // 2), warm=1) * 1e3 / n_e2e
    d_l, d_h, d_t = d_in[0]
    if ws.status() != 0 or tk_ws.status() != 0:
        raise RuntimeError(f"{name}: device status set")
    h2d = (d_l.numel() + d_h.numel() + d_t.numel()) * es
    out = {"tier": (wl.tiers[tier] if wl.tiers else None), "B": B, "K": wl.K, "D": wl.D,
           "us_per_call": round(us_call, 2), "sequences_per_s": round(B / (us_call * 1e-6), 1),
           "calls_per_s": round(1e6 / us_call, 1), "launches_per_call": launches,
           "distinct_batches": nb,
           "e2e": {"us_per_call": round(us_e2e, 2),
                   "sequences_per_s": round(B / (us_e2e * 1e-6), 1),
                   "h2d_bytes_per_call": h2d, "d2h_bytes_per_call": B * wl.L * 4}}
    out.update(roofline_fracs(wl, B, us_call, us_topk, pk))
    out["two_batches_in_flight"] = two_stream_calls(ll, wl, W, E, head, ws, logits, hidden, target,
                                                    tokens, stream, reps)
    out["walk"] = walk_latency(ll, head, logits[0], hidden[0], target[0], ws, B, stream)
    head.close()
    del logits, hidden, target, h_in, d_in, flat
    torch.cuda.empty_cache()
    return out


def two_stream_calls(ll, wl, W, E, head, ws, logits, hidden, target, tokens, stream, reps):
    """The same calls with two batches in flight: consecutive calls alternate between two
    streams, each with its own head (weights, side streams, events) and workspace, so one
    call's top-K pass and prologue overlap the other's network on the SMs it leaves idle."""
    nb = logits.shape[0]
    head2 = ll.Head.from_workload(wl, W, E)
    ws2 = head2.workspace(wl.B)
    pair = [(head, ws), (head2, ws2)]
    n = 2 * max(nb, 4)
    side = [torch.cuda.Stream(), torch.cuda.Stream()]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        cap = torch.cuda.current_stream()
        start = torch.cuda.Event()
        start.record(cap)
        for s_ in side:
            s_.wait_event(start)
        for i in range(n):
            h_, w_ = pair[i % 2]
            with torch.cuda.stream(side[i % 2]):
                ll.select_block(h_, logits[i % nb], hidden[i % nb], target[i % nb], ws=w_,
                                tokens=tokens[i % nb])
        for s_ in side:
            e = torch.cuda.Event()
            e.record(s_)
            cap.wait_event(e)
    us = time_replays([g], stream, reps) * 1e3 / n
    if ws.status() != 0 or ws2.status() != 0:
        raise RuntimeError(f"{wl.name}: device status set (two streams)")
    head2.close()
    return {"us_per_call": round(us, 2), "sequences_per_s": round(wl.B / (us * 1e-6), 1),
            "note": "consecutive calls alternate between two streams, each with its own head "
                    "and workspace (two batches resident)"}


def pipelined_e2e_graph(select, h_in, d_in, h_tok, d_tok, order, copy_streams, d2h_stream):
    """One CUDA graph of len(order) end-to-end calls: call j copies host item order[j]
    (pinned tensors h_in[k][i]) into device buffer set j % 2 on the copy streams, runs
    ``select(inputs, tokens)`` on the capturing stream once its copies have landed, and
    copies the tokens back to h_tok[i] on d2h_stream. The copies of call j + 1 run while
    call j computes (a buffer set is refilled, and a token buffer rewritten, only after the
    call two back has finished with it); the logits, the largest input, are split across
    the copy streams."""
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        s0 = torch.cuda.current_stream()
        start = torch.cuda.Event()
        start.record(s0)
        for cs in copy_streams + [d2h_stream]:
            cs.wait_event(start)
        done = []
        fetched = []
        nc = len(copy_streams)
        for j, i in enumerate(order):
            b = j % 2
            landed = []
            for k, cs in enumerate(copy_streams):
                with torch.cuda.stream(cs):
                    if j >= 2:
                        cs.wait_event(done[j - 2])
                    for t, (h, d) in enumerate(zip(h_in, d_in[b])):
                        if t == 0:          # logits: one slice of rows per copy stream
                            hv, dv = h[i].view(-1, h.shape[-1]), d.view(-1, d.shape[-1])
                            r0 = hv.shape[0] * k // nc
                            r1 = hv.shape[0] * (k + 1) // nc
                            if r1 > r0:
                                dv[r0:r1].copy_(hv[r0:r1], non_blocking=True)
                        elif k == t % nc:
                            d.copy_(h[i], non_blocking=True)
                    e = torch.cuda.Event()
                    e.record(cs)
                    landed.append(e)
            for e in landed:
                s0.wait_event(e)
            if j >= 2:
                s0.wait_event(fetched[j - 2])       # token buffer b has been read back
            select(d_in[b], d_tok[b])
            e = torch.cuda.Event()
            e.record(s0)
            done.append(e)
            with torch.cuda.stream(d2h_stream):
                d2h_stream.wait_event(e)
                h_tok[i].copy_(d_tok[b], non_blocking=True)
                f = torch.cuda.Event()
                f.record(d2h_stream)
                fetched.append(f)
        for cs in copy_streams + [d2h_stream]:
            e = torch.cuda.Event()
            e.record(cs)
            s0.wait_event(e)
    return g


def walk_latency(ll, head, logits, hidden, target, ws, B, stream, n=50):
    """Steps (3) and (4) on their own, after one selection: the pair-score kernel on the
    call's unit vectors, the greedy walk and the exact best path on its scores, each
    captured n times in a graph (us per launch, launch overhead included)."""
    ll.select_block(head, logits, hidden, target, ws=ws)
    inter = ll.select_block_intermediates(head, B, ws)
    ids, logp = inter["ids"].clone(), inter["logp"].clone()
    out, inn, anc = ll.embed_in_out(head, ids, logp, hidden, target)
    A, P = ll.pair_scores(out, inn, anc)
    ll.greedy_walk(A, P, ids)
    ll.best_path(A, P, ids)
    torch.cuda.synchronize()

    def per_call(fn):
        return round(time_replays([graph_of([fn] * n)], stream, 3, warm=1) * 1e3 / n, 2)
    return {"pair_scores_us": per_call(lambda: ll.pair_scores(out, inn, anc)),
            "greedy_walk_us": per_call(lambda: ll.greedy_walk(A, P, ids)),
            "best_path_us": per_call(lambda: ll.best_path(A, P, ids)),
            "note": f"standalone launches on one call's outputs (B = {B}), {n} per graph; in "
                    "select_block the cluster network kernel forms the pair scores and walks "
                    "in its own tail (no launch), elsewhere the pair kernel walks in its last CTA"}


BATCHED = [("serving_b32", 0), ("entropy_tiers_b64", 0), ("entropy_tiers_b64", 1),
           ("entropy_tiers_b64", 2), ("ties_b256", 0)]


def run_ours(args, world, rank, local, pool):
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_20530_gb300 as ll
    from paper_2608_20530_gb300 import shards

    dev = torch.device("cuda", torch.cuda.current_device())
    wl = workloads.WORKLOADS[args.workload]
    es = 2 if wl.dtype == "bf16" else 4
    W = workloads.head_weights(wl)
    E = workloads.embed_table(wl.V, wl.H, wl.dtype)
    head = ll.Head.from_workload(wl, W, E)
    stream = torch.cuda.current_stream()
    pk, pk_kind = peaks()

    batch1 = wl.blocks > 1
    nblk = default_blocks(wl, args)
    if batch1:
        seeds = [s + rank * nblk for s in wl.block_seeds()[:nblk]] if nblk <= wl.blocks else \
            [wl.seed_base + i + rank * nblk for i in range(nblk)]
        logits, hidden, target, planted = gen_blocks(wl, seeds, dev)
        B = 1
    else:
        # several distinct batches per step, captured together like the batch-1 blocks (a
        # serving loop does not pay one graph launch per call)
        B = wl.B
        logits, hidden, target = gen_batches(wl, nblk, 0, rank, dev)
        planted = None
    ws = head.workspace(B)
    tokens = torch.empty((nblk, B, wl.L), dtype=torch.int32, device=dev)

    # one call outside capture (configures kernels, counts launches per call)
    n0 = ll.launch_count()
    ll.select_block(head, logits[0], hidden[0], target[0], ws=ws, tokens=tokens[0])
    launches_per_call = ll.launch_count() - n0
    torch.cuda.synchronize()
    if ws.status() != 0:
        raise RuntimeError("device status set on the first call")

    G = max(1, min(GRAPH_CALLS, nblk))
    graphs = []
    for i0 in range(0, nblk, G):
        graphs.append(graph_of([lambda i=i: ll.select_block(head, logits[i], hidden[i], target[i],
                                                            ws=ws, tokens=tokens[i])
                                for i in range(i0, min(i0 + G, nblk))]))
    torch.cuda.synchronize()

    def step():
        for g in graphs:
            g.replay()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    clocks = ClockSampler()
    clocks.start()
    time.sleep(0.25)
    barrier(world)
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_stop = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for _ in range(args.steps):
        step()
    t_stop.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clk = clocks.stop()
    ms = t_start.elapsed_time(t_stop)
    ms = max_over_ranks(world, ms)
    units = nblk * B * args.steps * world
    value = units / (ms / 1e3) if not batch1 else nblk * args.steps * world / (ms / 1e3)
    ms_per_step = ms / args.steps
    if ws.status() != 0:
        raise RuntimeError("device status set during the timed region")

    # ---- end to end: pinned host inputs -> device -> select -> tokens back to pinned host;
    # each graph holds G calls, the next call's copies overlapping this call's compute
    nh = min(args.e2e_host_blocks, nblk)
    h_in = [logits[:nh].cpu().pin_memory(), hidden[:nh].cpu().pin_memory(),
            target[:nh].cpu().pin_memory()]
    h_tokens = torch.empty((nh, B, wl.L), dtype=torch.int32).pin_memory()
    d_in = [[torch.empty_like(t[0]) for t in (logits, hidden, target)] for _ in range(2)]
    d_tok = [torch.empty((B, wl.L), dtype=torch.int32, device=dev) for _ in range(2)]
    copy_streams = [torch.cuda.Stream() for _ in range(args.copy_streams)]
    d2h_stream = torch.cuda.Stream()
    sel = lambda x, tok: ll.select_block(head, x[0], x[1], x[2], ws=ws, tokens=tok)
    e2e_graphs = [pipelined_e2e_graph(sel, h_in, d_in, h_tokens, d_tok,
                                      [(k * G + j) % nh for j in range(G)], copy_streams,
                                      d2h_stream)
                  for k in range(-(-nh // G))]
    n_e2e_replays = -(-nblk // G)
    e2e_calls = n_e2e_replays * G
    d_logits, d_hidden, d_target = d_in[0]
    d_tokens = d_tok[0]

    def e2e_step():
        for r in range(n_e2e_replays):
            e2e_graphs[r % len(e2e_graphs)].replay()

    for _ in range(max(1, args.warmup)):
        e2e_step()
    torch.cuda.synchronize()
    barrier(world)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    e2e_ms = max_over_ranks(world, e0.elapsed_time(e1))
    e2e_value = e2e_calls * (1 if batch1 else B) * args.steps * world / (e2e_ms / 1e3)
    h2d = (d_logits.numel() * d_logits.element_size() + d_hidden.numel() * d_hidden.element_size()
           + d_target.numel() * d_target.element_size()) * e2e_calls
    d2h = d_tokens.numel() * 4 * e2e_calls
    del h_in, e2e_graphs

    # ---- the exact best path (App. E) in place of the greedy walk: the same calls on a
    # sample of the blocks, both walks captured alike and timed back to back
    nv = min(nblk, 100)
    walk_ms = {}
    for walk in (("greedy", "viterbi") if not args.no_extras else ()):
        gl = [graph_of([lambda i=i: ll.select_block(head, logits[i], hidden[i], target[i], ws=ws,
                                                     tokens=tokens[i], walk=walk)
                        for i in range(i0, min(i0 + G, nv))]) for i0 in range(0, nv, G)]
        walk_ms[walk] = min(time_replays(gl, stream, 1, warm=1 if k == 0 else 0)
                            for k in range(3)) / nv
    if ws.status() != 0:
        raise RuntimeError("device status set by the walk comparison")
    walk = (walk_latency(ll, head, logits[0], hidden[0], target[0], ws, B, stream)
            if not args.no_extras else None)

    # ---- diagnostics of the chosen blocks (Eq. "localar" probabilities and gaps along the
    # walk; coverage / oracle prefix / accepted prefix against the planted tokens)
    diag = None
    if planted is not None and not args.no_extras:
        nd = min(nblk, 100)
        prefix_sum = acc_sum = 0
        for i in range(nd):
            tok = ll.select_block(head, logits[i], hidden[i], target[i], ws=ws, tokens=tokens[i])
            inter = ll.select_block_intermediates(head, B, ws)
            truth = torch.from_numpy(planted[i]).to(dev)
            _, pre, acc = ll.block_acceptance(inter["ids"], tok, truth)
            prefix_sum += int(pre.sum())
            acc_sum += int(acc.sum())
        inter = ll.select_block_intermediates(head, B, ws)
        truth = torch.from_numpy(planted[nd - 1]).to(dev)

        def diag_call():
            ll.path_probs(inter["A"], inter["P"], inter["choice"])
            ll.block_acceptance(inter["ids"], tokens[nd - 1], truth)
        diag_call()
        torch.cuda.synchronize()
        dg = graph_of([diag_call] * 50)
        diag = {"truth": "planted token per slot", "blocks": nd * B,
                "mean_oracle_prefix": round(prefix_sum / (nd * B), 3),
                "mean_accepted": round(acc_sum / (nd * B), 3),
                "us_per_call": round(time_replays([dg], stream, 1, warm=1) * 1e3 / 50, 2),
                "note": "path_probs + block_acceptance on one call's outputs"}

    # ---- roofline of the top-K pass: its launches back to back in one captured graph,
    # CUDA events on the launching stream around the replay
    rows = B * wl.L
    tk_ws = ll.Workspace(ll.lib().lilicorr_topk_lse_workspace_bytes(rows, wl.V, wl.K))
    flat = logits.view(nblk, rows, wl.V)
    reps = nblk if batch1 else 50
    for i in range(min(reps, 8)):
        ll.topk_lse(flat[i % nblk], wl.K, ws=tk_ws)
    torch.cuda.synchronize()
    tg = graph_of([lambda i=i: ll.topk_lse(flat[i % nblk], wl.K, ws=tk_ws) for i in range(reps)])
    tk_ms = time_replays([tg], stream, 1, warm=1) / reps
    alg_bytes = rows * wl.V * es
    hbm = float(pk.get("hbm_gbs", FALLBACK_HBM_GBS))
    achieved = alg_bytes / (tk_ms / 1e3) / 1e9
    roofline = {"kernel": "topk_lse_kernel", "bound": "hbm", "achieved": round(achieved, 1),
                "peak": hbm, "peak_kind": pk_kind, "unit": "GB/s", "frac": round(achieved / hbm, 4),
                "frac_nominal": round(achieved / NOMINAL_HBM_GBS, 4),
                "traffic": profiled_traffic("topk_lse.cu", wl.name),
                "alg_bytes_per_launch": alg_bytes, "us_per_launch": round(tk_ms * 1e3, 3)}

    # ---- the vocabulary-sharded pass (a tensor-parallel LM head's logits), simulated on
    # this GPU: P contiguous vocabulary slices, each summarised into per-row records
    # (what one rank computes), then the merge of the gathered records
    def timed(fn, n=20):
        fn()
        torch.cuda.synchronize()
        return time_replays([graph_of([fn] * n)], stream, 1, warm=1) * 1e3 / n

    sharded = lm_head = None
    P = 4
    if args.no_extras:
        P = 0                                   # the sections below are skipped
    sl = [flat[0][:, a:b].contiguous() for a, b in shards.bounds(wl.V, P)] if P else []
    if P:
        sws = [ll.Workspace(ll.lib().lilicorr_topk_lse_partial_workspace_bytes(rows, t.shape[1], wl.K))
               for t in sl]
        recs = torch.stack([ll.topk_lse_partial(t, wl.K, a, ws=w)
                            for t, (a, _), w in zip(sl, shards.bounds(wl.V, P), sws)])
        torch.cuda.synchronize()
        part_us = timed(lambda: ll.topk_lse_partial(sl[0], wl.K, 0, ws=sws[0]))
        merge_us = timed(lambda: ll.topk_lse_merge(recs, wl.K))
        sharded = {"shards": P, "partial_us_per_rank": round(part_us, 2),
                   "merge_us": round(merge_us, 2),
                   "gather_bytes_per_rank": rows * ll.topk_partial_bytes(wl.K),
                   "note": "one rank's slice (V/%d columns of every row) and the merge of %d "
                           "ranks' records, both on this GPU; the all-gather itself is not timed"
                           % (P, P)}
        del sl, sws, recs

    # ---- the LM-head projection fused with the top-K pass (logits never written): this
    # workload's drafter hidden states against a random bf16 vocabulary projection of the
    # workload's shape, next to the unfused pair (cuBLAS bf16 product writing the logits,
    # then the top-K pass)
    if wl.dtype == "bf16" and not args.no_extras:
        gW = torch.Generator(device=dev).manual_seed(1_000_033)
        Wv = (0.02 * torch.randn((wl.V, wl.H), generator=gW, device=dev)).to(torch.bfloat16)
        hrows = hidden[0].reshape(rows, wl.H)
        lws = ll.Workspace(ll.lib().lilicorr_lm_head_topk_workspace_bytes(rows, wl.H, wl.V, wl.K))
        fused_us = timed(lambda: ll.lm_head_topk(hrows, Wv, wl.K, ws=lws), n=5)
        if ws.status() != 0 or lws.status() != 0:
            raise RuntimeError("device status set by the fused LM head")
        logits_tmp = torch.empty((rows, wl.V), dtype=torch.bfloat16, device=dev)

        def unfused():
            torch.matmul(hrows, Wv.t(), out=logits_tmp)
            ll.topk_lse(logits_tmp, wl.K, ws=tk_ws)
        unfused_us = timed(unfused, n=5)
        flops = 2.0 * rows * wl.H * wl.V
        w_bytes = wl.V * wl.H * 2
        bf16_peak = float(pk.get("bf16_tflops", 1900.0))
        lm_head = {"rows": rows, "H": wl.H, "V": wl.V, "us_per_call": round(fused_us, 2),
                   "tflops": round(flops / (fused_us * 1e-6) / 1e12, 1),
                   "tensor_frac": round(flops / (fused_us * 1e-6) / 1e12 / bf16_peak, 4),
                   "weight_gbs": round(w_bytes / (fused_us * 1e-6) / 1e9, 1),
                   "hbm_frac": round(w_bytes / (fused_us * 1e-6) / 1e9 / hbm, 4),
                   "unfused_us_per_call": round(unfused_us, 2),
                   "note": "hidden[rows, H] @ W_vocab[V, H]^T reduced to top-K + lse in one "
                           "tcgen05 pass; unfused = cuBLAS bf16 GEMM writing the logits, then "
                           "topk_lse; fractions of the measured bf16 and copy peaks"}
        del Wv, logits_tmp, lws

    l2_bytes = torch.cuda.get_device_properties(dev).L2_cache_size
    in_bytes = logits.numel() * es
    del logits, hidden, target, flat, graphs
    head.close()
    torch.cuda.empty_cache()

    # ---- the batched workloads (spec batch >= 32): each tier on its own
    by_workload = None
    if args.by_workload and batch1:
        bclk = ClockSampler()
        bclk.start()
        by_workload = {}
        for name, tier in BATCHED:
            key = name if not workloads.WORKLOADS[name].tiers else f"{name}.tau{workloads.WORKLOADS[name].tiers[tier]}"
            by_workload[key] = bench_batched(ll, name, tier, dev, stream, E, pk, rank, copy_streams,
                                             d2h_stream)
        by_workload["clocks"] = bclk.stop()
        by_workload["note"] = ("each: select_block over distinct resident batches (>= 0.6 GB of "
                               "logits, larger than L2) in one CUDA graph, CUDA events; topk_* = "
                               "the top-K pass alone over the same batches (fractions of the "
                               "measured copy bandwidth and of the nominal 7.9 TB/s); e2e_frac = "
                               "max(bytes/HBM, flops/sustained bf16) over the call time, "
                               "algorithmic bytes and flops per call; e2e = the same calls with "
                               "their inputs copied from pinned host memory and tokens back; "
                               "two_batches_in_flight = the same calls alternating between two "
                               "streams, each with its own head and workspace")

    config = workload_config(wl, nblk, world)
    if in_bytes <= l2_bytes:
        config["l2"] = ("inputs fit in L2 (%.2f GB of logits, L2 %.0f MB): a profiling size, "
                        "not a bench configuration" % (in_bytes / 1e9, l2_bytes / 1e6))
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": config,
        "us_per_block": ms_per_step * 1e3 / nblk,
        "clocks": clk,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "note": f"pinned host blocks cycled ({nh} distinct); each call's input copies "
                        f"(logits split over {args.copy_streams} copy streams) and token read-back "
                        f"(its own stream) captured with it, overlapping the neighbouring calls' "
                        f"compute"},
        "gpu_launches": launches_per_call * nblk * args.steps,
        "roofline": roofline,
        "by_workload": by_workload,
        "diagnostics": diag,
        "walk_viterbi": ({"us_per_call": round(walk_ms["viterbi"] * 1e3, 2),
                          "greedy_us_per_call": round(walk_ms["greedy"] * 1e3, 2),
                          "block_rate_cost": round(walk_ms["viterbi"] / walk_ms["greedy"] - 1, 4),
                          "sample": f"{nv} calls of this workload, best of 3"}
                         if walk_ms else None),
        "walk": walk,
        "vocab_sharded": sharded,
        "lm_head_fused": lm_head,
    }
    if pool is not None:
        seeds_cpu = wl.block_seeds() if batch1 else wl.seeds()
        v, n, dt = pool.rate(seeds_cpu, args.cpu_seconds)
        result["cpu_baseline"] = {
            "value": v, "unit": UNIT, "cores": pool.cores, "kind": "oracle",
            "sample": f"{n} sequences of the {wl.name} workload in {dt:.1f} s, one per worker "
                      f"process on {pool.cores} host cores (fp64 NumPy, 1 BLAS thread each)"}
    if rank == 0:
        print(json.dumps(result))


def main():
    args = parse_args()
    rank = int(os.environ.get("RANK", "0"))
    pool = None
    if rank == 0 and (args.impl == "reference" or not args.no_cpu_baseline):
        # forked before this process initialises CUDA
        wl = workloads.WORKLOADS[args.workload]
        pool = OraclePool(wl, workloads.head_weights(wl))
    world, rank, local = dist_setup(args)
    try:
        if args.impl == "reference":
            run_reference(args, world, rank, pool)
        else:
            run_ours(args, world, rank, local, pool)
    finally:
        if pool is not None:
            pool.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
