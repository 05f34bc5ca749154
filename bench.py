#!/usr/bin/env python
"""Benchmark of the LiLiCorr per-block draft-selection path (one process per GPU).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Default workload: single requests (batch 1, L = 16 slots, V = 151936 bf16 logits,
K = 8, d = 256, H = 4096), 1000 distinct blocks drawn from seeds 1..1000 and
resident in HBM (4.9 GB of logits, larger than L2, so no L2 flush is needed).
One step selects all 1000 blocks one after another, each a complete batch-1
call of lilicorr_select_block; the calls are captured 25 to a CUDA graph and the
graphs replayed. Batched
workloads (``--workload serving_b32`` etc.) time one call over the batch per step.

Prints one JSON line (rank 0): device-timed throughput (``value``), the same
metric end to end through pinned host buffers (``e2e``), the top-K kernel's
roofline measured live with CUDA events, SM clocks sampled during the timed
region, and the CPU oracle timed on a bounded sample (``cpu_baseline``).
``--impl reference`` times the CPU oracle itself as the reference arm.
"""
from __future__ import annotations

import os

for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")          # the oracle baseline runs on one core

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
    p.add_argument("--calls-per-graph", type=int, default=25,
                   help="batch-1 select_block calls captured in one CUDA graph")
    p.add_argument("--cpu-seconds", type=float, default=15.0)
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
def oracle_blocks_per_s(wl, W, seeds, seconds: float):
    """The oracle, as it stands, selecting whole blocks one after another on the host."""
    import oracle
    emb = lambda ids: workloads.embed_rows(wl.V, wl.H, wl.dtype, ids)
    done, t0 = 0, time.perf_counter()
    for seed in seeds:
        inp = workloads.sequence_inputs(wl, seed)
        oracle.select_sequence(inp["logits"], inp["hidden"], inp["target"], emb, W, wl.K)
        done += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    return done / dt, done, dt


def run_reference(args, world, rank):
    """Reference arm: the CPU oracle on the host cores, one block per step."""
    if rank != 0:
        return
    wl = workloads.WORKLOADS[args.workload]
    W = workloads.head_weights(wl)
    seeds = wl.block_seeds() if wl.blocks > 1 else wl.seeds()
    workloads.embed_table(wl.V, wl.H, wl.dtype)          # generate once, outside the timing
    for i in range(args.warmup):
        oracle_blocks_per_s(wl, W, [seeds[i % len(seeds)]], 0.0)
    t0 = time.perf_counter()
    for i in range(args.steps):
        oracle_blocks_per_s(wl, W, [seeds[(args.warmup + i) % len(seeds)]], 0.0)
    dt = time.perf_counter() - t0
    v = args.steps / dt
    sample = f"{args.steps} sequences of the {wl.name} workload, one per step"
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": wl.name, "B": 1, "L": wl.L, "V": wl.V,
                                        "K": wl.K, "d": wl.d, "H": wl.H},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# --------------------------------------------------------------------------- GPU arm
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


def run_ours(args, world, rank, local):
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

    batch1 = wl.blocks > 1
    if batch1:
        nblk = args.blocks or wl.blocks
        seeds = [s + rank * nblk for s in wl.block_seeds()[:nblk]] if nblk <= wl.blocks else \
            [wl.seed_base + i + rank * nblk for i in range(nblk)]
        logits, hidden, target, planted = gen_blocks(wl, seeds, dev)
        B = 1
    else:
        # several distinct batches per step, captured together like the batch-1 blocks (a
        # serving loop does not pay one graph launch per call)
        batch_bytes = wl.B * wl.L * wl.V * es
        nblk = args.batches or max(1, min(8, int(1.6e9 // batch_bytes)))
        B = wl.B
        tdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
        logits = torch.empty((nblk, B, wl.L, wl.V), dtype=tdt, device=dev)
        hidden = torch.empty((nblk, B, wl.L, wl.H), dtype=tdt, device=dev)
        target = torch.empty((nblk, B, wl.n_tgt, wl.H), dtype=tdt, device=dev)
        planted = None
        for j in range(nblk):
            inp = workloads.batch_inputs(wl, [s + rank * 100000 + j * 1000003 for s in wl.seeds()])
            logits[j] = upload(inp["logits"], wl.dtype, dev)
            hidden[j] = upload(inp["hidden"], wl.dtype, dev)
            target[j] = upload(inp["target"], wl.dtype, dev)
            if inp["planted"] is not None:
                if planted is None:
                    planted = np.zeros((nblk,) + inp["planted"].shape, np.int32)
                planted[j] = inp["planted"]
            del inp
    ws = head.workspace(B)
    tokens = torch.empty((nblk, B, wl.L), dtype=torch.int32, device=dev)

    # one call outside capture (configures kernels, counts launches per call)
    n0 = ll.launch_count()
    ll.select_block(head, logits[0], hidden[0], target[0], ws=ws, tokens=tokens[0])
    launches_per_call = ll.launch_count() - n0
    torch.cuda.synchronize()
    if ws.status() != 0:
        raise RuntimeError("device status set on the first call")

    G = max(1, min(args.calls_per_graph, nblk))
    graphs = []
    for i0 in range(0, nblk, G):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for i in range(i0, min(i0 + G, nblk)):
                ll.select_block(head, logits[i], hidden[i], target[i], ws=ws, tokens=tokens[i])
        graphs.append(g)
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

    # ---- end to end: pinned host inputs -> device -> select -> tokens back to pinned host
    nh = min(args.e2e_host_blocks, nblk)
    h_logits = torch.empty((nh,) + tuple(logits.shape[1:]), dtype=logits.dtype).pin_memory()
    h_hidden = torch.empty((nh,) + tuple(hidden.shape[1:]), dtype=hidden.dtype).pin_memory()
    h_target = torch.empty((nh,) + tuple(target.shape[1:]), dtype=target.dtype).pin_memory()
    h_logits.copy_(logits[:nh].cpu())
    h_hidden.copy_(hidden[:nh].cpu())
    h_target.copy_(target[:nh].cpu())
    h_tokens = torch.empty((nh, B, wl.L), dtype=torch.int32).pin_memory()
    d_logits = torch.empty_like(logits[0])
    d_hidden = torch.empty_like(hidden[0])
    d_target = torch.empty_like(target[0])
    d_tokens = torch.empty((B, wl.L), dtype=torch.int32, device=dev)
    # each e2e graph holds G calls, each: its inputs host -> device, select, tokens -> host
    e2e_graphs = []
    for k in range(-(-nh // G)):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for j in range(G):
                i = (k * G + j) % nh
                d_logits.copy_(h_logits[i], non_blocking=True)
                d_hidden.copy_(h_hidden[i], non_blocking=True)
                d_target.copy_(h_target[i], non_blocking=True)
                ll.select_block(head, d_logits, d_hidden, d_target, ws=ws, tokens=d_tokens)
                h_tokens[i].copy_(d_tokens, non_blocking=True)
        e2e_graphs.append(g)
    n_e2e_replays = -(-nblk // G)
    e2e_calls = n_e2e_replays * G

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
    e2e_value = e2e_calls * B * args.steps * world / (e2e_ms / 1e3) if not batch1 else \
        e2e_calls * args.steps * world / (e2e_ms / 1e3)
    h2d = (d_logits.numel() * d_logits.element_size() + d_hidden.numel() * d_hidden.element_size()
           + d_target.numel() * d_target.element_size()) * e2e_calls
    d2h = d_tokens.numel() * 4 * e2e_calls

    # ---- the exact best path (App. E) in place of the greedy walk: the same calls on a
    # sample of the blocks, both walks captured alike and timed back to back
    nv = min(nblk, 100)
    walk_ms = {}
    for walk in ("greedy", "viterbi"):
        gl = []
        for i0 in range(0, nv, G):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                for i in range(i0, min(i0 + G, nv)):
                    ll.select_block(head, logits[i], hidden[i], target[i], ws=ws, tokens=tokens[i],
                                    walk=walk)
            gl.append(g)
        for g in gl:
            g.replay()
        torch.cuda.synchronize()
        best = None
        for _ in range(3):
            w0 = torch.cuda.Event(enable_timing=True)
            w1 = torch.cuda.Event(enable_timing=True)
            w0.record(stream)
            for g in gl:
                g.replay()
            w1.record(stream)
            torch.cuda.synchronize()
            t = w0.elapsed_time(w1)
            best = t if best is None else min(best, t)
        walk_ms[walk] = best / nv
    if ws.status() != 0:
        raise RuntimeError("device status set by the walk comparison")

    # ---- diagnostics of the chosen blocks (Eq. "localar" probabilities and gaps along the
    # walk; coverage / oracle prefix / accepted prefix against the planted tokens)
    diag = None
    if planted is not None:
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
        dg = torch.cuda.CUDAGraph()
        with torch.cuda.graph(dg):
            for _ in range(50):
                diag_call()
        dg.replay()
        torch.cuda.synchronize()
        d0 = torch.cuda.Event(enable_timing=True)
        d1 = torch.cuda.Event(enable_timing=True)
        d0.record(stream)
        dg.replay()
        d1.record(stream)
        torch.cuda.synchronize()
        diag = {"truth": "planted token per slot", "blocks": nd * B,
                "mean_oracle_prefix": round(prefix_sum / (nd * B), 3),
                "mean_accepted": round(acc_sum / (nd * B), 3),
                "us_per_call": round(d0.elapsed_time(d1) * 1e3 / 50, 2),
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
    tg = torch.cuda.CUDAGraph()
    with torch.cuda.graph(tg):
        for i in range(reps):
            ll.topk_lse(flat[i % nblk], wl.K, ws=tk_ws)
    tg.replay()
    torch.cuda.synchronize()
    k0 = torch.cuda.Event(enable_timing=True)
    k1 = torch.cuda.Event(enable_timing=True)
    k0.record(stream)
    tg.replay()
    k1.record(stream)
    torch.cuda.synchronize()
    tk_ms = k0.elapsed_time(k1) / reps
    alg_bytes = rows * wl.V * es
    pk, pk_kind = peaks()
    hbm = float(pk.get("hbm_gbs", FALLBACK_HBM_GBS))
    achieved = alg_bytes / (tk_ms / 1e3) / 1e9
    roofline = {"kernel": "topk_lse_kernel", "bound": "hbm", "achieved": round(achieved, 1),
                "peak": hbm, "peak_kind": pk_kind, "unit": "GB/s", "frac": round(achieved / hbm, 4),
                "traffic": profiled_traffic("topk_lse.cu", wl.name),
                "alg_bytes_per_launch": alg_bytes, "us_per_launch": round(tk_ms * 1e3, 3)}

    # ---- the vocabulary-sharded pass (a tensor-parallel LM head's logits), simulated on
    # this GPU: P contiguous vocabulary slices, each summarised into per-row records
    # (what one rank computes), then the merge of the gathered records
    P = 4
    sl = [flat[0][:, a:b].contiguous() for a, b in shards.bounds(wl.V, P)]
    sws = [ll.Workspace(ll.lib().lilicorr_topk_lse_partial_workspace_bytes(rows, t.shape[1], wl.K))
           for t in sl]
    recs = torch.stack([ll.topk_lse_partial(t, wl.K, a, ws=w)
                        for t, (a, _), w in zip(sl, shards.bounds(wl.V, P), sws)])
    torch.cuda.synchronize()

    def timed(fn, n=20):
        fn()
        torch.cuda.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr):
            for _ in range(n):
                fn()
        gr.replay()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        gr.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / n

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
    lm_head = None
    if wl.dtype == "bf16":
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
    if in_bytes > l2_bytes:
        l2_note = "inputs larger than L2 (%.0f MB): %.2f GB of logits" % (l2_bytes / 1e6, in_bytes / 1e9)
        l2_note += (" in %d distinct resident blocks" % nblk if batch1 else
                    " in %d distinct resident batches" % nblk)
    else:
        l2_note = ("inputs fit in L2 (%.2f GB of logits, L2 %.0f MB): a profiling size, "
                   "not a bench configuration" % (in_bytes / 1e9, l2_bytes / 1e6))
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": {"workload": wl.name, "B": B, "L": wl.L, "V": wl.V, "K": wl.K, "d": wl.d,
                   "D": wl.D, "H": wl.H, "blocks_per_step": nblk,
                   "l2": l2_note,
                   "graphs": f"{G} select_block calls per CUDA graph, replayed",
                   "parallelism": f"dp{world}"},
        "us_per_block": ms_per_step * 1e3 / nblk,
        "clocks": clk,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "note": f"pinned host blocks cycled ({nh} distinct), copies captured with each call"},
        "gpu_launches": launches_per_call * nblk * args.steps,
        "diagnostics": diag,
        "walk_viterbi": {"us_per_call": round(walk_ms["viterbi"] * 1e3, 2),
                         "greedy_us_per_call": round(walk_ms["greedy"] * 1e3, 2),
                         "block_rate_cost": round(walk_ms["viterbi"] / walk_ms["greedy"] - 1, 4),
                         "sample": f"{nv} calls of this workload, best of 3"},
        "vocab_sharded": sharded,
        "lm_head_fused": lm_head,
        "roofline": roofline,
    }
    if rank == 0 and not args.no_cpu_baseline:
        seeds_cpu = wl.block_seeds() if batch1 else wl.seeds()
        v, n, dt = oracle_blocks_per_s(wl, W, seeds_cpu, args.cpu_seconds)
        result["cpu_baseline"] = {
            "value": v, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{n} sequences of the {wl.name} workload in {dt:.1f} s (fp64 NumPy, 1 thread)"}
    if rank == 0:
        print(json.dumps(result))
    head.close()


def main():
    args = parse_args()
    world, rank, local = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_ours(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
