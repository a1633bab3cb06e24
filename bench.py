#!/usr/bin/env python3
"""Benchmark: CURE repair-verify steps per second on the batched serving shape.

One step = the six stages over one batch (score_draft, build_tree, 28 layers
of tree attention, target argmax + acceptance walk, resync of every layer's
cache), all through the C ABI on one stream, inputs resident in HBM.

Workload (synthetic, seeded): batch 32, block 16, vocab 151936, tau 0.8,
budget 16 repair nodes, 3 branches at a UFP; 28 layers of 28 query / 4 kv
heads, head_dim 128, cache lengths U[1024, 8192] in shuffled 16-token pages.
The KV traffic of one step (about 8.5 GB) is far larger than L2, so no L2
flush is needed between steps.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
Under torchrun each rank runs its own batch (weak scaling, no collective on
the data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

# DRAM bytes (read + write) of one tree-attention launch on this workload, from
# one ncu capture (dram__bytes_read.sum + dram__bytes_write.sum) of the kernel
# source with the given sha256 prefix; another source reports null
ATTN_TRAFFIC = {"2d1748d0f70bce81": 312700160}

METRIC = "repair-verify steps/s at batch 32, block 16; tree-attn & vocab-scan HBM GB/s vs peak"
WORKLOAD = "serve32"


def attn_source_digest() -> str:
    import hashlib
    src = os.path.join(ROOT, "paper_2608_00531_gb300", "csrc", "k_attn_tc.cu")
    with open(src, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:16]


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return dict(hbm_gbs=float(d["hbm_gbs"]), bf16_tflops=float(d["bf16_tflops"]),
                    bf16_tflops_sustained=float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                    source="measured")
    return dict(hbm_gbs=6800.0, bf16_tflops=1900.0, bf16_tflops_sustained=1700.0, source="fallback")


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """Samples SM clocks and throttle reasons with nvidia-smi while the timed
    region runs; samples are time-stamped on arrival and only those taken
    between `mark_start` and `mark_stop` are summarised."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    INTERVAL_MS = 50

    def __init__(self, dev_index: int):
        self.proc = None
        self.dev_index = dev_index
        self.lines = []
        self.t0 = self.t1 = None
        self.thread = None

    def start(self, wait_first_s: float = 5.0):
        import threading
        try:
            bus = None
            try:
                pr = torch.cuda.get_device_properties(self.dev_index)
                bus = "%08X:%02X:%02X.0" % (pr.pci_domain_id, pr.pci_bus_id, pr.pci_device_id)
            except Exception:
                bus = None
            cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                   "-lms", str(self.INTERVAL_MS)]
            if bus:
                cmd += ["--id=" + bus]
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return

        def reader():
            for line in self.proc.stdout:
                self.lines.append((time.time(), line))

        self.thread = threading.Thread(target=reader, daemon=True)
        self.thread.start()
        t_end = time.time() + wait_first_s   # the first sample shows the sampler is live
        while not self.lines and time.time() < t_end and self.proc.poll() is None:
            time.sleep(0.01)

    def mark_start(self):
        self.t0 = time.time()

    def mark_stop(self):
        self.t1 = time.time()

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(2 * self.INTERVAL_MS / 1e3)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)
        t0 = self.t0 if self.t0 is not None else 0.0
        t1 = self.t1 if self.t1 is not None else time.time()
        inside = [ln for ts, ln in self.lines if t0 <= ts <= t1 + self.INTERVAL_MS / 1e3]
        sm, mx, reasons = [], [], set()
        for line in inside:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, val in zip(("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                                  "sw_power_cap"), parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm), "interval_ms": self.INTERVAL_MS}


# ------------------------------------------------------------------ ranks
def rank_seed(base_seed: int, rank: int) -> int:
    """Each rank draws its own batch (weak scaling: the per-GPU work is fixed)."""
    return base_seed + 7 * rank


def max_over_ranks(ms: float, world: int, device) -> float:
    """The job's time is the slowest rank's; every rank gets it."""
    if world == 1:
        return ms
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_steps_per_s(ms_max: float, steps: int, world: int) -> float:
    """Whole-job throughput: the steps all ranks ran over the slowest rank's time."""
    return world * steps / (ms_max / 1e3)


# ------------------------------------------------------------------ workload
POOL = 4  # draft/target input sets cycled over the steps, so that tree shapes vary


def make_workload(dev, rank: int, layers_override=None, pool: int = POOL):
    from paper_2608_00531_gb300 import cure, workload as W
    from paper_2608_00531_gb300.step import RepairVerifyStep, StepInputs
    w = W.WORKLOADS[WORKLOAD]
    seed = rank_seed(w.seed, rank)
    layers = layers_override or w.layers
    B, K, N, D = w.batch, w.block, w.n_max, 128
    L = W.cache_lengths(w, seed=seed)
    # pages for slots up to L_b + n_max - 1: room for the in-place layout's tree rows
    table, npages = W.block_table(L, N - 1, seed)
    g = torch.Generator(device=dev).manual_seed(seed)

    def rnd(*shape, std=1.0):
        return (torch.randn(*shape, generator=g, device=dev) * std).to(torch.bfloat16)

    kcs = [rnd(npages, 16, w.heads_kv, D) for _ in range(layers)]
    vcs = [rnd(npages, 16, w.heads_kv, D) for _ in range(layers)]
    q = rnd(layers, B, N, w.heads_q, D)
    tk = rnd(layers, B, N, w.heads_kv, D)
    tv = rnd(layers, B, N, w.heads_kv, D)
    bt = torch.from_numpy(table).to(dev)
    kv = cure.kv_desc(w.heads_kv, D, table.shape[1], bt, 16, npages)
    st = RepairVerifyStep(B, K, w.vocab, w.topk, w.tau, w.budget, w.branches, 1, layers, w.heads_q, kv, dev)
    lens = torch.from_numpy(L).to(dev)
    xs, trees = [], []
    for i in range(pool):
        # each set: its own draft block (so its own tree) and target; the
        # target's logits come from a stand-in target model applied to the
        # tree the set produces (built once here, outside the timed region)
        si = seed + 1009 * i
        d = W.draft_block(w, seed=si)
        draft = d.logits.to(dev)
        root = torch.from_numpy(d.root_tok).to(dev)
        ids, vals, margin, lp = cure.cure_score_draft(draft, w.topk)
        tree = cure.cure_build_tree(ids, margin, root, lens, w.tau, w.budget, w.branches)
        th = {k_: v.cpu().numpy() for k_, v in tree.items()}
        truth = W.target_truth(w, d, si)
        targ = W.synthetic_target_ids(truth, th["n_nodes"], th["tok"], th["parent"], th["depth"], w.vocab, si)
        tl = W.target_logits(targ, w.vocab, si).to(dev)
        xs.append(StepInputs(draft, root, lens, None, q, tk, tv, tl))
        trees.append(th)
    return dict(w=w, st=st, x=xs[0], xs=xs, kcs=kcs, vcs=vcs, kv=kv, L=L, tree=trees[0], trees=trees, seed=seed,
                layers=layers, npages=npages, table=table)


def algorithmic(wl, th=None):
    """Bytes and flops the method must move or compute per step, per stage
    (for the input set whose tree is th)."""
    w, L = wl["w"], wl["L"].astype(np.int64)
    th = wl["tree"] if th is None else th
    B, K, N, V, D = w.batch, w.block, w.n_max, w.vocab, 128
    Hq, Hkv, layers = w.heads_q, w.heads_kv, wl["layers"]
    n = th["n_nodes"].astype(np.int64)
    anc_sizes = np.array([[bin(int(x)).count("1") for x in th["anc"][b, :, 0].view(np.uint64)]
                          for b in range(B)])
    vis = sum(int(L[b]) * int(n[b]) + int(anc_sizes[b, :n[b]].sum()) for b in range(B))
    attn_bytes = int((L * Hkv * D * 2 * 2).sum() + (n * (2 * Hq + 2 * Hkv) * D * 2).sum())
    attn_flops = 4 * Hq * D * vis
    scan_bytes = B * K * V * 2
    argmax_bytes = int(n.sum()) * V * 2
    return dict(attn_bytes=attn_bytes, attn_flops=attn_flops, scan_bytes=scan_bytes,
                argmax_bytes=argmax_bytes, mean_nodes=float(n.mean()))


def w_heads_kv(wl):
    return wl["w"].heads_kv


def resync_bytes(acc_len, layers, Hkv, D=128):
    rows = int((acc_len.astype(np.int64) + 1).sum())
    return 2 * 2 * rows * layers * Hkv * D * 2   # read + write, K and V


# ------------------------------------------------------------------ cpu baseline (oracle)
def cpu_baseline(budget_s: float = 12.0):
    """The oracle, as it stands, timed on host cores over a bounded sample of the
    workload and extrapolated to one full step."""
    import oracle
    from paper_2608_00531_gb300 import workload as W
    w = W.WORKLOADS[WORKLOAD]
    B, K, N, V, k = w.batch, w.block, w.n_max, w.vocab, w.topk
    d = W.draft_block(w)
    L = W.cache_lengths(w)
    table, npages = W.block_table(L, K, w.seed)
    x = W.bf16_to_f64(d.logits).reshape(B, K, V)
    rng = np.random.default_rng(0)
    t_score = t_tree = t_attn = t_acc = t_rs = 0.0
    seqs = 0
    t_start = time.perf_counter()
    ids_all = np.zeros((B, K, k), np.int64)
    m_all = np.zeros((B, K), np.float32)
    # stage 1 + 2/3 over sequences until the budget's first third is used
    for b in range(B):
        t0 = time.perf_counter()
        ids, _, m, _, _ = oracle.score_draft(x[b], k)
        t_score += time.perf_counter() - t0
        ids_all[b], m_all[b] = ids, m.astype(np.float32)
        seqs += 1
        if time.perf_counter() - t_start > budget_s / 3:
            break
    t0 = time.perf_counter()
    t = oracle.build_tree(ids_all[:seqs], m_all[:seqs], d.root_tok[:seqs], L[:seqs], w.tau, w.budget,
                          w.branches, 1)
    t_tree = time.perf_counter() - t0
    # stage 4: one layer for the sampled sequences (sequence-layer units)
    Hq, Hkv, D = w.heads_q, w.heads_kv, 128
    attn_units = 0
    t_att0 = time.perf_counter()
    for b in range(seqs):
        Lb = int(L[b])
        kc = rng.standard_normal((Lb, Hkv, D)).astype(np.float32)
        vc = rng.standard_normal((Lb, Hkv, D)).astype(np.float32)
        q = rng.standard_normal((1, N, Hq, D))
        tk = rng.standard_normal((1, N, Hkv, D))
        t0 = time.perf_counter()
        oracle.tree_attn(q, tk, tk, kc[None], vc[None], np.array([Lb]), t["n_nodes"][b:b + 1],
                         t["anc"][b:b + 1], 1.0 / math.sqrt(D))
        t_attn += time.perf_counter() - t0
        attn_units += 1
        if time.perf_counter() - t_att0 > budget_s / 2:
            break
    # stage 5 for the sampled sequences
    tl = rng.standard_normal((seqs * N, V))
    t0 = time.perf_counter()
    targ = oracle.row_argmax(tl).reshape(seqs, N)
    acc = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], K)
    t_acc = time.perf_counter() - t0
    # stage 6 for the sampled sequences, one layer (per sequence-layer)
    kcs = [np.zeros((npages, 16, Hkv, D))]
    vcs = [np.zeros((npages, 16, Hkv, D))]
    trk = rng.standard_normal((1, seqs, N, Hkv, D))
    t0 = time.perf_counter()
    oracle.resync(kcs, vcs, trk, trk, acc["path_nodes"], acc["accept_len"], acc["diverge_depth"],
                  acc["out_tokens"], L[:seqs], K, table[:seqs], 16)
    t_rs = time.perf_counter() - t0
    per_step = (t_score / seqs * B + t_tree / seqs * B + t_attn / attn_units * B * w.layers
                + t_acc / seqs * B + t_rs / seqs * B * w.layers)
    sample = (f"oracle (numpy fp64, 1 thread) on {seqs} of {B} sequences for the scan/tree/accept stages, "
              f"{attn_units} sequence-layers of tree attention and one layer of resync; extrapolated "
              f"linearly to 32 sequences x {w.layers} layers")
    return dict(value=1.0 / per_step, unit="steps/s", cores=1, kind="oracle", sample=sample,
                seconds_per_step_extrapolated=per_step,
                stage_seconds=dict(score=t_score / seqs * B, tree=t_tree / seqs * B,
                                   attn=t_attn / attn_units * B * w.layers, accept=t_acc / seqs * B,
                                   resync=t_rs / seqs * B * w.layers))


# ------------------------------------------------------------------ main
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--layers", type=int, default=None, help=argparse.SUPPRESS)
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return
        run_reference(args)
        return

    os.environ.setdefault("OMP_NUM_THREADS", "1")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import cure

    wl = make_workload(dev, rank, args.layers)
    st, xs, kcs, vcs = wl["st"], wl["xs"], wl["kcs"], wl["vcs"]
    P = len(xs)
    stream = torch.cuda.current_stream()

    acc_lens = [None] * P
    for i in range(max(args.warmup, P)):
        r = st.run(xs[i % P], kcs, vcs)
        torch.cuda.synchronize()
        acc_lens[i % P] = r["acc"]["accept_len"].cpu().numpy()
    assert cure.cure_device_error() == 0
    algs = [algorithmic(wl, th) for th in wl["trees"]]
    # the timed steps cycle over the sets: per-step averages
    sel = [s % P for s in range(args.steps)]
    alg = {k_: float(np.mean([algs[i][k_] for i in sel])) for k_ in algs[0]}

    # per-op events inside the timed region (same stream as the launches)
    Ly = wl["layers"]
    # one event pair around the step's attention launches (events between
    # the launches would stop each from starting its set-up under the
    # previous one, which it does as a programmatic dependent launch)
    ev_attn = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    ev_scan = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    ev_rs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]

    def timed_step(s):
        x = xs[s % P]
        e = ev_scan[s]
        e[0].record(stream)
        cure.cure_score_draft(x.draft_logits, st.k, out=st.score)
        e[1].record(stream)
        tree = cure.cure_build_tree(st.score[0], st.score[2], x.root_tok, x.cache_len, st.tau, st.R,
                                    st.branches, st.depth, x.redraft, st.max_ufp, out=st.tree)
        ea = ev_attn[s]
        ea[0].record(stream)
        for l in range(Ly):
            cure.cure_tree_attn(x.q[l], x.tree_k[l], x.tree_v[l], kcs[l], vcs[l], st.kv, x.cache_len,
                                tree["n_nodes"], tree["anc"], st.scale, out=st.attn_out[l],
                                workspace=st.workspace)
        ea[1].record(stream)
        acc = cure.cure_accept(tree, st.K, target_logits=x.target_logits, targ=st.targ, out=st.acc)
        ev_rs[s][0].record(stream)
        cure.cure_resync_kv(kcs, vcs, st.kv, x.tree_k, x.tree_v, acc, x.cache_len, st.K,
                            cache_len_out=st.cache_len_out, out=st.rs)
        ev_rs[s][1].record(stream)

    clk = ClockSampler(local)
    clk.start()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    clk.mark_start()
    t0.record(stream)
    for s in range(args.steps):
        timed_step(s)
    t1.record(stream)
    torch.cuda.synchronize()
    clk.mark_stop()
    clocks = clk.stop()
    ms = max_over_ranks(t0.elapsed_time(t1), world, dev)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    assert cure.cure_device_error() == 0
    attn_ms = [ev_attn[s][0].elapsed_time(ev_attn[s][1]) / Ly for s in range(args.steps)]
    scan_ms = [ev_scan[s][0].elapsed_time(ev_scan[s][1]) for s in range(args.steps)]
    rs_ms = float(np.mean([ev_rs[s][0].elapsed_time(ev_rs[s][1]) for s in range(args.steps)]))
    rs_b = float(np.mean([resync_bytes(acc_lens[i], Ly, w_heads_kv(wl)) for i in sel]))
    attn_avg = float(np.mean(attn_ms))
    scan_avg = float(np.mean(scan_ms))

    # the same step replayed as CUDA graphs (one per input set), timed the same way
    graph = None
    rs_graph_ms = None
    scan_graph_ms = None
    if not args.no_graph:
        graph = run_graphs(st, xs, kcs, vcs, args.steps, world, dev)
        rs_graph_ms = resync_graph_ms(st, xs[sel[-1]], kcs, vcs)
        scan_graph_ms = call_graph_ms(lambda: cure.cure_score_draft(xs[sel[-1]].draft_logits, st.k, out=st.score))

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(wl, st, kcs, vcs, dev, max(3, min(args.steps, 10)), world)

    # the in-place tree-KV layout on the same shapes; last, since its resync
    # moves rows inside the caches
    in_place = None
    if not args.no_graph:
        in_place = in_place_stage(st, xs[sel[-1]], kcs, vcs)

    if rank != 0:
        return
    pk = peaks()
    ms_step = ms / args.steps
    value = job_steps_per_s(ms, args.steps, world)
    attn_gbs = alg["attn_bytes"] / (attn_avg * 1e-3) / 1e9
    attn_tflops = alg["attn_flops"] / (attn_avg * 1e-3) / 1e12
    scan_gbs = alg["scan_bytes"] / (scan_avg * 1e-3) / 1e9
    intensity = alg["attn_flops"] / alg["attn_bytes"]
    ridge = pk["bf16_tflops_sustained"] * 1e12 / (pk["hbm_gbs"] * 1e9)
    bound = "hbm" if intensity < ridge else "tensor"
    if bound == "hbm":
        roof = {"bound": "hbm", "achieved": round(attn_gbs, 1), "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": round(attn_gbs / pk["hbm_gbs"], 4)}
    else:
        roof = {"bound": "tensor", "achieved": round(attn_tflops, 1), "peak": pk["bf16_tflops_sustained"],
                "unit": "TFLOP/s", "frac": round(attn_tflops / pk["bf16_tflops_sustained"], 4)}
    roof.update({"traffic": ATTN_TRAFFIC.get(attn_source_digest()),
                 "traffic_source": "ncu dram__bytes_read.sum + dram__bytes_write.sum of this kernel source "
                                   "(one layer of this workload); null when the source has changed",
                 "kernel": "tree attention (tree_attn_tc_kernel, persistent, split units merged in-kernel), per layer: "
                           "the step's 28 back-to-back launches timed together, divided by 28",
                 "algorithmic_bytes_per_launch": alg["attn_bytes"],
                 "algorithmic_flops_per_launch": alg["attn_flops"], "avg_launch_ms": round(attn_avg, 4),
                 "peak_source": pk["source"] + " (MEASURED_PEAKS.json hbm_gbs)"})
    out = {
        "metric": METRIC, "value": round(value, 3), "unit": "steps/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "batch 32, block 16, vocab 151936, tau 0.8, R 16, top-3 branches; 28 layers "
                               "of tree attention 28q/4kv heads x 128, KV lengths U[1024,8192] paged 16",
                   "batch": 32, "block": 16, "vocab": 151936, "layers": Ly, "heads_q": 28, "heads_kv": 4,
                   "head_dim": 128, "paged": True, "per_gpu_batch": 32,
                   "l2": "no flush: inputs larger than L2 (KV read per step %.1f GB)" % (alg["attn_bytes"] * Ly / 1e9)},
        "roofline": roof,
        "stages": {"vocab_scan_ms": round(scan_avg, 4), "vocab_scan_gbs": round(scan_gbs, 1),
                   "vocab_scan_graph_ms": None if scan_graph_ms is None else round(scan_graph_ms, 4),
                   "vocab_scan_graph_frac": None if scan_graph_ms is None else
                   round(alg["scan_bytes"] / (scan_graph_ms * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                   "vocab_scan_frac": round(scan_gbs / pk["hbm_gbs"], 4),
                   "resync_call_ms": round(rs_ms, 4),
                   "resync_call_gbs": round(rs_b / (rs_ms * 1e-3) / 1e9, 1),
                   "resync_call_frac": round(rs_b / (rs_ms * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                   "resync_graph_ms": None if rs_graph_ms is None else round(rs_graph_ms, 4),
                   "resync_graph_frac": None if rs_graph_ms is None else
                   round(resync_bytes(acc_lens[sel[-1]], Ly, w_heads_kv(wl)) / (rs_graph_ms * 1e-3) / 1e9
                         / pk["hbm_gbs"], 4),
                   "tree_attn_ms_per_layer": round(attn_avg, 4),
                   "tree_attn_tflops": round(attn_tflops, 1), "tree_attn_intensity_flop_per_byte": round(intensity, 1),
                   "mean_tree_nodes": round(alg["mean_nodes"], 3),
                   "mean_accept_len": round(float(np.mean([acc_lens[i].mean() for i in sel])), 3),
                   "input_sets": P, "in_place": in_place},
        "gpu_launches": st.launches_per_step * args.steps,
        "clocks": clocks,
    }
    if e2e:
        out["e2e"] = e2e
    if graph:
        out["graph"] = graph
    if not args.no_cpu_baseline and world == 1:
        out["cpu_baseline"] = cpu_baseline()
    print(json.dumps(out), flush=True)


def in_place_stage(st, x, kcs, vcs):
    """The in-place tree-KV layout (node j's K/V rows at cache slot L + j, no
    tree tensors) on the step's shapes: the layers of tree attention replayed
    as a CUDA graph, per layer, and the resync call, replayed alone.  The cache
    contents are the bench's random rows: these are timings, not results."""
    try:
        from paper_2608_00531_gb300 import cure
        tree, Ly = st.tree, st.layers

        def attn():
            for l in range(Ly):
                p = st.layer_map[l]
                cure.cure_tree_attn(x.q[l], None, None, kcs[p], vcs[p], st.kv, x.cache_len, tree["n_nodes"],
                                    tree["anc"], st.scale, out=st.attn_out[l], workspace=st.workspace)

        def resync():
            kl = [kcs[st.layer_map[l]] for l in range(Ly)]
            vl = [vcs[st.layer_map[l]] for l in range(Ly)]
            cure.cure_resync_kv(kl, vl, st.kv, None, None, st.acc, x.cache_len, st.K, n_max=st.n_max,
                                cache_len_out=st.cache_len_out, out=st.rs)

        a_ms = call_graph_ms(attn, calls=2, reps=5)
        r_ms = call_graph_ms(resync)
        if cure.cure_device_error() != 0:
            return None
        return {"tree_attn_ms_per_layer": None if a_ms is None else round(a_ms / Ly, 4),
                "resync_graph_ms": None if r_ms is None else round(r_ms, 4),
                "note": "tree rows written by the target at cache slots L + j; resync moves only the rows "
                        "past the divergence depth"}
    except Exception as e:  # reported as missing, the bench line stands
        print(f"in-place timing failed: {type(e).__name__}: {e}"[:300], file=sys.stderr)
        return None


def call_graph_ms(fn, calls=20, reps=5):
    """One library call, back to back inside a CUDA graph (consecutive
    launches overlap programmatically as in the step): its device time
    without the event pair's launch gap.  None if the capture fails."""
    try:
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            fn()
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(calls):
                fn()
        g.replay()
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            g.replay()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / (calls * reps)
    except Exception as e:  # reported as missing, the bench line stands
        print(f"graph timing failed: {type(e).__name__}: {e}"[:300], file=sys.stderr)
        return None


def resync_graph_ms(st, x, kcs, vcs, calls=20, reps=5):
    """The resync call alone, back to back inside a CUDA graph (its launches
    overlap programmatically as they do in the step): the call's device time
    without the event pair's launch gap.  The calls rewrite the same cache
    slots with the same rows."""
    try:
        from paper_2608_00531_gb300 import cure
        acc = st.acc
        def call():
            cure.cure_resync_kv(kcs, vcs, st.kv, x.tree_k, x.tree_v, acc, x.cache_len, st.K,
                                cache_len_out=st.cache_len_out, out=st.rs)
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            call()
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(calls):
                call()
        g.replay()
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            g.replay()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / (calls * reps)
    except Exception as e:  # reported as missing, the bench line stands
        print(f"resync graph timing failed: {type(e).__name__}: {e}"[:300], file=sys.stderr)
        return None


def run_graphs(st, xs, kcs, vcs, steps, world, dev):
    """The step captured once per input set as a CUDA graph (launches and
    their programmatic edges recorded) and replayed, cycling over the sets."""
    try:
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            for x in xs:
                st.run(x, kcs, vcs)
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        graphs = []
        for x in xs:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                st.run(x, kcs, vcs)
            graphs.append(g)
        for g in graphs:
            g.replay()
        torch.cuda.synchronize()
        if world > 1:
            import torch.distributed as dist
            dist.barrier()
        stream = torch.cuda.current_stream()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for s in range(steps):
            graphs[s % len(graphs)].replay()
        b.record(stream)
        torch.cuda.synchronize()
        ms = max_over_ranks(a.elapsed_time(b), world, dev) / steps
        return {"value": round(job_steps_per_s(ms * steps, steps, world), 3), "unit": "steps/s",
                "ms_per_step": round(ms, 4), "steps": steps}
    except Exception as e:  # report, do not fail the bench line
        return {"error": f"{type(e).__name__}: {e}"[:200]}


def run_e2e(wl, st, kcs, vcs, dev, steps, world=1):
    """Same step through the public API with inputs in pinned host memory
    (RepairVerifyStep.run_from_host): host-to-device copies of the step's
    inputs and a device-to-host read of the accept results inside the timed
    region.  Whole-job value over ranks."""
    from paper_2608_00531_gb300.step import StepInputs
    x = wl["x"]
    host = {k_: getattr(x, k_).cpu().pin_memory() for k_ in ("draft_logits", "root_tok", "cache_len", "q",
                                                               "tree_k", "tree_v", "target_logits")}
    outs = torch.empty(4, st.B, st.K + 2, dtype=torch.int32).pin_memory()
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    d2h = outs.numel() * outs.element_size()
    stream = torch.cuda.current_stream()
    xh = StepInputs(host["draft_logits"], host["root_tok"], host["cache_len"], None, host["q"], host["tree_k"],
                    host["tree_v"], host["target_logits"])

    def one():
        # the public step with host inputs: it streams them in on a copy
        # stream, each stage waiting for its own inputs
        r = st.run_from_host(xh, kcs, vcs)
        outs[0, :, 0].copy_(r["acc"]["accept_len"], non_blocking=True)
        outs[1].copy_(r["acc"]["out_tokens"], non_blocking=True)
        outs[2].copy_(r["resync"]["replay_tokens"], non_blocking=True)
        outs[3, :, 0].copy_(r["resync"]["n_replay"], non_blocking=True)
        stream.synchronize()

    for _ in range(2):
        one()
    torch.cuda.synchronize()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(steps):
        one()
    b.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(a.elapsed_time(b), world, dev) / steps
    return {"value": round(job_steps_per_s(ms * steps, steps, world), 3), "unit": "steps/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "ms_per_step": round(ms, 4), "steps": steps}


def run_reference(args):
    """The reference arm: the oracle (the paper's method restated on the CPU),
    timed as it stands on host cores, each step a bounded sample of the workload."""
    vals = []
    budget = max(2.0, min(12.0, 150.0 / max(1, args.steps + args.warmup)))
    for i in range(args.warmup + args.steps):
        cb = cpu_baseline(budget_s=budget)
        if i >= args.warmup:
            vals.append(cb["seconds_per_step_extrapolated"])
    sec = float(np.mean(vals))
    v = 1.0 / sec
    out = {"impl": "reference", "metric": METRIC, "value": v, "unit": "steps/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": "batch 32, block 16, vocab 151936, tau 0.8, R 16, top-3 branches; 28 layers "
                                  "of tree attention 28q/4kv heads x 128, KV lengths U[1024,8192] paged 16"},
           "cpu_baseline": {"value": v, "unit": "steps/s", "cores": 1, "kind": "oracle",
                            "sample": cb["sample"]},
           "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
