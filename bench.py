#!/usr/bin/env python3
"""Benchmark: CURE repair-verify steps per second, one configuration per run.

One step = the six stages over one batch (score_draft, build_tree, one tree
attention per layer, target argmax + acceptance walk, resync of every layer's
cache), all through the C ABI on one stream, inputs resident in HBM.

Workloads (synthetic, seeded; --workload, default serve32, the headline):
  serve32   batch 32, block 16, vocab 151936, tau 0.8, budget 16 repair nodes,
            3 branches at a UFP; 28 layers of 28 query / 4 kv heads,
            head_dim 128, cache lengths U[1024, 8192] in shuffled 16-token pages
  tiny      batch 1, block 8, vocab 32000, 1 layer 8/2 heads, L 512
  single8b  batch 1, block 16, vocab 128256, 32 layers 32/8 heads, L 4096
  long64    batch 64, block 16, vocab 128256, 80 layers 64/8 heads, L 32768,
            depth-2 repairs; 80 logical layers run over 8 physical caches
            (logical layer l uses cache l mod 8: 687 GB of KV does not fit)
  sweep16   batch 16, block 32, vocab 151936, 28 layers 28/4 heads, L 8192,
            every budget R in {0,4,8,16,32,64} x tau in {0.25,0.5,1,2,4}
The KV traffic of a step is far larger than L2 at serve32, long64 and sweep16
(the config's "l2" entry says so); the small configurations are latency-bound
and report per-stage microseconds against their roofline time.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                       [--workload NAME]
Under torchrun each rank runs its own batch (weak scaling, no collective on
the data path); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import contextlib
import gc
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# the CPU baseline is the oracle on one host thread: numpy's BLAS pool is
# sized from these before numpy loads
for _v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")
import numpy as np  # noqa: E402
import torch  # noqa: E402

# DRAM bytes (read + write) of one tree-attention launch on this workload, from
# one ncu capture (dram__bytes_read.sum + dram__bytes_write.sum) of the kernel
# sources with the given sha256 prefix; other sources report null
ATTN_SOURCES = ("k_attn_tc.cu", "k_attn.cu", "attn_common.cuh", "tc_ptx.cuh", "common.cuh")
ATTN_TRAFFIC = {"d26aa4a3b7c38beb": 313468672}

DEFAULT_WORKLOAD = "serve32"
# the target model width behind each configuration's LM head (for the fused
# LM-head stage): Qwen3-8B and Llama-3-8B class 4096, the 70B class 8192
D_MODEL = {"tiny": 4096, "single8b": 4096, "serve32": 4096, "long64": 8192, "sweep16": 4096}
CACHE_BUDGET_BYTES = 72e9   # physical KV caches held at once; more layers alias


@contextlib.contextmanager
def quiet_host():
    """A timed region without Python's cyclic garbage collector: a collection
    of the large heap the workload builds would stall the launching thread."""
    gc.collect()
    gc.disable()
    try:
        yield
    finally:
        gc.enable()


def metric_for(w) -> str:
    return (f"repair-verify steps/s at batch {w.batch}, block {w.block}; "
            "tree-attn & vocab-scan HBM GB/s vs peak")


def workload_text(w, layers, phys) -> str:
    cache = (f"KV lengths U[{w.len_lo},{w.len_hi}]" if w.len_lo != w.len_hi else f"KV length {w.len_lo}")
    cache += " paged 16" if w.paged else " contiguous"
    alias = "" if phys == layers else f", {layers} logical layers over {phys} physical caches (l mod {phys})"
    return (f"{w.name}: batch {w.batch}, block {w.block}, vocab {w.vocab}, tau {w.tau}, R {w.budget}, "
            f"top-{w.branches} branches, repair depth {w.repair_depth}; {layers} layers of tree attention "
            f"{w.heads_q}q/{w.heads_kv}kv heads x 128, {cache}{alias}")


def attn_source_digest() -> str:
    """sha256 prefix of the sources the tree-attention launch is built from:
    the kernel, its launch and schedule, and the PTX helpers it inlines."""
    import hashlib
    h = hashlib.sha256()
    for name in ATTN_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_00531_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


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


def target_logits_dev(ids, vocab, seed, dev):
    """The stand-in target's logits drawn on the device: N(0, 1) bf16 with the
    given id of each row planted at +8 (the distribution of
    workload.target_logits, drawn where it is used)."""
    g = torch.Generator(device=dev).manual_seed(int(seed) + 15485863)
    B, N = ids.shape
    x = torch.randn(B, N, vocab, generator=g, device=dev).to(torch.bfloat16)
    x.scatter_(2, torch.from_numpy(ids.astype(np.int64)).to(dev)[:, :, None], 8.0)
    return x


def make_caches(w, L, N, layers, dev, seed):
    """Physical KV caches (as many as fit the cache budget; logical layer l
    uses cache l mod P), the kv descriptor and the block table."""
    from paper_2608_00531_gb300 import cure, workload as W
    D = 128
    g = torch.Generator(device=dev).manual_seed(seed)
    if w.paged:
        # pages for slots up to L_b + n_max - 1: room for the in-place layout's tree rows
        table, npages = W.block_table(L, N - 1, seed)
        shape = (npages, 16, w.heads_kv, D)
        bt = torch.from_numpy(table).to(dev)
        kv = cure.kv_desc(w.heads_kv, D, table.shape[1], bt, 16, npages)
    else:
        table, npages, bt = None, 0, None
        shape = (w.batch, int(L.max()) + N, w.heads_kv, D)
        kv = cure.kv_desc(w.heads_kv, D, shape[1])
    per_layer = 2 * 2 * int(np.prod(shape))
    phys = max(1, min(layers, int(CACHE_BUDGET_BYTES // per_layer)))
    kcs = [(torch.randn(*shape, generator=g, device=dev)).to(torch.bfloat16) for _ in range(phys)]
    vcs = [(torch.randn(*shape, generator=g, device=dev)).to(torch.bfloat16) for _ in range(phys)]
    return dict(kcs=kcs, vcs=vcs, kv=kv, table=table, npages=npages, bt=bt, phys=phys)


def make_workload(dev, rank: int, name: str = DEFAULT_WORKLOAD, layers_override=None, pool: int = POOL,
                  caches=None, **over):
    """The step's inputs for one configuration: `pool` input sets (each its own
    draft block, so its own tree, and its own target), shared Q/K/V and
    caches.  `over` replaces fields of the configuration (tau, budget)."""
    from paper_2608_00531_gb300 import cure, workload as W
    from paper_2608_00531_gb300.step import RepairVerifyStep, StepInputs
    w = W.WORKLOADS[name].replace(**over) if over else W.WORKLOADS[name]
    seed = rank_seed(w.seed, rank)
    layers = layers_override or w.layers
    B, K, N, D = w.batch, w.block, w.n_max, 128
    L = W.cache_lengths(w, seed=seed)
    if caches is None:
        caches = make_caches(w, L, N, layers, dev, seed)
    kcs, vcs, kv, phys = caches["kcs"], caches["vcs"], caches["kv"], caches["phys"]
    g = torch.Generator(device=dev).manual_seed(seed + 1)

    def rnd(*shape, std=1.0):
        return (torch.randn(*shape, generator=g, device=dev) * std).to(torch.bfloat16)

    q = rnd(layers, B, N, w.heads_q, D)
    tk = rnd(layers, B, N, w.heads_kv, D)
    tv = rnd(layers, B, N, w.heads_kv, D)
    st = RepairVerifyStep(B, K, w.vocab, w.topk, w.tau, w.budget, w.branches, w.repair_depth, layers, w.heads_q,
                          kv, dev, layer_map=[l % phys for l in range(layers)])
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
        red = torch.from_numpy(d.redraft).to(dev) if w.repair_depth == 2 else None
        ids, vals, margin, lp = cure.cure_score_draft(draft, w.topk)
        tree = cure.cure_build_tree(ids, margin, root, lens, w.tau, w.budget, w.branches, w.repair_depth, red)
        th = {k_: v.cpu().numpy() for k_, v in tree.items()}
        truth = W.target_truth(w, d, si)
        targ = W.synthetic_target_ids(truth, th["n_nodes"], th["tok"], th["parent"], th["depth"], w.vocab, si)
        tl = target_logits_dev(targ, w.vocab, si, dev)
        xs.append(StepInputs(draft, root, lens, red, q, tk, tv, tl))
        trees.append(th)
    return dict(w=w, st=st, x=xs[0], xs=xs, kcs=kcs, vcs=vcs, kv=kv, L=L, tree=trees[0], trees=trees, seed=seed,
                layers=layers, phys=phys, npages=caches["npages"], table=caches["table"], caches=caches)


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


def resync_bytes(acc_len, layers, Hkv, D=128):
    rows = int((acc_len.astype(np.int64) + 1).sum())
    return 2 * 2 * rows * layers * Hkv * D * 2   # read + write, K and V


# ------------------------------------------------------------------ cpu baseline (oracle)
# the fixed sample of the CPU baseline per configuration: sequences for the
# scan / tree / argmax / walk stages, sequence-layers of attention, sequences
# of the resync (one layer); the same in both arms
CPU_SAMPLE = {"tiny": (1, 1, 1), "single8b": (1, 1, 1), "serve32": (4, 2, 4), "long64": (2, 1, 2),
              "sweep16": (2, 1, 2)}


def cpu_baseline(name: str = DEFAULT_WORKLOAD):
    """The oracle, as it stands, timed on one host core over a fixed sample of
    the configuration (its first sequences, with the configuration's shapes,
    cache lengths, trees and value distributions), extrapolated linearly to
    one full step: sequences and layers are independent in every stage."""
    import oracle
    from paper_2608_00531_gb300 import workload as W
    w = W.WORKLOADS[name]
    n_seq, n_attn, n_rs = CPU_SAMPLE.get(name, (2, 1, 2))
    B, K, N, V, k = w.batch, w.block, w.n_max, w.vocab, w.topk
    Hq, Hkv, D = w.heads_q, w.heads_kv, 128
    d = W.draft_block(w, batch=n_seq)
    L = W.cache_lengths(w)
    rng = np.random.default_rng(w.seed)
    x = W.bf16_to_f64(d.logits).reshape(n_seq, K, V)
    t0 = time.perf_counter()
    ids_all = np.zeros((n_seq, K, k), np.int64)
    m_all = np.zeros((n_seq, K), np.float32)
    for b in range(n_seq):
        ids, _, m, _, _ = oracle.score_draft(x[b], k)
        ids_all[b], m_all[b] = ids, m.astype(np.float32)
    t_score = time.perf_counter() - t0
    t0 = time.perf_counter()
    t = oracle.build_tree(ids_all, m_all, d.root_tok, L[:n_seq], w.tau, w.budget, w.branches, w.repair_depth,
                          d.redraft)
    t_tree = time.perf_counter() - t0
    # tree attention: n_attn sequence-layers with the configuration's cache
    # lengths and trees, N(0, 1) bf16 values as in the benchmark
    t_attn = 0.0
    for b in range(n_attn):
        Lb = int(L[b])
        kc = W.bf16_to_f64(W.normal_bf16((1, Lb, Hkv, D), 1.0, rng))
        vc = W.bf16_to_f64(W.normal_bf16((1, Lb, Hkv, D), 1.0, rng))
        q = W.bf16_to_f64(W.normal_bf16((1, N, Hq, D), 1.0, rng))
        tk = W.bf16_to_f64(W.normal_bf16((1, N, Hkv, D), 1.0, rng))
        tv = W.bf16_to_f64(W.normal_bf16((1, N, Hkv, D), 1.0, rng))
        t0 = time.perf_counter()
        oracle.tree_attn(q, tk, tv, kc, vc, np.array([Lb]), t["n_nodes"][b:b + 1], t["anc"][b:b + 1],
                         1.0 / math.sqrt(D))
        t_attn += time.perf_counter() - t0
    # target argmax and walk for the sampled sequences
    truth = W.target_truth(w, d)
    targ_ids = W.synthetic_target_ids(truth, t["n_nodes"], t["tok"], t["parent"], t["depth"], V, w.seed)
    tl = W.bf16_to_f64(W.target_logits(targ_ids, V, w.seed))
    t0 = time.perf_counter()
    targ = np.full((n_seq, N), -1, dtype=np.int64)
    for b in range(n_seq):
        targ[b, :t["n_nodes"][b]] = oracle.row_argmax(tl[b, :t["n_nodes"][b]])
    acc = oracle.accept(targ, t["n_nodes"], t["tok"], t["parent"], t["depth"], t["anc"], K)
    t_acc = time.perf_counter() - t0
    # resync of one layer for n_rs sequences
    cap = int(L[:n_rs].max()) + N
    kcs = [np.zeros((n_rs, cap, Hkv, D))]
    vcs = [np.zeros((n_rs, cap, Hkv, D))]
    trk = rng.standard_normal((1, n_rs, N, Hkv, D))
    t0 = time.perf_counter()
    oracle.resync(kcs, vcs, trk, trk, acc["path_nodes"][:n_rs], acc["accept_len"][:n_rs],
                  acc["diverge_depth"][:n_rs], acc["out_tokens"][:n_rs], L[:n_rs], K)
    t_rs = time.perf_counter() - t0
    stage = dict(score=t_score / n_seq * B, tree=t_tree / n_seq * B, attn=t_attn / n_attn * B * w.layers,
                 accept=t_acc / n_seq * B, resync=t_rs / n_rs * B * w.layers)
    per_step = sum(stage.values())
    sample = (f"oracle (numpy fp64, 1 thread) on a fixed sample of {name}: the first {n_seq} of {B} sequences "
              f"for the scan, tree, argmax and walk, {n_attn} sequence-layer(s) of tree attention and {n_rs} "
              f"sequence(s) of one layer's resync, with the configuration's shapes, cache lengths and trees; "
              f"extrapolated linearly to {B} sequences x {w.layers} layers")
    return dict(value=1.0 / per_step, unit="steps/s", cores=1, host_cores=os.cpu_count(), kind="oracle",
                sample=sample, seconds_per_step_extrapolated=per_step,
                stage_seconds={k_: round(v, 4) for k_, v in stage.items()})


# ------------------------------------------------------------------ main
def stage_roofs(alg, pk, w, Ly):
    """The roofline time of each stage (bytes / measured HBM peak), in us."""
    bw = pk["hbm_gbs"] * 1e9
    return {"vocab_scan_us": round(alg["scan_bytes"] / bw * 1e6, 2),
            "tree_attn_us_per_layer": round(max(alg["attn_bytes"] / bw,
                                                alg["attn_flops"] / (pk["bf16_tflops_sustained"] * 1e12)) * 1e6, 2),
            "target_argmax_us": round(alg["argmax_bytes"] / bw * 1e6, 2)}


def timed_steps(st, xs, kcs, vcs, steps, stream, world, dev, events=True):
    """`steps` steps cycling over the input sets; returns the total device ms
    and, with `events`, the per-stage ms from an event pair around each stage
    group (an event between two launches keeps the second from starting its
    set-up under the first, so the step's own time is taken without them)."""
    from paper_2608_00531_gb300 import cure
    P = len(xs)
    Ly = st.layers
    names = ("scan", "tree", "attn", "accept", "resync")
    ev = {k_: [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(steps)] for k_ in names}

    def mark(k_, s, i):
        if events:
            ev[k_][s][i].record(stream)

    def one(s):
        x = xs[s % P]
        mark("scan", s, 0)
        cure.cure_score_draft(x.draft_logits, st.k, out=st.score)
        mark("scan", s, 1)
        mark("tree", s, 0)
        tree = cure.cure_build_tree(st.score[0], st.score[2], x.root_tok, x.cache_len, st.tau, st.R,
                                    st.branches, st.depth, x.redraft, st.max_ufp, out=st.tree)
        mark("tree", s, 1)
        # one event pair around the step's attention launches (events between
        # the launches would stop each from starting its set-up under the
        # previous one, which it does as a programmatic dependent launch)
        mark("attn", s, 0)
        for l in range(Ly):
            p_ = st.layer_map[l]
            cure.cure_tree_attn(x.q[l], x.tree_k[l], x.tree_v[l], kcs[p_], vcs[p_], st.kv, x.cache_len,
                                tree["n_nodes"], tree["anc"], st.scale, out=st.attn_out[l],
                                workspace=st.workspace)
        mark("attn", s, 1)
        mark("accept", s, 0)
        acc = cure.cure_accept(tree, st.K, target_logits=x.target_logits, targ=st.targ, out=st.acc)
        mark("accept", s, 1)
        mark("resync", s, 0)
        kl = [kcs[st.layer_map[l]] for l in range(Ly)]
        vl = [vcs[st.layer_map[l]] for l in range(Ly)]
        cure.cure_resync_kv(kl, vl, st.kv, x.tree_k, x.tree_v, acc, x.cache_len, st.K,
                            cache_len_out=st.cache_len_out, out=st.rs)
        mark("resync", s, 1)

    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for s in range(steps):
        one(s)
    t1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(t0.elapsed_time(t1), world, dev)
    per = None
    if events:
        per = {k_: float(np.mean([ev[k_][s][0].elapsed_time(ev[k_][s][1]) for s in range(steps)])) for k_ in names}
        per["attn"] /= Ly
    return ms, per


def warm(st, xs, kcs, vcs, n):
    """n untimed steps; the accept lengths of each input set."""
    from paper_2608_00531_gb300 import cure
    P = len(xs)
    acc_lens = [None] * P
    for i in range(max(n, P)):
        r = st.run(xs[i % P], kcs, vcs)
        torch.cuda.synchronize()
        acc_lens[i % P] = r["acc"]["accept_len"].cpu().numpy()
    assert cure.cure_device_error() == 0
    return acc_lens


def sweep_points(wl, dev, steps, warmup, world, rank):
    """The (R, tau) grid on the sweep configuration: per point its own trees
    and targets (two input sets), steps/s and the mean accepted length.  At
    R = 0 the tree is the draft chain alone, and the accepted lengths must
    equal plain prefix verification of the chain against the target's tokens
    (checked here on the device's own outputs)."""
    out = []
    stream = torch.cuda.current_stream()
    for R in (0, 4, 8, 16, 32, 64):
        for tau in (0.25, 0.5, 1.0, 2.0, 4.0):
            p = make_workload(dev, rank, wl["w"].name, pool=2, caches=wl["caches"], tau=tau, budget=R)
            st, xs = p["st"], p["xs"]
            acc_lens = warm(st, xs, p["kcs"], p["vcs"], warmup)
            prefix_ok = None
            if R == 0:
                prefix_ok = True
                for i, x in enumerate(xs):
                    st.run(x, p["kcs"], p["vcs"])
                    torch.cuda.synchronize()
                    tok = st.tree["tok"].cpu().numpy()
                    targ = st.targ.cpu().numpy()
                    a = st.acc["accept_len"].cpu().numpy()
                    K = st.K
                    for b in range(st.B):
                        e = 0
                        while e < K and tok[b, e + 1] == targ[b, e]:
                            e += 1
                        prefix_ok &= bool(a[b] == e)
            ms, _ = timed_steps(st, xs, p["kcs"], p["vcs"], steps, stream, world, dev, events=False)
            _, per = timed_steps(st, xs, p["kcs"], p["vcs"], steps, stream, world, dev)
            algs = [algorithmic(p, th) for th in p["trees"]]
            out.append({"budget": R, "tau": tau, "steps_per_s": round(job_steps_per_s(ms, steps, world), 2),
                        "ms_per_step": round(ms / steps, 4),
                        "mean_accept_len": round(float(np.mean([a_.mean() for a_ in acc_lens])), 3),
                        "mean_tree_nodes": round(float(np.mean([a_["mean_nodes"] for a_ in algs])), 2),
                        "tree_attn_ms_per_layer": round(per["attn"], 4),
                        "r0_equals_prefix_verification": prefix_ok})
            del p, st, xs
            torch.cuda.empty_cache()
    return out


def profile_stage(args):
    """Runs one stage alone on the configuration's shapes, `--steps` calls
    after `--warmup`, and prints nothing: the command an ncu capture of that
    stage's kernel wraps (a few GB on the device at most)."""
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import cure, workload as W
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = W.WORKLOADS[args.workload]
    g = torch.Generator(device=dev).manual_seed(7)
    name = args.profile_stage
    if name == "lm_head":
        rows = int(round(w.batch * (w.block + 1 + 0.55 * w.budget)))   # about the realised tree nodes
        d_model = D_MODEL[w.name]
        wl = (torch.randn(w.vocab, d_model, generator=g, device=dev) * d_model ** -0.5).to(torch.bfloat16)
        h = torch.randn(rows, d_model, generator=g, device=dev).to(torch.bfloat16)
        out = torch.empty(rows, dtype=torch.int32, device=dev)
        ws = torch.empty(max(256, cure.cure_lm_head_workspace_size(rows, w.vocab)), dtype=torch.uint8, device=dev)
        fn = lambda: cure.cure_lm_head_argmax(h, wl, out=out, workspace=ws)  # noqa: E731
    elif name in ("sample", "argmax"):
        B, N = w.batch, w.n_max
        tl = torch.randn(B, N, w.vocab, generator=g, device=dev).to(torch.bfloat16)
        n = torch.full((B,), N, dtype=torch.int32, device=dev)
        uni = torch.rand(B, N, generator=g, device=dev)
        targ = torch.empty(B, N, dtype=torch.int32, device=dev)
        if name == "sample":
            fn = lambda: cure.cure_sample_target(tl, n, uni, 0.8, out=targ)  # noqa: E731
        else:
            tree = dict(n_nodes=n, tok=torch.zeros(B, N, dtype=torch.int32, device=dev),
                        parent=torch.zeros(B, N, dtype=torch.int32, device=dev),
                        depth=torch.zeros(B, N, dtype=torch.int32, device=dev),
                        anc=torch.ones(B, N, (N + 63) // 64, dtype=torch.int64, device=dev))
            fn = lambda: cure.cure_accept(tree, w.block, target_logits=tl, targ=targ)  # noqa: E731
    elif name == "scan":
        x = W.draft_block(w).logits.to(dev)
        fn = lambda: cure.cure_score_draft(x, w.topk)  # noqa: E731
    else:
        raise SystemExit(f"unknown stage {name}")
    for _ in range(args.warmup + args.steps):
        fn()
    torch.cuda.synchronize()
    assert cure.cure_device_error() == 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD,
                    choices=["tiny", "single8b", "serve32", "long64", "sweep16"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--layers", type=int, default=None, help=argparse.SUPPRESS)
    ap.add_argument("--profile-stage", default=None, choices=["lm_head", "sample", "argmax", "scan"],
                    help="run one stage alone (for a profiler capture) and print nothing")
    args = ap.parse_args()
    if args.profile_stage:
        profile_stage(args)
        return
    args.warmup = max(3, args.warmup)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return
        run_reference(args)
        return

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_00531_gb300 import cure

    wl = make_workload(dev, rank, args.workload, args.layers)
    w = wl["w"]
    st, xs, kcs, vcs = wl["st"], wl["xs"], wl["kcs"], wl["vcs"]
    P = len(xs)
    stream = torch.cuda.current_stream()
    Ly = wl["layers"]

    acc_lens = warm(st, xs, kcs, vcs, args.warmup)
    algs = [algorithmic(wl, th) for th in wl["trees"]]
    # the timed steps cycle over the sets: per-step averages
    sel = [s % P for s in range(args.steps)]
    alg = {k_: float(np.mean([algs[i][k_] for i in sel])) for k_ in algs[0]}

    clk = ClockSampler(local)
    clk.start()
    with quiet_host():
        clk.mark_start()
        ms, _ = timed_steps(st, xs, kcs, vcs, args.steps, stream, world, dev, events=False)
        clk.mark_stop()
    clocks = clk.stop()
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    assert cure.cure_device_error() == 0
    # the per-stage times from a second pass of the same steps, with an event
    # pair around each stage group
    with quiet_host():
        _, per = timed_steps(st, xs, kcs, vcs, args.steps, stream, world, dev)
    attn_avg, scan_avg, acc_avg, rs_ms = per["attn"], per["scan"], per["accept"], per["resync"]
    rs_b = float(np.mean([resync_bytes(acc_lens[i], Ly, w.heads_kv) for i in sel]))

    # the same step replayed as CUDA graphs (one per input set), timed the same way
    graph = None
    rs_graph_ms = scan_graph_ms = acc_graph_ms = sample_graph_ms = None
    if not args.no_graph:
        with quiet_host():
            graph = run_graphs(st, xs, kcs, vcs, args.steps, world, dev)
        xl = xs[sel[-1]]
        rs_graph_ms = resync_graph_ms(st, xl, kcs, vcs)
        scan_graph_ms = call_graph_ms(lambda: cure.cure_score_draft(xl.draft_logits, st.k, out=st.score))
        acc_graph_ms = call_graph_ms(lambda: cure.cure_accept(st.tree, st.K, target_logits=xl.target_logits,
                                                               targ=st.targ, out=st.acc))
        # stochastic verification on the same rows: the target's token sampled
        # per node at T = 0.8 with seeded uniforms
        uni = torch.rand(st.B, st.n_max, generator=torch.Generator(device=dev).manual_seed(5), device=dev)
        samp_out = torch.empty(st.B, st.n_max, dtype=torch.int32, device=dev)
        sample_graph_ms = call_graph_ms(lambda: cure.cure_sample_target(xl.target_logits, st.tree["n_nodes"], uni,
                                                                       0.8, out=samp_out))
        # the walk after each call (graph-replayed) reads st.tree: restore the last set's tree
        st.run(xl, kcs, vcs)
        torch.cuda.synchronize()

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        with quiet_host():
            e2e = run_e2e(wl, st, kcs, vcs, dev, max(3, min(args.steps, 10)), world)

    # the in-place tree-KV layout on the same shapes; last, since its resync
    # moves rows inside the caches
    in_place = None
    if not args.no_graph:
        in_place = in_place_stage(st, xs[sel[-1]], kcs, vcs)

    pk = peaks()
    lm_head = None
    if not args.no_graph:
        lm_head = lm_head_stage(int(round(alg["mean_nodes"] * st.B)), st.V, dev, pk, D_MODEL[w.name])

    sweep = None
    if w.name == "sweep16" and not args.no_sweep:
        sweep = sweep_points(wl, dev, max(3, min(args.steps, 10)), args.warmup, world, rank)

    if rank != 0:
        return
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
    traffic = ATTN_TRAFFIC.get(attn_source_digest()) if w.name == DEFAULT_WORKLOAD else None
    roof.update({"traffic": traffic,
                 "traffic_source": "ncu dram__bytes_read.sum + dram__bytes_write.sum of this kernel source "
                                   "(one layer of the serving workload); null when the source has changed or for "
                                   "another workload",
                 "kernel": f"tree attention (tree_attn_tc_kernel, persistent, split units merged in-kernel), per "
                           f"layer: the step's {Ly} back-to-back launches timed together, divided by {Ly}",
                 "algorithmic_bytes_per_launch": alg["attn_bytes"],
                 "algorithmic_flops_per_launch": alg["attn_flops"], "avg_launch_ms": round(attn_avg, 4),
                 "peak_source": pk["source"] + (" (MEASURED_PEAKS.json hbm_gbs)" if bound == "hbm" else
                                                " (MEASURED_PEAKS.json bf16_tflops_sustained)")})
    big = alg["attn_bytes"] * Ly > 2 * 129e6
    out = {
        "metric": metric_for(w), "value": round(value, 3), "unit": "steps/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": workload_text(w, Ly, wl["phys"]),
                   "batch": w.batch, "block": w.block, "vocab": w.vocab, "tau": w.tau, "budget": w.budget,
                   "branches": w.branches, "repair_depth": w.repair_depth, "layers": Ly,
                   "physical_cache_layers": wl["phys"], "heads_q": w.heads_q, "heads_kv": w.heads_kv,
                   "head_dim": 128, "paged": w.paged, "per_gpu_batch": w.batch,
                   "l2": ("no flush: inputs larger than L2 (KV read per step %.1f GB)" % (alg["attn_bytes"] * Ly / 1e9))
                   if big else ("no flush: a latency-bound configuration whose step reads %.1f MB; its stages are "
                                "reported in us beside their roofline time" % (alg["attn_bytes"] * Ly / 1e6))},
        "roofline": roof,
        "stages": {"vocab_scan_ms": round(scan_avg, 4), "vocab_scan_gbs": round(scan_gbs, 1),
                   "vocab_scan_graph_ms": None if scan_graph_ms is None else round(scan_graph_ms, 4),
                   "vocab_scan_graph_frac": None if scan_graph_ms is None else
                   round(alg["scan_bytes"] / (scan_graph_ms * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                   "vocab_scan_frac": round(scan_gbs / pk["hbm_gbs"], 4),
                   "build_tree_ms": round(per["tree"], 4),
                   "resync_call_ms": round(rs_ms, 4),
                   "resync_call_gbs": round(rs_b / (rs_ms * 1e-3) / 1e9, 1),
                   "resync_call_frac": round(rs_b / (rs_ms * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                   "resync_graph_ms": None if rs_graph_ms is None else round(rs_graph_ms, 4),
                   "resync_graph_frac": None if rs_graph_ms is None else
                   round(resync_bytes(acc_lens[sel[-1]], Ly, w.heads_kv) / (rs_graph_ms * 1e-3) / 1e9
                         / pk["hbm_gbs"], 4),
                   "target_argmax_accept_ms": round(acc_avg, 4),
                   "target_argmax_accept_frac": round(alg["argmax_bytes"] / (acc_avg * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                   "target_argmax_accept_graph_ms": None if acc_graph_ms is None else round(acc_graph_ms, 4),
                   "target_argmax_accept_graph_frac": None if acc_graph_ms is None else
                   round(algs[sel[-1]]["argmax_bytes"] / (acc_graph_ms * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                   "target_argmax_bytes": int(alg["argmax_bytes"]),
                   "sample_target_graph_ms": None if sample_graph_ms is None else round(sample_graph_ms, 4),
                   "sample_target_graph_frac": None if sample_graph_ms is None else
                   round(algs[sel[-1]]["argmax_bytes"] / (sample_graph_ms * 1e-3) / 1e9 / pk["hbm_gbs"], 4),
                   "tree_attn_ms_per_layer": round(attn_avg, 4),
                   "tree_attn_tflops": round(attn_tflops, 1), "tree_attn_gbs": round(attn_gbs, 1),
                   "tree_attn_intensity_flop_per_byte": round(intensity, 1),
                   "roofline_us": stage_roofs(alg, pk, w, Ly),
                   "mean_tree_nodes": round(alg["mean_nodes"], 3),
                   "mean_accept_len": round(float(np.mean([acc_lens[i].mean() for i in sel])), 3),
                   "input_sets": P, "in_place": in_place, "lm_head_argmax": lm_head},
        "gpu_launches": st.launches_per_step * args.steps,
        "clocks": clocks,
    }
    if e2e:
        out["e2e"] = e2e
    if graph:
        out["graph"] = graph
    if sweep is not None:
        out["sweep"] = sweep
    if not args.no_cpu_baseline and world == 1:
        out["cpu_baseline"] = cpu_baseline(w.name)
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


def lm_head_stage(rows, vocab, dev, pk, d_model=4096):
    """The fused LM head + argmax (the target's greedy token per node straight
    from its final hidden state) on the step's realised tree nodes, timed alone
    (graph-replayed calls), against the tensor peak; beside it, the unfused
    alternative's contraction alone (a cuBLAS GEMM writing the bf16 logits),
    which the argmax scan would then read.  Random weight and hidden states:
    timings, not results."""
    try:
        from paper_2608_00531_gb300 import cure
        g = torch.Generator(device=dev).manual_seed(99)
        w = (torch.randn(vocab, d_model, generator=g, device=dev) * d_model ** -0.5).to(torch.bfloat16)
        h = torch.randn(rows, d_model, generator=g, device=dev).to(torch.bfloat16)
        out = torch.empty(rows, dtype=torch.int32, device=dev)
        ws = torch.empty(max(256, cure.cure_lm_head_workspace_size(rows, vocab)), dtype=torch.uint8, device=dev)
        fused = call_graph_ms(lambda: cure.cure_lm_head_argmax(h, w, out=out, workspace=ws), calls=5, reps=4)
        logits = torch.empty(rows, vocab, dtype=torch.bfloat16, device=dev)
        gemm = call_graph_ms(lambda: torch.matmul(h, w.t(), out=logits), calls=5, reps=4)
        flops = 2.0 * rows * vocab * d_model
        if cure.cure_device_error() != 0:
            return None
        del w, logits
        return {"rows": rows, "d_model": d_model, "vocab": vocab,
                "fused_ms": None if fused is None else round(fused, 4),
                "fused_tflops": None if fused is None else round(flops / (fused * 1e-3) / 1e12, 1),
                "fused_frac": None if fused is None else round(flops / (fused * 1e-3) / 1e12 / pk["bf16_tflops"], 4),
                "cublas_gemm_ms": None if gemm is None else round(gemm, 4),
                "cublas_gemm_tflops": None if gemm is None else round(flops / (gemm * 1e-3) / 1e12, 1),
                "peak": pk["bf16_tflops"], "peak_note": "bf16 burst (kernel timed alone), " + pk["source"],
                "note": "fused = tcgen05 contraction with the argmax in its epilogue + per-row merge; the logits "
                        "are never written. cublas_gemm = the unfused path's contraction alone (bf16 logits "
                        "written, argmax scan not included)"}
    except Exception as e:  # reported as missing, the bench line stands
        print(f"lm head timing failed: {type(e).__name__}: {e}"[:300], file=sys.stderr)
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
        kl = [kcs[st.layer_map[l]] for l in range(st.layers)]
        vl = [vcs[st.layer_map[l]] for l in range(st.layers)]

        def call():
            cure.cure_resync_kv(kl, vl, st.kv, x.tree_k, x.tree_v, acc, x.cache_len, st.K,
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
    fields = ("draft_logits", "root_tok", "cache_len", "q", "tree_k", "tree_v", "target_logits")
    if x.redraft is not None:
        fields += ("redraft",)
    host = {k_: getattr(x, k_).cpu().pin_memory() for k_ in fields}
    outs = torch.empty(4, st.B, st.K + 2, dtype=torch.int32).pin_memory()
    d2h = outs.numel() * outs.element_size() + (st.B * 4 if x.target_logits.numel() * 2 >= st.NODE_ROWS_MIN_BYTES else 0)  # results; node counts read mid-step
    h2d_steps = []
    stream = torch.cuda.current_stream()
    xh = StepInputs(host["draft_logits"], host["root_tok"], host["cache_len"], host.get("redraft"), host["q"],
                    host["tree_k"], host["tree_v"], host["target_logits"])

    def one():
        # the public step with host inputs: it streams them in on a copy
        # stream, each stage waiting for its own inputs
        r = st.run_from_host(xh, kcs, vcs)
        h2d_steps.append(st.last_h2d_bytes)
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
    h2d = float(np.mean(h2d_steps[-steps:]))
    return {"value": round(job_steps_per_s(ms * steps, steps, world), 3), "unit": "steps/s", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "ms_per_step": round(ms, 4), "steps": steps}


def run_reference(args):
    """The reference arm: the oracle (the paper's method restated on the CPU),
    timed as it stands on one host core, each step the same fixed sample of
    the workload extrapolated to a full step (as the repo arm's cpu_baseline)."""
    from paper_2608_00531_gb300 import workload as W
    w = W.WORKLOADS[args.workload]
    vals = []
    cb = None
    for i in range(args.warmup + args.steps):
        cb = cpu_baseline(args.workload)
        if i >= args.warmup:
            vals.append(cb["seconds_per_step_extrapolated"])
    sec = float(np.mean(vals))
    v = 1.0 / sec
    out = {"impl": "reference", "metric": metric_for(w), "value": v, "unit": "steps/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": workload_text(w, w.layers, w.layers)},
           "cpu_baseline": {"value": v, "unit": "steps/s", "cores": 1, "host_cores": os.cpu_count(),
                            "kind": "oracle", "sample": cb["sample"]},
           "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
