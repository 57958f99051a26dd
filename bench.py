#!/usr/bin/env python
"""Throughput of true-tail memory maintenance rounds on one GB300 per rank.

A step is one maintenance round (every hot-path row): removal of superseded KV
by compaction in every attention layer, then every layer in model order
(RoPE at the true tail + cache append + causal GQA attention for attention
layers; chunked gated delta rule from the carried state for recurrent
layers), then the cursor advance.  Default workload ("long", the largest
single-GPU configuration): 48 layers in a 3:1 delta:attention pattern (delta
16 heads, d_k = d_v = 128; attention 16 query / 2 KV heads, head_dim 256,
RoPE on 64 dims), a 32768-token prefix built by a GPU refill, one round
removing 3% of the entries in 10 spans and appending 1024 tail tokens.
`--workload npc|pop|refill|tiny` selects the other configurations.  Steps
cycle through the workload's chain of rounds; before round 0 of each chain
the working state is forked from the prefix root and before every step L2 is
flushed (a 256 MiB write), both outside the timed events.

Prints one JSON line (rank 0).  `--impl reference` times the fp64 CPU oracle
on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from workload import synth as W  # noqa: E402

# tail tokens per step of the reference arm and of the cpu_baseline sample
# (one hybrid block of character 0's round 0): a reference step takes a few
# seconds, the cpu_baseline sample 10-30 s on 16 cores
REFERENCE_TOKENS = {"tiny": 16, "npc": 8, "long": 4, "pop": 8, "refill": 8}
CPU_BASELINE_TOKENS = {"tiny": 64, "npc": 96, "long": 48, "pop": 96, "refill": 64}
METRIC = "tail tokens/sec per maintenance round and ms/round; % of HBM/tensor roofline"
UNIT = "tail tokens/s"
EVENT_POOL = 4096     # launches the library can time between two reads (kvm_profile_read)

WORKLOAD_TEXT = {
    "tiny": "1 delta-rule (8 heads, d 64) + 1 GQA attention layer (8/2 heads, D 64, RoPE 64), prefix 512, "
            "2 spans totalling 64 removed, tail 64, one round",
    "npc": "NPC context: 4 layers 3:1 (delta 16 heads d_k=d_v=128; attention 16 Q / 2 KV heads, D 256, "
           "partial RoPE 64 dims), prefix 8192, 8 chained rounds, 1-4 spans ~5% removed, tail 256 per round",
    "long": "long-lived character: 48 layers 3:1 (npc shapes), prefix 32768, 10 spans = 3% removed, tail 1024",
    "pop": "population: 32 characters varlen-packed, prefixes U[2048,16384], 2-8% removed in 1-6 spans, "
           "tails U[64,512], 12 layers 3:1 (npc shapes)",
    "refill": "npc stack, no removals, prefix 16384 + tail 512 as a tail update",
}


# ----------------------------------------------------------------------------
# accounting (algorithmic work per round)
# ----------------------------------------------------------------------------
def attention_flops(shape, Lp, tails):
    """4 D Hq (M L' + M (M+1)/2) per attention layer, summed over characters."""
    D, Hq = shape.head_dim, shape.n_q_heads
    return sum(4.0 * D * Hq * (m * l + m * (m + 1) / 2) for l, m in zip(Lp, tails))


def attention_bytes(shape, Lp, tails):
    """K and V of the surviving keys once per KV head, q, k_new and v_new of
    the tail, and the output, per attention layer."""
    Hq, Hkv, D = shape.n_q_heads, shape.n_kv_heads, shape.head_dim
    return float(sum(l for l, m in zip(Lp, tails) if m > 0) * Hkv * D * 2 * 2
                 + sum(tails) * (2 * Hq + 2 * Hkv) * D * 2)


def gdn_flops(shape, tails):
    return 6.0 * shape.d_k * shape.d_v * shape.n_gdn_heads * sum(tails)


def gdn_bytes(shape, tails):
    """q, k, v, o (bf16) and alpha, beta (fp32) of every tail token and head,
    plus the state read and written once per character and head."""
    H, dk, dv = shape.n_gdn_heads, shape.d_k, shape.d_v
    per_tok = H * ((2 * dk + 2 * dv) * 2 + 8)
    return float(sum(tails) * per_tok + sum(1 for m in tails if m > 0) * H * dv * dk * 4 * 2)


def rope_bytes(shape, tails):
    """Read q, k, v of the tail; write the rotated q (staging), k and v."""
    Hq, Hkv, D = shape.n_q_heads, shape.n_kv_heads, shape.head_dim
    return float(sum(tails) * (Hq + 2 * Hkv) * D * 2 * 2)


def compaction_bytes(shape, moved_rows):
    n_attn = len(shape.attn_layers)
    row = shape.n_kv_heads * shape.head_dim * 2 * 2 * n_attn + 4     # K and V of every layer + position
    return 2.0 * moved_rows * row


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def ncu_traffic(kernel_file: str, kernel: str):
    """dram bytes per launch from a committed ncu summary, if it was taken on
    the current source of the kernel (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)[kernel]
        src = open(os.path.join(ROOT, "paper_2609_18935_gb300", "csrc", kernel_file), "rb").read()
        if hashlib.sha256(src).hexdigest() != d["src_sha256"]:
            return None
        return d["bytes_per_launch"]
    except Exception:
        return None


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.samples = []          # (t, sm, max, reasons set)
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm, mx = float(parts[1]), float(parts[2])
            except ValueError:
                continue
            reasons = {n for n, v in zip(names, parts[5:9]) if v.lower().startswith("active")}
            self.samples.append((time.time(), sm, mx, reasons))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0, t1):
        inside = [s for s in self.samples if t0 <= s[0] <= t1]
        window = "timed"
        if not inside:                      # region shorter than the sampling period
            inside = [s for s in self.samples if t0 - 1.0 <= s[0] <= t1 + 0.25]
            window = "timed +/- sampling period"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0, "window": "none"}
        reasons = sorted(set().union(*[s[3] for s in inside]))
        return {"sm_mhz": statistics.median(s[1] for s in inside), "sm_max_mhz": max(s[2] for s in inside),
                "reasons": reasons, "samples": len(inside), "window": window}


# ----------------------------------------------------------------------------
# CPU oracle sample (cpu_baseline leg and the reference arm)
# ----------------------------------------------------------------------------
def oracle_block(w):
    """Layers of the CPU sample: the first hybrid block of the stack (three
    delta-rule layers and one attention layer in the 3:1 pattern; the whole
    stack when it is shorter), and how many such blocks the stack has."""
    kinds = w.shape.layer_kind
    n = min(4, len(kinds))
    return list(range(n)), len(kinds) / n


def oracle_state(w):
    """The fp64 oracle's state of character 0 before round 0, restricted to
    the sample's layers (prefix cache and recurrent states as the GPU arm
    draws them)."""
    from oracle import kvm_oracle as O
    s = w.shape
    N = w.prefix_len[0]
    layers, _ = oracle_block(w)
    caches, states = {}, {}
    for l in layers:
        if s.layer_kind[l] == W.ATTN:
            K, V, pos = W.prefix_cache(w, 0, l, N)
            caches[l] = O.AttnCache(O.bf16_to_f64(K), O.bf16_to_f64(V), pos)
        else:
            states[l] = O.f32_to_f64(W.prefix_state(w, 0, l))
    return O.CharacterState(caches, states, N)


def oracle_sample(w, st, m_sample: int):
    """Time the fp64 oracle on round 0 of character 0 for the sample's layers
    (oracle_block), restricted to the first m_sample tail tokens: compaction
    of the block's attention layer, then every layer of the block.  Returns
    (seconds, tail tokens, blocks in the stack): the whole stack takes about
    `blocks` times as long, since its blocks have the same shapes."""
    from oracle import kvm_oracle as O
    s = w.shape
    N = w.prefix_len[0]
    layers, blocks = oracle_block(w)
    cu, sb, se, tails = W.round_plan(w, 0, [N] + [0] * (w.n_chars - 1))
    m = min(m_sample, tails[0])
    full = W.tail_inputs(w, 0, [m], layers=layers)
    ins = {}
    for l in layers:
        ins[l] = {k: (O.bf16_to_f64(v) if v.dtype == np.uint16 else O.f32_to_f64(v)) for k, v in full[l].items()}
    kinds = [s.layer_kind[l] for l in layers]
    t0 = time.perf_counter()
    O.maintenance_round(st, kinds, sb[cu[0]:cu[1]], se[cu[0]:cu[1]], ins, s.rotary_dim, s.rope_theta)
    return time.perf_counter() - t0, m, blocks


def sample_text(w, m, secs=None):
    layers, blocks = oracle_block(w)
    txt = (f"character 0, round 0 of the workload (prefix {w.prefix_len[0]}): compaction + layers "
           f"{layers[0]}-{layers[-1]} (one 3:1 hybrid block) for the first {m} tail tokens, fp64 numpy; "
           f"tokens/s scaled to the {len(w.shape.layer_kind)}-layer stack by its {blocks:g} blocks of the "
           f"same shapes")
    return txt + (f"; {secs:.1f} s" if secs is not None else "")


def blas_threads() -> int:
    try:
        from threadpoolctl import threadpool_info
        n = [d.get("num_threads", 0) for d in threadpool_info() if d.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count() or 1


# ----------------------------------------------------------------------------
# ranks (one process per GPU; replicas maintain different characters)
# ----------------------------------------------------------------------------
def dist_env():
    """(rank, world size, local rank) from the launcher's environment."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def replica_seed(rank: int) -> int:
    """Seed base of a rank's characters: every rank maintains its own."""
    return 7919 * (rank + 1)


def rank_share(w, rank: int, world: int):
    """The characters rank `rank` maintains.  A population (several
    characters) is partitioned over the ranks by kvm_plan_partition, balanced
    by each character's round-0 attention work M (L' + (M + 1) / 2); the
    ranks need no exchange on the data path, and the job's total work stays
    fixed as ranks are added (strong scaling).  A single character cannot be
    split: every rank maintains its own replica (weak scaling).
    Returns (workload of this rank, scaling)."""
    if world <= 1 or w.n_chars <= 1:
        return w, "weak"
    from paper_2609_18935_gb300 import kvm
    cu, sb, se, tails = W.round_plan(w, 0, list(w.prefix_len))
    after = [w.prefix_len[b] - int((se[cu[b]:cu[b + 1]] - sb[cu[b]:cu[b + 1]]).sum()) for b in range(w.n_chars)]
    rank_of, _ = kvm.plan_partition(kvm.round_cost(after, tails), world)
    return w.subset([b for b in range(w.n_chars) if rank_of[b] == rank]), "strong"


def max_over_ranks(x: float, world: int, device="cpu") -> float:
    """The job's time is the slowest rank's (all_reduce MAX); x itself on one rank."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: float, world: int, device="cpu") -> float:
    """Sum of x over the ranks (all_reduce SUM); x itself on one rank."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def job_throughput(world: int, tokens_per_rank: float, ms: float) -> float:
    """Whole-job tail tokens/s: every rank processes tokens_per_rank in the
    job's time (the slowest rank's) of ms milliseconds."""
    return world * tokens_per_rank / (ms / 1e3)


def workload_config(w, args, world):
    s = w.shape
    full = W.make_workload(args.workload, args.layers)
    if world > 1 and full.n_chars > 1:
        par = f"population of {full.n_chars} characters partitioned over {world} ranks (balanced by M L')"
    else:
        par = f"{world} independent replica(s), characters per rank fixed"
    text = WORKLOAD_TEXT[args.workload]
    if args.layers:
        text += f" (shortened to {len(s.layer_kind)} layers for a profiling capture)"
    return {"workload": text, "name": args.workload, "chars": full.n_chars,
            "layers": len(s.layer_kind), "chain_rounds": w.rounds,
            "l2": "flushed before every step (256 MiB write), outside the timed events",
            "parallelism": par}


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    w = W.make_workload(args.workload, args.layers)
    m = REFERENCE_TOKENS[args.workload]
    st = oracle_state(w)
    for _ in range(args.warmup):
        oracle_sample(w, st, m)
    secs, toks = 0.0, 0
    for _ in range(args.steps):
        t, n, blocks = oracle_sample(w, st, m)
        secs += t * blocks
        toks += n
    value = toks / secs
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(w, args, world),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
                             "sample": "each step: " + sample_text(w, m)},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------
# GPU arm
# ----------------------------------------------------------------------------
def from_scratch_prefill(w, plan, mk, flush, args, seed_base):
    """The refill workload's other arm: the text of round 0 (prefix + tail)
    computed from an empty cache and zero states in one round, the dense
    refill that the tail update avoids (§5.2).  Median device time of
    max(3, min(16, steps / 8)) runs after `warmup` untimed ones; before each run the
    context is reset by a fork of an empty one and L2 is flushed, both
    outside the timed events."""
    import torch
    s = w.shape
    n_all = [a + b for a, b in zip(w.prefix_len, plan[0][3])]
    tot = sum(n_all)
    empty, fresh = mk(tot), mk(tot)
    ins = W.device_round_inputs(w, seed_base + 7777, n_all)
    outs = {l: torch.empty((tot, s.n_q_heads, s.head_dim) if k == W.ATTN else (tot, s.n_gdn_heads, s.d_v),
                           dtype=torch.bfloat16, device="cuda") for l, k in enumerate(s.layer_kind)}
    zero_cu = np.zeros(w.n_chars + 1, np.int32)
    cu_all = np.concatenate([[0], np.cumsum(n_all)]).astype(np.int32)
    stream = torch.cuda.current_stream()
    evs = []
    for i in range(args.warmup + max(3, min(16, args.steps // 8))):
        fresh.fork_from(empty)
        flush.fill_(i & 0x7F)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        fresh.update_round(zero_cu, [], [], cu_all, ins, outs)
        e1.record(stream)
        if i >= args.warmup:
            evs.append((e0, e1))
    torch.cuda.synchronize()
    fresh.check()
    ms = float(np.median([a.elapsed_time(b) for a, b in evs]))
    del ins, outs, empty, fresh
    torch.cuda.empty_cache()
    return {"what": "the same text as a from-scratch prefill: empty cache, zero states, one round",
            "tokens": tot, "ms": ms, "runs": len(evs)}


def run_kvm(args):
    import torch
    import torch.distributed as dist
    from paper_2609_18935_gb300 import build_lib, kvm

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if not os.path.exists(kvm.LIB_PATH):
        if rank == 0:
            build_lib.build()
        if world > 1:
            dist.barrier()
    kvm.load_library()

    w, scaling = rank_share(W.make_workload(args.workload, args.layers), rank, world)
    s = w.shape
    plan = W.simulate_plan(w)
    R = len(plan)
    caps = w.capacity()
    mk = lambda max_tail: kvm.Context(s.layer_kind, s.n_q_heads, s.n_kv_heads, s.head_dim, s.rotary_dim,
                                      s.rope_theta, s.n_gdn_heads, s.d_k, s.d_v, caps, max_tail)
    seed_base = replica_seed(rank)

    # ---- prefix root: a GPU refill of the prefix (no removals, tail = prefix)
    N = list(w.prefix_len)
    root = mk(sum(N))
    ins = W.device_round_inputs(w, seed_base, N)
    tot = sum(N)
    outs = {l: torch.empty((tot, s.n_q_heads, s.head_dim) if k == W.ATTN else (tot, s.n_gdn_heads, s.d_v),
                           dtype=torch.bfloat16, device="cuda") for l, k in enumerate(s.layer_kind)}
    zero_cu = np.zeros(w.n_chars + 1, np.int32)
    root.update_round(zero_cu, [], [], np.concatenate([[0], np.cumsum(N)]), ins, outs)
    root.check()
    del ins, outs
    torch.cuda.empty_cache()

    # ---- per-round inputs (device) and their pinned host copies (end to end)
    max_tail = max(sum(p[3]) for p in plan)
    work = mk(max_tail)
    rounds = []
    for r, (cu, sb, se, tails) in enumerate(plan):
        tail_cu = np.concatenate([[0], np.cumsum(tails)]).astype(np.int32)
        d_in = W.device_round_inputs(w, seed_base + 1 + r, tails)
        tot = int(tail_cu[-1])
        d_out = {l: torch.empty((tot, s.n_q_heads, s.head_dim) if k == W.ATTN else (tot, s.n_gdn_heads, s.d_v),
                                dtype=torch.bfloat16, device="cuda") for l, k in enumerate(s.layer_kind)}
        h_in = kvm.pinned_layer_inputs(d_in)              # one pinned arena per layer
        h_out = {l: torch.empty(o.shape, dtype=o.dtype).pin_memory() for l, o in d_out.items()}
        rounds.append(dict(cu=cu, sb=sb, se=se, tails=tails, tail_cu=tail_cu, d_in=d_in, d_out=d_out,
                           h_in=h_in, h_out=h_out))
    # per-round algorithmic work (live lengths follow the plan from the prefix)
    live = list(N)
    for rd in rounds:
        cu, sb, se, tails = rd["cu"], rd["sb"], rd["se"], rd["tails"]
        Lp, moved = [], 0
        for b in range(w.n_chars):
            rem = int((se[cu[b]:cu[b + 1]] - sb[cu[b]:cu[b + 1]]).sum())
            Lp.append(live[b] - rem)
            if cu[b + 1] > cu[b]:
                moved += live[b] - rem - int(sb[cu[b]])
            live[b] = live[b] - rem + tails[b]
        rd["attn_flops"] = attention_flops(s, Lp, tails)        # per attention layer
        rd["attn_bytes"] = attention_bytes(s, Lp, tails)        # per attention layer
        rd["gdn_flops"] = gdn_flops(s, tails)                   # per delta-rule layer
        rd["compact_bytes"] = compaction_bytes(s, moved)
        rd["gdn_bytes"] = gdn_bytes(s, tails)                   # per delta-rule layer
        rd["rope_bytes"] = rope_bytes(s, tails)                 # per attention layer
        rd["h2d"] = sum(t.numel() * t.element_size() for x in rd["h_in"].values() for t in x.values())
        rd["d2h"] = sum(t.numel() * t.element_size() for t in rd["h_out"].values())

    flush = torch.empty(256 << 20, dtype=torch.int8, device="cuda")
    stream = torch.cuda.current_stream()

    def one_step(i, host_io):
        r = i % R
        rd = rounds[r]
        if r == 0:
            work.fork_from(root)
        flush.fill_(i & 0x7F)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        if host_io:
            work.update_round(rd["cu"], rd["sb"], rd["se"], rd["tail_cu"], rd["h_in"], rd["h_out"], io_on_host=True)
        else:
            work.update_round(rd["cu"], rd["sb"], rd["se"], rd["tail_cu"], rd["d_in"], rd["d_out"])
        e1.record(stream)
        return e0, e1, r

    def timed(host_io, profile=False):
        """Warm-up steps, then K timed steps.  With `profile`, every library
        launch is bracketed by CUDA events (per-kernel durations); those
        events sit between kernels and keep consecutive launches from
        overlapping, so the headline steps run without them.  The profiled
        pass runs as many steps as the library's event pool can time (all
        of them when they fit)."""
        n_steps = min(args.steps, max(1, EVENT_POOL // max(1, launches_per_step))) if profile else args.steps
        for i in range(args.warmup):
            one_step(i, host_io)
        work.check()
        # restart the chain so the timed steps begin at round 0
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        launches0 = work.launch_count()
        work.profile_enable(profile)
        work.profile_read(0, reset=True)
        t0 = time.time()
        evs = [one_step(i, host_io) for i in range(n_steps)]
        torch.cuda.synchronize()
        t1 = time.time()
        if world > 1:
            dist.barrier()
        work.check()
        ms = [a.elapsed_time(b) for a, b, _ in evs]
        kernels = {}
        for kfam, name in enumerate(kvm.KERNEL_NAMES):
            n, kms = work.profile_read(kfam)
            if n:
                kernels[name] = {"launches": n, "total_ms": kms}
        work.profile_read(0, reset=True)
        work.profile_enable(False)
        launches = work.launch_count() - launches0
        total_ms = max_over_ranks(float(sum(ms)), world, device="cuda")
        return total_ms, [r for _, _, r in evs], kernels, launches, (t0, t1), ms

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    launches_per_step = 1
    total_ms, rids, _, launches, (t0, t1), _ = timed(host_io=False)
    launches_per_step = -(-launches // args.steps)
    clk = clocks.summary(t0, t1)
    # per-kernel durations: the same steps again (as many as the event pool times) with per-launch events
    prof_ms, prof_rids, kernels, _, _, _ = timed(host_io=False, profile=True)
    e2e_ms, e2e_rids, _, _, _, e2e_steps = timed(host_io=True)
    scratch = from_scratch_prefill(w, plan, mk, flush, args, seed_base) if args.workload == "refill" else None
    clocks.stop()

    # every rank's tail tokens over the job's time (replicas process equal
    # shares; a partitioned population does not)
    toks_job = sum_over_ranks(float(sum(sum(rounds[r]["tails"]) for r in rids)), world, device="cuda")
    value = job_throughput(1, toks_job, total_ms)
    e2e_value = job_throughput(1, sum_over_ranks(float(sum(sum(rounds[r]["tails"]) for r in e2e_rids)), world,
                                                 device="cuda"), e2e_ms)
    hbm, tc_burst, tc_sust, peak_src = load_peaks()
    n_attn, n_gdn = len(s.attn_layers), len(s.gdn_layers)
    # algorithmic work of every kernel family over the steps of the per-kernel pass
    work = {
        "tail_attention": ("tensor", sum(rounds[r]["attn_flops"] * n_attn for r in prof_rids)),
        "gdn": ("hbm", sum(rounds[r]["gdn_bytes"] * n_gdn for r in prof_rids)),
        "kv_compact": ("hbm", sum(rounds[r]["compact_bytes"] for r in prof_rids)),
        "rope_append": ("hbm", sum(rounds[r]["rope_bytes"] * n_attn for r in prof_rids)),
    }
    fam = {k: dict(v) for k, v in kernels.items()}
    if "gdn_chunk_scan" in fam:
        prep = fam.get("gdn_chunk_prep", {"total_ms": 0.0})
        fam["gdn"] = {"launches": fam["gdn_chunk_scan"]["launches"],
                      "total_ms": fam["gdn_chunk_scan"]["total_ms"] + prep["total_ms"]}
    rooflines = {}
    for name, (bound, amount) in work.items():
        d = fam.get(name)
        if not d or d["total_ms"] <= 0 or d["launches"] == 0:
            continue
        secs = d["total_ms"] / 1e3
        if bound == "tensor":
            ach, peak, unit = amount / secs / 1e12, tc_burst, "TFLOP/s"
        else:
            ach, peak, unit = amount / secs / 1e9, hbm, "GB/s"
        rooflines[name] = {"bound": bound, "achieved": ach, "peak": peak, "unit": unit, "frac": ach / peak,
                           "share": d["total_ms"] / prof_ms, "per_launch": amount / d["launches"],
                           "per_launch_unit": "flop" if bound == "tensor" else "byte"}
    # the dominant kernel family is the one with the largest share of the step
    dominant = max(rooflines, key=lambda k: rooflines[k]["share"]) if rooflines else None
    kfile = {"tail_attention": "tail_attn_tc.cu", "gdn": "gdn_scan_tc.cu", "kv_compact": "kv_compact.cu",
             "rope_append": "tail_attn.cu"}
    roofline = None
    if dominant:
        rf = rooflines[dominant]
        roofline = {"bound": rf["bound"], "kernel": dominant, "achieved": rf["achieved"], "peak": rf["peak"],
                    "unit": rf["unit"], "frac": rf["frac"],
                    "peak_kind": (f"bf16 dense burst, {peak_src}" if rf["bound"] == "tensor"
                                  else f"HBM copy bandwidth, {peak_src}"),
                    "traffic": ncu_traffic(kfile[dominant], dominant),
                    "algorithmic_per_launch": rf["per_launch"], "share_of_step": rf["share"]}
    # round roofline: every kernel family at the larger of its tensor and HBM
    # times (algorithmic work over the measured peaks), summed over the round
    per_round = []
    for r in rids:
        rd = rounds[r]
        t = n_attn * (max(rd["attn_flops"] / (tc_burst * 1e12), rd["attn_bytes"] / (hbm * 1e9))
                      + rd["rope_bytes"] / (hbm * 1e9))
        t += n_gdn * max(rd["gdn_flops"] / (tc_burst * 1e12), rd["gdn_bytes"] / (hbm * 1e9))
        t += rd["compact_bytes"] / (hbm * 1e9)
        per_round.append(t)
    roof_us = 1e6 * sum(per_round) / len(per_round)
    round_roofline = {"time_us": roof_us, "measured_us": 1e3 * total_ms / args.steps,
                      "frac": roof_us / (1e3 * total_ms / args.steps),
                      "model": "sum over the round's kernels of max(flops / bf16 peak, bytes / HBM peak), "
                               f"algorithmic work, {peak_src} peaks"}
    if rank != 0:
        return
    # ---- CPU oracle sample (rank 0 only, single GPU runs only)
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        secs, m, blocks = oracle_sample(w, oracle_state(w), CPU_BASELINE_TOKENS[args.workload])
        cpu = {"value": m / (secs * blocks), "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
               "sample": sample_text(w, m, secs)}
    per_kernel = {}
    for name, d in kernels.items():
        per_kernel[name] = {"launches": d["launches"], "avg_us": 1e3 * d["total_ms"] / d["launches"],
                            "share": d["total_ms"] / prof_ms}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": scaling, "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(w, args, world),
        "roofline": roofline,
        "round_roofline": round_roofline,
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": UNIT,
                "h2d_bytes_per_step": int(np.mean([rounds[r]["h2d"] for r in e2e_rids])),
                "d2h_bytes_per_step": int(np.mean([rounds[r]["d2h"] for r in e2e_rids])),
                "ms_per_step": e2e_ms / args.steps,
                # the host link is shared with the node's other jobs: the
                # spread of the steps shows whether one of them stalled
                "ms_per_step_median": float(np.median(e2e_steps)), "ms_per_step_max": float(np.max(e2e_steps))},
        "gpu_launches": launches,
        "kernels": per_kernel,
        "kernel_timing": ("per-launch CUDA events in a second pass over the same steps (events between "
                          "kernels stop launches from overlapping, so the headline pass runs without them); "
                          f"that pass took {prof_ms / len(prof_rids):.4f} ms per step over {len(prof_rids)} steps"),
        "rooflines": rooflines,
        "clocks": clk,
    }
    if scratch is not None:
        scratch["tail_update_ms"] = total_ms / args.steps
        scratch["ratio"] = scratch["ms"] / scratch["tail_update_ms"]
        line["refill_from_scratch"] = scratch
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=160)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", choices=["kvm", "reference"], default="kvm")
    ap.add_argument("--workload", choices=list(WORKLOAD_TEXT), default="long")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--layers", type=int, default=None,
                    help="shorter stack of the same 3:1 pattern and shapes (profiling captures that must hold "
                         "a few GB on the device); the default is the workload's own stack")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_kvm(args)


if __name__ == "__main__":
    main()
