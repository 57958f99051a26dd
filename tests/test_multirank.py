"""The multi-rank host path of bench.py on CPU: two gloo ranks.

bench.py runs one process per GPU; ranks are independent replicas (each
maintains its own characters) joined only by a barrier and the max over
ranks of the timed region.  These tests run that host logic with the gloo
backend on CPU, and the reference arm under torchrun (rank 0 prints the one
JSON line, the other ranks exit 0 without output)."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, local = bench.dist_env()
    ms = 10.0 + 5.0 * rank                       # rank 1 is the slower one
    job_ms = bench.max_over_ranks(ms, w)
    dist.barrier()
    out.put((r, w, local, job_ms, bench.replica_seed(r), bench.job_throughput(w, 256.0 * 8, job_ms)))
    dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, w0, l0, ms0, seed0, v0), (r1, w1, l1, ms1, seed1, v1) = res
    assert (r0, r1) == (0, 1) and w0 == w1 == 2 and (l0, l1) == (0, 1)
    assert ms0 == ms1 == 15.0                     # max over ranks
    assert seed0 != seed1                         # replicas maintain different characters
    assert v0 == v1 == pytest.approx(2 * 256 * 8 / 0.015)


def test_single_rank_needs_no_process_group():
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.job_throughput(1, 100.0, 50.0) == pytest.approx(2000.0)


def test_reference_arm_under_torchrun_prints_on_rank_zero_only():
    pytest.importorskip("torch")
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--workload", "tiny", "--steps", "1", "--warmup", "3"]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [json.loads(x) for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    line = lines[0]
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"


def _partition_rank_main(rank, world, port, out):
    """One rank of a partitioned population: plan the partition (every rank
    computes the same plan), maintain only its own characters for a round
    with the fp64 oracle, and gather the outputs on every rank."""
    import numpy as np
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    full = _tiny_population()
    mine, scaling = bench.rank_share(full, rank, world)
    outs = _oracle_round(mine)
    gathered = [None] * world
    dist.all_gather_object(gathered, (rank, list(mine.char_ids), scaling, outs))
    if rank == 0:
        out.put(gathered)
    dist.destroy_process_group()


def _tiny_population():
    from workload import synth as W
    shape = W.ModelShape([W.GDN, W.ATTN], 4, 2, 16, 8, 1e4, 2, 8, 8)
    rng = np.random.default_rng(8)
    n = [int(x) for x in rng.integers(8, 80, size=7)]
    w = W.Workload("tiny-pop", 9, shape, n, 1)
    w.plan = [[(float(rng.uniform(0.05, 0.2)), int(rng.integers(1, 3)), int(rng.integers(1, 20))) for _ in n]]
    return w


def _oracle_round(w):
    """Round 0 of every character of w on the oracle: {population id: outputs}."""
    from oracle import kvm_oracle as O
    from workload import synth as W
    s = w.shape
    cu, sb, se, tails = W.round_plan(w, 0, list(w.prefix_len))
    ins = W.tail_inputs(w, 0, tails)
    tc = np.concatenate([[0], np.cumsum(tails)])
    res = {}
    for b in range(w.n_chars):
        N = w.prefix_len[b]
        caches, states = {}, {}
        for l in s.attn_layers:
            K, V, pos = W.prefix_cache(w, b, l, N)
            caches[l] = O.AttnCache(O.bf16_to_f64(K), O.bf16_to_f64(V), pos)
        for l in s.gdn_layers:
            states[l] = O.f32_to_f64(W.prefix_state(w, b, l))
        st = O.CharacterState(caches, states, N)
        x = {l: {k: (O.bf16_to_f64(v[tc[b]:tc[b + 1]]) if v.dtype == np.uint16 else O.f32_to_f64(v[tc[b]:tc[b + 1]]))
                 for k, v in d.items()} for l, d in ins.items()}
        o, _ = O.maintenance_round(st, s.layer_kind, sb[cu[b]:cu[b + 1]], se[cu[b]:cu[b + 1]], x, s.rotary_dim,
                                   s.rope_theta)
        res[w.gid(b)] = {l: v for l, v in o.items()}
    return res


def test_population_partition_over_two_gloo_ranks():
    """§8(e): a population split over two ranks by kvm_plan_partition.  Every
    character lands on exactly one rank, the heavier rank exceeds the mean
    cost by less than the largest character, and the ranks' outputs, put
    together, equal a one-rank run of the whole population (each character
    draws the same inputs on its rank)."""
    pytest.importorskip("torch")
    import torch.multiprocessing as mp
    from paper_2609_18935_gb300 import kvm
    from workload import synth as W
    import bench
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_partition_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    gathered = q.get(timeout=300)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    full = _tiny_population()
    owners = {}
    for rank, ids, scaling, outs in gathered:
        assert scaling == "strong"
        assert sorted(outs) == sorted(ids)
        for b in ids:
            assert b not in owners, f"character {b} on two ranks"
            owners[b] = rank
    assert sorted(owners) == list(range(full.n_chars))
    cu, sb, se, tails = W.round_plan(full, 0, list(full.prefix_len))
    after = [full.prefix_len[b] - int((se[cu[b]:cu[b + 1]] - sb[cu[b]:cu[b + 1]]).sum()) for b in range(full.n_chars)]
    cost = kvm.round_cost(after, tails)
    loads = [sum(cost[b] for b in owners if owners[b] == r) for r in range(2)]
    assert max(loads) - sum(cost) / 2 < max(cost)
    ref = _oracle_round(full)
    for rank, ids, scaling, outs in gathered:
        for b in ids:
            for l in ref[b]:
                np.testing.assert_array_equal(outs[b][l], ref[b][l])
    single, scaling = bench.rank_share(full, 0, 1)
    assert single is full and scaling == "weak"
