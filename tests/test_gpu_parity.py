"""GPU parity: the CUDA library (through its C ABI) against the fp64 oracle.

Bar: compaction indices, cache bytes and positions bit-exact; attention
outputs, delta-rule outputs and carried states within relative L2 5e-3 of the
oracle (bf16 inputs, fp32 accumulation), after every round of a chain.
"""
import numpy as np
import pytest

from workload import synth as W

pytestmark = pytest.mark.gpu

TOL = 5e-3


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18935_gb300 import kvm
    kvm.load_library()


def _assert_errs(errs, tol=TOL, what=""):
    bad = {k: v for k, v in errs.items() if not (v <= tol)}
    assert not bad, f"{what} rel-L2 above {tol}: {bad}"


def test_tiny_round_matches_oracle():
    from harness import Pair
    w = W.make_workload("tiny")
    pair = Pair(w.shape, w.prefix_len, w.capacity(), 64, seed_index=w.index, prefix="refill")
    live = [pair.ctx.get_live(0)[0]]
    span_cu, sb, se, tails = W.round_plan(w, 0, live)
    assert int((se - sb).sum()) == 64 and len(sb) == 2
    errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails))
    _assert_errs(errs, what="tiny")


def test_tiny_round_via_separate_entry_points():
    from harness import Pair
    w = W.make_workload("tiny")
    pair = Pair(w.shape, w.prefix_len, w.capacity(), 64, seed_index=w.index, prefix="refill")
    span_cu, sb, se, tails = W.round_plan(w, 0, [512])
    errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails), via="entry_points")
    _assert_errs(errs, what="tiny/entry points")


@pytest.mark.parametrize("state_chain", [True, False])
def test_npc_shape_eight_chained_rounds(state_chain):
    """NPC-shaped stack (D 256, 16/2 heads, delta d 128, 3:1), shorter prefix so
    the oracle keeps up; 8 chained rounds, ragged tail (96 tokens: 1.5 chunks,
    12 query tiles); both forms of the delta-rule chain."""
    from harness import Pair
    shape = W.npc_shape(4)
    N, M = 1024, 96
    w = W.Workload("npc-small", 11, shape, [N], 8)
    w.plan = [[(0.05, 1 + r % 4, M)] for r in range(8)]
    pair = Pair(shape, [N], w.capacity(), M, seed_index=w.index)
    pair.ctx.set_gdn_state_chain(state_chain)
    for r in range(8):
        live = [pair.ctx.get_live(0)[0]]
        span_cu, sb, se, tails = W.round_plan(w, r, live)
        errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, r, tails))
        _assert_errs(errs, what=f"round {r}")


def test_population_varlen_edge_cases():
    """Several characters packed: a character with nothing removed, one whose
    whole cache is removed (the tail attends to itself only), one with no tail
    this round, spans at the very start and end, tails of 1 and 130 tokens."""
    from harness import Pair
    shape = W.ModelShape([W.GDN, W.ATTN, W.GDN, W.ATTN], 8, 2, 128, 64, 1e4, 4, 64, 96)
    prefix = [300, 64, 517, 129, 40]
    caps = [640, 256, 768, 384, 256]
    pair = Pair(shape, prefix, caps, 512, seed_index=21)
    spans = {0: ([], []), 1: ([0], [64]), 2: ([0, 100, 510], [3, 300, 517]), 3: ([5], [6]), 4: ([39], [40])}
    tails = [70, 33, 1, 0, 130]
    cu, sb, se = [0], [], []
    for b in range(5):
        sb += spans[b][0]
        se += spans[b][1]
        cu.append(len(sb))
    w = W.Workload("edge", 21, shape, prefix, 1)
    w.plan = [[(0, 0, m) for m in tails]]
    ins = W.tail_inputs(w, 0, tails)
    errs = pair.run_round(np.array(cu, np.int32), np.array(sb, np.int32), np.array(se, np.int32), tails, ins)
    _assert_errs(errs, what="edge")
    # a second round on the same population (earlier tails become removable)
    spans2 = [([0], [10]), ([2], [30]), ([100], [200]), ([0], [128]), ([0], [1])]
    cu, sb, se = [0], [], []
    for b in range(5):
        sb += spans2[b][0]
        se += spans2[b][1]
        cu.append(len(sb))
    tails2 = [64, 64, 64, 64, 64]
    w.plan = [[(0, 0, m) for m in tails2]]
    errs = pair.run_round(np.array(cu, np.int32), np.array(sb, np.int32), np.array(se, np.int32), tails2,
                          W.tail_inputs(w, 0, tails2))
    _assert_errs(errs, what="edge round 2")


@pytest.mark.parametrize("head_dim", [256, 128])
def test_many_ragged_tiles_without_key_splits(head_dim):
    """Enough query tiles to fill several waves of the attention grid, so each
    tile runs with its whole key range (no split-combine), and every
    character's last tile is ragged: the epilogue writes the output directly
    with some rows of the tile empty."""
    import torch
    from harness import Pair
    rng = np.random.default_rng(51)
    n_chars = 16
    tails = [int(m) for m in rng.integers(60, 330, n_chars)]
    tails = [m + 1 if m % 16 == 0 else m for m in tails]
    prefix = [int(n) for n in rng.integers(64, 400, n_chars)]
    caps = [((n + m + 127) // 128) * 128 for n, m in zip(prefix, tails)]
    shape = W.ModelShape([W.ATTN], 16, 2, head_dim, 64, 1e4, 1, 64, 32)
    tiles = sum(2 * ((m + 15) // 16) for m in tails)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    if tiles < 2 * sms:
        pytest.skip(f"{tiles} query tiles do not fill two waves on {sms} SMs")
    pair = Pair(shape, prefix, caps, sum(tails), seed_index=51)
    w = W.Workload("ragged-tiles", 51, shape, prefix, 1)
    w.plan = [[(0.05, 2, m) for m in tails]]
    span_cu, sb, se, tails = W.round_plan(w, 0, prefix)
    errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails))
    _assert_errs(errs, what=f"ragged tiles D={head_dim}")


def test_decode_after_maintenance_and_forked_roots():
    """After a maintenance round, one-token rounds (no removals, one tail
    token per character: decode steps) continue from the maintained state.
    A root forked after the maintenance (kvm_fork) decodes other tokens on its
    own and matches its own copy of the oracle state, while the original
    keeps matching its own."""
    from harness import Pair
    shape = W.npc_shape(4)
    N = [700, 1100]
    steps = 3
    w = W.Workload("decode", 23, shape, N, 1 + 2 * steps)
    w.plan = [[(0.05, 2, 80), (0.03, 1, 64)]] + [[(0.0, 0, 1), (0.0, 0, 1)]] * (2 * steps)
    pair = Pair(shape, N, w.capacity(), 80 + 64, seed_index=w.index)
    live = [pair.ctx.get_live(b)[0] for b in range(2)]
    span_cu, sb, se, tails = W.round_plan(w, 0, live)
    _assert_errs(pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails)), what="maintenance")
    task = pair.fork()
    for i in range(steps):
        for p, rnd in ((pair, 1 + i), (task, 1 + steps + i)):      # different tokens on each root
            live = [p.ctx.get_live(b)[0] for b in range(2)]
            span_cu, sb, se, tails = W.round_plan(w, rnd, live)
            assert len(sb) == 0 and tails == [1, 1]
            _assert_errs(p.run_round(span_cu, sb, se, tails, W.tail_inputs(w, rnd, tails)), what=f"decode {i}")


def test_large_cursor_positions():
    """Positions far beyond the live length (holes only in position space)."""
    from harness import Pair
    shape = W.ModelShape([W.ATTN], 16, 2, 256, 64, 1e4, 1, 64, 32)
    pair = Pair(shape, [200], [512], 64, seed_index=31, cursor_offset=479_000)
    w = W.Workload("far", 31, shape, [200], 1)
    w.plan = [[(0.1, 3, 64)]]
    span_cu, sb, se, tails = W.round_plan(w, 0, [200])
    errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails))
    _assert_errs(errs, what="far positions")


def test_rejected_calls_leave_state_unchanged():
    import torch
    from harness import Pair
    from paper_2609_18935_gb300 import kvm
    shape = W.TINY
    pair = Pair(shape, [100], [256], 64, seed_index=41)
    before = pair.snapshot_kv()
    S_before = pair.ctx.get_state(0).cpu()
    bad = [([0, 2], [30, 10], [20, 40]),    # overlap
           ([0, 1], [50], [50]),            # empty
           ([0, 1], [90], [101]),           # outside live
           ([0, 2], [40, 10], [50, 20])]    # unsorted
    for cu, b, e in bad:
        with pytest.raises(kvm.KvmError) as ei:
            pair.ctx.kv_compact(np.array(cu), np.array(b), np.array(e))
        assert ei.value.code == kvm.KVM_E_SPAN
    q = torch.zeros((200, 8, 64), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((200, 2, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvm.KvmError) as ei:     # 100 live + 200 > capacity 256
        pair.ctx.tail_attn_prefill(1, np.array([0, 200]), q, kv, kv, q)
    assert ei.value.code == kvm.KVM_E_CAPACITY
    with pytest.raises(kvm.KvmError) as ei:     # wrong layer kind
        pair.ctx.tail_attn_prefill(0, np.array([0, 10]), q, kv, kv, q)
    assert ei.value.code == kvm.KVM_E_INVAL
    pair.ctx.check()
    after = pair.snapshot_kv()
    for key in before:
        for x, y in zip(before[key], after[key]):
            assert np.array_equal(x, y)
    assert torch.equal(S_before, pair.ctx.get_state(0).cpu())
    assert pair.ctx.get_live(0) == (100, 100)


def test_spans_from_positions():
    from harness import Pair
    from paper_2609_18935_gb300 import kvm
    pair = Pair(W.TINY, [50], [256], 64, seed_index=51, cursor_offset=1000)
    sb, se = pair.ctx.spans_from_positions(0, [1005, 1040], [1010, 1041])
    assert list(sb) == [5, 40] and list(se) == [10, 41]
    with pytest.raises(kvm.KvmError):
        pair.ctx.spans_from_positions(0, [0], [10])     # covers no live entry


@pytest.mark.parametrize("arena", [False, True])
def test_host_resident_round_equals_device_round(arena):
    """kvm_update_round with host-resident (pinned) inputs and outputs runs
    the same kernels as with device tensors: outputs, caches and states
    bit-identical, over two chained rounds of a 2-character population.
    With `arena`, each layer's inputs sit back to back in one pinned buffer
    and go up in one copy."""
    import torch
    from paper_2609_18935_gb300 import kvm
    shape = W.ModelShape([W.GDN, W.ATTN, W.GDN, W.ATTN], 8, 2, 128, 64, 1e4, 4, 64, 96)
    prefix = [300, 517]
    caps = [640, 768]
    w = W.Workload("host-io", 61, shape, prefix, 2)
    w.plan = [[(0.05, 2, 70), (0.03, 1, 133)], [(0.02, 1, 64), (0.04, 3, 1)]]
    mk = lambda: kvm.Context(shape.layer_kind, shape.n_q_heads, shape.n_kv_heads, shape.head_dim,
                             shape.rotary_dim, shape.rope_theta, shape.n_gdn_heads, shape.d_k, shape.d_v, caps, 256)
    N = sum(prefix)
    ins = W.device_round_inputs(w, 7, prefix)
    outs = {l: torch.empty((N, shape.n_q_heads, shape.head_dim) if k == W.ATTN else (N, shape.n_gdn_heads, shape.d_v),
                           dtype=torch.bfloat16, device="cuda") for l, k in enumerate(shape.layer_kind)}
    root2 = kvm.Context(shape.layer_kind, shape.n_q_heads, shape.n_kv_heads, shape.head_dim, shape.rotary_dim,
                        shape.rope_theta, shape.n_gdn_heads, shape.d_k, shape.d_v, caps, N)
    root2.update_round(np.zeros(3, np.int32), [], [], np.array([0, prefix[0], N], np.int32), ins, outs)
    root2.check()
    dev, host = mk(), mk()
    dev.fork_from(root2)
    host.fork_from(root2)
    live = list(prefix)
    for r in range(2):
        span_cu, sb, se, tails = W.round_plan(w, r, live)
        tail_cu = np.concatenate([[0], np.cumsum(tails)]).astype(np.int32)
        T = int(tail_cu[-1])
        d_in = W.device_round_inputs(w, 100 + r, tails)
        h_in = (kvm.pinned_layer_inputs(d_in) if arena
                else {l: {k: t.cpu().pin_memory() for k, t in x.items()} for l, x in d_in.items()})
        shp = lambda l: (T, shape.n_q_heads, shape.head_dim) if shape.layer_kind[l] == W.ATTN else (T, shape.n_gdn_heads, shape.d_v)
        d_out = {l: torch.empty(shp(l), dtype=torch.bfloat16, device="cuda") for l in range(len(shape.layer_kind))}
        h_out = {l: torch.empty(shp(l), dtype=torch.bfloat16).pin_memory() for l in range(len(shape.layer_kind))}
        dev.update_round(span_cu, sb, se, tail_cu, d_in, d_out)
        host.update_round(span_cu, sb, se, tail_cu, h_in, h_out, io_on_host=True)
        dev.check()
        host.check()
        for l in range(len(shape.layer_kind)):
            assert torch.equal(d_out[l].cpu().view(torch.int16), h_out[l].view(torch.int16)), (r, l)
            if shape.layer_kind[l] == W.GDN:
                assert torch.equal(dev.get_state(l).cpu(), host.get_state(l).cpu()), (r, l)
            else:
                for b in range(2):
                    kd, vd = dev.get_kv(l, b)
                    kh, vh = host.get_kv(l, b)
                    assert torch.equal(kd.view(torch.int16), kh.view(torch.int16)) and torch.equal(
                        vd.view(torch.int16), vh.view(torch.int16)), (r, l, b)
        live = [dev.get_live(b)[0] for b in range(2)]
        assert live == [host.get_live(b)[0] for b in range(2)]


@pytest.mark.parametrize("state_chain", [True, False])
@pytest.mark.parametrize("n_chars,tails", [(1, [256]), (1, [1024]), (2, [130, 64]), (1, [1])])
def test_delta_rule_launch_plans_agree(n_chars, tails, state_chain):
    """The delta-rule layer as one launch (prep workers publishing records
    to chain blocks in the same grid) and as separate launches run the same
    arithmetic: outputs and states bit-identical, over two rounds, in both
    forms of the chain."""
    import torch
    from paper_2609_18935_gb300 import kvm
    shape = W.ModelShape([W.GDN, W.GDN], 16, 2, 256, 64, 1e4, 16, 128, 128)
    mk = lambda: kvm.Context(shape.layer_kind, 16, 2, 256, 64, 1e4, 16, 128, 128, [2 * max(tails) + 64] * n_chars,
                             sum(tails))
    a, b = mk(), mk()
    a.set_gdn_state_chain(state_chain)
    b.set_gdn_state_chain(state_chain)
    b.set_gdn_fusion(False)
    w = W.Workload("plans", 55, shape, [0] * n_chars, 2)
    for ctx in (a, b):
        for l in (0, 1):
            ctx.set_state(l, torch.from_numpy(np.stack([W.prefix_state(w, c, l) for c in range(n_chars)])).cuda())
    tail_cu = np.concatenate([[0], np.cumsum(tails)]).astype(np.int32)
    z = np.zeros(n_chars + 1, np.int32)
    for r in range(2):
        ins = W.device_round_inputs(w, 900 + r, tails)
        outs = [{l: torch.empty((sum(tails), 16, 128), dtype=torch.bfloat16, device="cuda") for l in (0, 1)}
                for _ in range(2)]
        a.update_round(z, [], [], tail_cu, ins, outs[0])
        b.update_round(z, [], [], tail_cu, ins, outs[1])
        a.check()
        b.check()
        for l in (0, 1):
            assert torch.equal(outs[0][l].view(torch.int16), outs[1][l].view(torch.int16)), (r, l)
            assert torch.equal(a.get_state(l), b.get_state(l)), (r, l)


@pytest.mark.parametrize("pattern", ["GAAGGA", "AGA"])
def test_compaction_scheduling_over_layer_patterns(pattern):
    """Layer orders that exercise how a round places its compactions: with
    recurrent layers before the first attention layer, each attention layer's
    cache is compacted in a launch of its own beside the layers before it
    (here two attention layers are also adjacent, so one such launch runs
    right at its layer); with an attention layer first, one launch on the
    caller's stream compacts every layer.  Two chained rounds against the
    oracle, caches bit-exact, outputs and states within the bar."""
    from harness import Pair
    kinds = [W.GDN if ch == "G" else W.ATTN for ch in pattern]
    shape = W.ModelShape(kinds, 8, 2, 64, 64, 1.0e4, 8, 64, 64)
    N = [300, 520]
    w = W.Workload("sched-" + pattern, 61, shape, N, 2)
    w.plan = [[(0.08, 3, 70), (0.05, 2, 40)], [(0.06, 2, 33), (0.04, 1, 90)]]
    pair = Pair(shape, N, w.capacity(), 70 + 90, seed_index=w.index)
    for rnd in range(2):
        live = [pair.ctx.get_live(b)[0] for b in range(2)]
        span_cu, sb, se, tails = W.round_plan(w, rnd, live)
        errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, rnd, tails))
        _assert_errs(errs, what=f"{pattern} round {rnd}")
