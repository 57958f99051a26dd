"""Host-side planning of the library, on CPU (no device).

kvm_plan_removal runs the span checks and the per-character bookkeeping of
kvm_kv_compact (Eq. 2); it is compared with the oracle's span validation and
keep mask.  kvm_plan_attention returns the attention's work partition (Eq. 3
over the compacted cache plus the tail); it is checked against what any
correct partition must satisfy: every (query tile, key tile) unit is
processed by exactly one block, in order, and the tiles shared by several
blocks are listed once each with the first block that starts inside them.
"""
import numpy as np
import pytest

from oracle import kvm_oracle as O
from paper_2609_18935_gb300 import kvm

KVM_E_INVAL, KVM_E_SPAN, KVM_E_UNSUPPORTED = kvm.KVM_E_INVAL, kvm.KVM_E_SPAN, kvm.KVM_E_UNSUPPORTED


@pytest.fixture(scope="module", autouse=True)
def lib():
    try:
        return kvm.load_library()
    except OSError as e:
        pytest.skip(f"library not built: {e}")


def _random_spans(rng, L):
    """Sorted disjoint non-empty spans inside [0, L), possibly none."""
    if L == 0 or rng.random() < 0.2:
        return [], []
    cuts = np.sort(rng.choice(np.arange(L + 1), size=2 * int(rng.integers(1, 5)), replace=True))
    b, e = [], []
    for lo, hi in zip(cuts[0::2], cuts[1::2]):
        if hi > lo and (not e or lo >= e[-1]):
            b.append(int(lo))
            e.append(int(hi))
    return b, e


def _spoil(rng, L, b, e):
    """One way of making a span list invalid (or None if it cannot be)."""
    kind = int(rng.integers(0, 4))
    if kind == 0 and b:                                 # empty span
        i = int(rng.integers(0, len(b)))
        return b[:i] + [b[i]] + b[i + 1:], e[:i] + [b[i]] + e[i + 1:]
    if kind == 1:                                       # outside the live range
        return b + [L], e + [L + 1]
    if kind == 2 and len(b) >= 2:                       # unsorted
        return [b[1], b[0]] + b[2:], [e[1], e[0]] + e[2:]
    if kind == 3 and b and e[0] - b[0] >= 2:            # overlapping
        mid = (b[0] + e[0]) // 2
        return [b[0], mid] + b[1:], [e[0], e[0]] + e[1:]
    return None


def test_plan_removal_matches_oracle():
    rng = np.random.default_rng(2609)
    for trial in range(400):
        B = int(rng.integers(1, 7))
        live = [int(rng.integers(0, 200)) for _ in range(B)]
        spans = [_random_spans(rng, L) for L in live]
        bad = None
        if trial % 3 == 0:
            bad = int(rng.integers(0, B))
            spoiled = _spoil(rng, live[bad], *spans[bad])
            if spoiled is not None:
                spans[bad] = spoiled
        cu = np.concatenate([[0], np.cumsum([len(b) for b, _ in spans])])
        sb = [x for b, _ in spans for x in b]
        se = [x for _, e in spans for x in e]
        expect_error = False
        for L, (b, e) in zip(live, spans):
            try:
                O.validate_spans(L, b, e)
            except O.SpanError:
                expect_error = True
        if expect_error:
            with pytest.raises(kvm.KvmError) as ei:
                kvm.plan_removal(live, cu, sb, se)
            assert ei.value.code == KVM_E_SPAN, (trial, live, spans)
            continue
        new_live, first = kvm.plan_removal(live, cu, sb, se)
        for j, (L, (b, e)) in enumerate(zip(live, spans)):
            keep = O.keep_mask(L, b, e)
            assert new_live[j] == int(keep.sum())
            removed = np.flatnonzero(~keep)
            assert first[j] == (int(removed[0]) if removed.size else int(keep.sum()))


def test_plan_removal_rejects_bad_offsets():
    with pytest.raises(kvm.KvmError) as ei:
        kvm.plan_removal([10], [1, 1], [0], [2])             # span_cu[0] != 0
    assert ei.value.code == KVM_E_INVAL
    with pytest.raises(kvm.KvmError) as ei:
        kvm.plan_removal([10, 10], [0, 2, 1], [0, 3], [2, 4])  # not monotone
    assert ei.value.code == KVM_E_INVAL
    with pytest.raises(kvm.KvmError) as ei:
        kvm.plan_removal([-1], [0, 0], [], [])               # negative live length
    assert ei.value.code == KVM_E_INVAL


def _units(live, tails, Hq, Hkv):
    """Per query tile (character, KV head, tile), its number of 64-key tiles."""
    tpt = 128 // (Hq // Hkv)
    nk = []
    for L, M in zip(live, tails):
        for _ in range(Hkv):
            for qt in range((M + tpt - 1) // tpt):
                nk.append((L + min(M, (qt + 1) * tpt) + 63) // 64)
    return nk


def _check_partition(live, tails, Hq, Hkv, max_blocks):
    cu = np.concatenate([[0], np.cumsum(tails)])
    plan = kvm.plan_attention(live, cu, Hq, Hkv, max_blocks)
    nk = _units(live, tails, Hq, Hkv)
    n_units = sum(nk)
    G, T = plan["n_blocks"], plan["n_tiles"]
    tile, key = plan["block_tile"], plan["block_key"]
    assert T == len(nk)
    assert 1 <= G <= max_blocks
    assert G == max(1, min(max_blocks, n_units // 4))
    assert (tile[0], key[0]) == (0, 0)
    assert (tile[G], key[G]) == (T, 0)
    # ranges are contiguous and in order: unit index of each cut point
    base = np.concatenate([[0], np.cumsum(nk)])
    at = []
    for c in range(G + 1):
        assert 0 <= tile[c] <= T
        assert tile[c] == T and key[c] == 0 or 0 <= key[c] < nk[tile[c]]
        at.append(base[tile[c]] + key[c])
    assert all(a <= b for a, b in zip(at, at[1:]))
    assert at[-1] == n_units
    # empty ranges only at the end (spare blocks)
    sizes = np.diff(at)
    nonempty = np.flatnonzero(sizes > 0)
    if nonempty.size:
        assert nonempty[-1] == nonempty.size - 1
    # shared tiles: those with units in two or more blocks, each listed once
    # with the first block that starts inside it
    owners = {}
    for c in range(G):
        if at[c + 1] > at[c]:
            t0 = int(np.searchsorted(base, at[c], side="right") - 1)
            t1 = int(np.searchsorted(base, at[c + 1] - 1, side="right") - 1)
            for t in range(t0, t1 + 1):
                owners.setdefault(t, []).append(c)
    assert sorted(owners) == list(range(T))
    expect = sorted(cs[1] for cs in owners.values() if len(cs) > 1)
    assert sorted(plan["split_first_block"].tolist()) == expect
    # balance: no block's cost (units + 8 per segment it starts) exceeds the
    # mean by more than two segments and a unit
    costs = []
    for c in range(G):
        if at[c + 1] == at[c]:
            continue
        t0 = int(np.searchsorted(base, at[c], side="right") - 1)
        t1 = int(np.searchsorted(base, at[c + 1] - 1, side="right") - 1)
        costs.append(at[c + 1] - at[c] + 8 * (t1 - t0 + 1))
    assert max(costs) <= sum(costs) / G + 2 * 8 + 1
    return plan


def test_plan_attention_partitions_every_unit_once():
    rng = np.random.default_rng(18935)
    for trial in range(150):
        B = int(rng.integers(1, 33))
        live = [int(rng.integers(0, 20000)) for _ in range(B)]
        tails = [int(rng.integers(0, 600)) if rng.random() > 0.1 else 0 for _ in range(B)]
        if sum(tails) == 0:
            tails[0] = 1
        Hq, Hkv = [(16, 2), (8, 2), (8, 8), (32, 4)][trial % 4]
        _check_partition(live, tails, Hq, Hkv, int(rng.choice([1, 7, 152, 320])))


def test_plan_attention_npc_round():
    """npc shape (16 / 2 heads, L' 7782, M 256) on 152 SMs: 32 query tiles
    of ~126 key tiles, all split between blocks."""
    plan = _check_partition([7782], [256], 16, 2, 152)
    assert plan["n_tiles"] == 32 and plan["n_blocks"] == 152
    assert len(plan["split_first_block"]) == 32


def test_plan_attention_rejects_bad_shapes():
    for args, code in [(([10], [0, 5], 12, 8, 152), KVM_E_UNSUPPORTED),   # 12 not a multiple of 8
                       (([10], [0, 5], 24, 2, 152), KVM_E_UNSUPPORTED),   # group 12, not a power of two
                       (([10], [0, 5], 16, 2, 0), KVM_E_INVAL),
                       (([10], [0, 5], 16, 2, 321), KVM_E_INVAL),
                       (([10, 10], [0, 5, 4], 16, 2, 152), KVM_E_INVAL)]:
        with pytest.raises(kvm.KvmError) as ei:
            kvm.plan_attention(*args)
        assert ei.value.code == code, args


def test_spans_from_positions_match_brute_force():
    """Position ranges [b, e) map to the live indices whose positions lie in
    them (the paper checks deletion ranges against live spans, §4.2): holes
    in the positions are skipped, and a range must be non-empty, in order,
    and cover at least one live entry."""
    rng = np.random.default_rng(479547)
    for trial in range(300):
        live = int(rng.integers(0, 60))
        positions = np.sort(rng.choice(np.arange(400), size=live, replace=False)).astype(np.int32)
        n = int(rng.integers(1, 5))
        cuts = np.sort(rng.integers(-5, 410, size=2 * n))
        pb, pe = cuts[0::2].tolist(), cuts[1::2].tolist()
        if trial % 5 == 0 and n >= 2:                        # out of order
            pb[0], pb[1], pe[0], pe[1] = pb[1], pb[0], pe[1], pe[0]
        expect, prev_end, bad = [], None, False
        for b, e in zip(pb, pe):
            idx = np.flatnonzero((positions >= b) & (positions < e))
            if b >= e or (prev_end is not None and b < prev_end) or idx.size == 0:
                bad = True
                break
            prev_end = e
            expect.append((int(idx[0]), int(idx[-1]) + 1))
        if bad:
            with pytest.raises(kvm.KvmError) as ei:
                kvm.plan_spans_from_positions(positions, pb, pe)
            assert ei.value.code == KVM_E_SPAN, (trial, positions, pb, pe)
            continue
        sb, se = kvm.plan_spans_from_positions(positions, pb, pe)
        assert list(zip(sb.tolist(), se.tolist())) == expect
        keep = O.keep_mask(live, sb, se)                     # the spans are a valid removal
        in_ranges = np.zeros(live, bool)
        for b, e in zip(pb, pe):
            in_ranges |= (positions >= b) & (positions < e)
        assert np.array_equal(~keep, in_ranges)


def test_spans_from_positions_rejects_bad_positions():
    with pytest.raises(kvm.KvmError) as ei:
        kvm.plan_spans_from_positions([3, -1, 4], [0], [5])   # a negative position id
    assert ei.value.code == KVM_E_INVAL


def test_spans_from_positions_out_of_order_brute_force():
    """After slot-preserving placement or re-rotation (§5.2) live positions
    need not increase: a range then maps to the live entries whose positions
    lie in it, which must form one contiguous run of live indices."""
    rng = np.random.default_rng(261955)
    checked = 0
    for trial in range(400):
        live = int(rng.integers(1, 40))
        positions = rng.choice(np.arange(200), size=live, replace=False).astype(np.int32)
        if trial % 2:                                        # mostly increasing, one block moved back
            positions = np.sort(positions)
            a = int(rng.integers(0, live))
            e = int(rng.integers(a, live)) + 1
            positions[a:e] = np.sort(rng.choice(np.arange(1000, 1100), size=e - a, replace=False))
        b0 = int(rng.integers(-5, 1100))
        e0 = b0 + int(rng.integers(1, 120))
        idx = np.flatnonzero((positions >= b0) & (positions < e0))
        ok = idx.size > 0 and idx[-1] - idx[0] + 1 == idx.size
        if not ok:
            with pytest.raises(kvm.KvmError) as ei:
                kvm.plan_spans_from_positions(positions, [b0], [e0])
            assert ei.value.code == KVM_E_SPAN
            continue
        sb, se = kvm.plan_spans_from_positions(positions, [b0], [e0])
        assert (int(sb[0]), int(se[0])) == (int(idx[0]), int(idx[-1]) + 1)
        checked += 1
    assert checked > 30


def test_probe_statistics_match_the_oracle():
    """kvm_effective_group_count and kvm_total_variation (host only) against
    the oracle's definitions, on random masses and distributions."""
    rng = np.random.default_rng(1832)
    for trial in range(50):
        n = int(rng.integers(1, 40))
        mass = rng.random(n) * (rng.random(n) < 0.7)
        if mass.sum() == 0:
            mass[0] = 1.0
        assert abs(kvm.effective_group_count(mass) - O.effective_group_count(mass)) < 1e-12
        p, q = rng.random(n), rng.random(n)
        p, q = p / p.sum(), q / q.sum()
        assert abs(kvm.total_variation(p, q) - O.total_variation(p, q)) < 1e-15
    with pytest.raises(kvm.KvmError):
        kvm.effective_group_count([0.0, 0.0])
    with pytest.raises(kvm.KvmError):
        kvm.effective_group_count([0.5, -0.1])


def test_partition_balance_and_brute_force():
    """kvm_plan_partition: each character on exactly one rank, the heaviest
    rank within the largest cost of the mean (the LPT bound), and within 4/3
    of the best partition found by enumeration on small populations."""
    import itertools
    rng = np.random.default_rng(31)
    for trial in range(60):
        n = int(rng.integers(1, 9))
        ranks = int(rng.integers(1, 4))
        cost = [int(x) for x in rng.integers(0, 10_000, size=n)]
        rank_of, loads = kvm.plan_partition(cost, ranks)
        assert len(rank_of) == n and all(0 <= r < ranks for r in rank_of)
        got = [sum(c for c, r in zip(cost, rank_of) if r == k) for k in range(ranks)]
        assert got == list(loads)
        assert max(got) <= sum(cost) / ranks + max(cost)
        best = min(max(sum(c for c, r in zip(cost, a) if r == k) for k in range(ranks))
                   for a in itertools.product(range(ranks), repeat=n))
        assert max(got) <= best * 4 / 3 + 1e-9
    assert list(kvm.plan_partition([5, 5, 5, 5], 2)[1]) == [10, 10]
    with pytest.raises(kvm.KvmError):
        kvm.plan_partition([1, -2], 2)
