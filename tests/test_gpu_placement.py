"""GPU parity of the placement variants (§5.2) and maintenance delimiters
(§4.2) against the fp64 oracle, through the C ABI.

* fresh gapped prefill: the text read from an empty state with position-id
  gaps of 10,000 between records (per-token positions on kvm_update_round);
* slot-preserving maintenance: the replacement rotated at, and stored with,
  the position ids of the record it replaces (so live positions stop
  increasing), then a later round that removes it again by position range;
* tail-and-relocate: a true-tail round, then the tail's stored keys turned
  back to the replaced record's ids (kvm_rerotate_keys), then a round that
  attends over them;
* delimiters: tail tokens processed and then removed from every cache.
Bar: cache bytes and positions bit-exact where nothing is computed, outputs,
appended and turned keys and states within relative L2 5e-3 per (layer,
character).
"""
import numpy as np
import pytest

from workload import synth as W

pytestmark = pytest.mark.gpu
TOL = 5e-3
SHAPE = W.ModelShape([W.GDN, W.ATTN, W.GDN, W.ATTN], 16, 2, 256, 64, 1e4, 4, 128, 128)


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18935_gb300 import kvm
    kvm.load_library()


def _ok(errs, what):
    assert errs, what
    bad = {k: v for k, v in errs.items() if not v <= TOL}
    assert not bad, f"{what}: rel-L2 above {TOL}: {bad}"


def _inputs(seed, tails, shape=SHAPE):
    w = W.Workload("placement", seed, shape, [0] * len(tails), 1)
    w.plan = [[(0.0, 0, m) for m in tails]]
    return W.tail_inputs(w, 0, tails)


@pytest.mark.parametrize("via", ["update_round", "entry_points"])
def test_fresh_gapped_prefill(via):
    from harness import Pair
    records = [[40, 33, 57, 20], [70, 5, 64]]
    tails = [sum(r) for r in records]
    pair = Pair(SHAPE, [0, 0], [256, 256], sum(tails), seed_index=71, prefix="empty")
    tail_pos = np.concatenate([np.arange(10_000 * k, 10_000 * k + n) for rec in records for k, n in enumerate(rec)])
    errs = pair.run_round(np.zeros(3, np.int32), np.zeros(0, np.int32), np.zeros(0, np.int32), tails,
                          _inputs(71, tails), via=via, tail_pos=tail_pos.astype(np.int32))
    _ok(errs, "gapped prefill")
    assert pair.ctx.get_live(0) == (150, 30_020) and pair.ctx.get_live(1) == (139, 20_064)


def test_slot_preserving_rounds():
    from harness import Pair
    pair = Pair(SHAPE, [600, 400], [768, 512], 128, seed_index=72)
    # round 0: records at live [100, 160) and [50, 90) are replaced by 60 and 40
    # tokens rotated at, and stored with, the replaced records' ids
    cu, sb, se = np.array([0, 1, 2], np.int32), np.array([100, 50], np.int32), np.array([160, 90], np.int32)
    tails = [60, 40]
    tail_pos = np.concatenate([np.arange(100, 160), np.arange(50, 90)]).astype(np.int32)
    _ok(pair.run_round(cu, sb, se, tails, _inputs(72, tails), tail_pos=tail_pos), "slot round 0")
    assert pair.ctx.get_live(0) == (600, 600) and pair.ctx.get_live(1) == (400, 400)   # the cursor stays
    # round 1: the slot-placed record of character 0 is removed again by its
    # position range (live positions are out of order now) along with an
    # older one, and a true-tail record is appended
    sb0, se0 = pair.ctx.spans_from_positions(0, [10, 100], [20, 160])
    assert list(sb0) == [10, 540] and list(se0) == [20, 600]
    sb1, se1 = pair.ctx.spans_from_positions(1, [300], [330])
    cu = np.array([0, 2, 3], np.int32)
    sb = np.concatenate([sb0, sb1]).astype(np.int32)
    se = np.concatenate([se0, se1]).astype(np.int32)
    tails = [33, 70]
    _ok(pair.run_round(cu, sb, se, tails, _inputs(73, tails)), "slot round 1")


def test_tail_and_relocate():
    from harness import Pair
    pair = Pair(SHAPE, [500, 300], [640, 512], 128, seed_index=74)
    cu, sb, se = np.array([0, 1, 2], np.int32), np.array([200, 0], np.int32), np.array([240, 30], np.int32)
    tails = [48, 77]
    _ok(pair.run_round(cu, sb, se, tails, _inputs(74, tails)), "relocate round 0")
    # turn the tails back to the replaced records' ids (positions 200.. and 0..)
    _ok(pair.rerotate(0, 460, 508, np.arange(200, 248, dtype=np.int32)), "rerotate 0")
    _ok(pair.rerotate(1, 270, 347, np.arange(0, 77, dtype=np.int32)), "rerotate 1")
    assert pair.ctx.get_live(0)[1] == 548                  # the cursor never moves back
    # a later round attends over the relocated keys
    cu, sb, se = np.array([0, 1, 1], np.int32), np.array([5], np.int32), np.array([9], np.int32)
    tails = [64, 1]
    _ok(pair.run_round(cu, sb, se, tails, _inputs(75, tails)), "relocate round 1")


def test_maintenance_delimiters():
    from harness import Pair
    pair = Pair(SHAPE, [300, 200, 150], [512, 512, 512], 256, seed_index=76)
    cu, sb, se = np.array([0, 1, 1, 2], np.int32), np.array([10, 0], np.int32), np.array([50, 20], np.int32)
    tails = [70, 40, 65]
    # character 0: delimiters at the start and in the middle; character 1:
    # none; character 2: at the start and the very end
    delim = (np.array([0, 2, 2, 4], np.int32), np.array([0, 30, 0, 64], np.int32),
             np.array([3, 32, 2, 65], np.int32))
    _ok(pair.run_round(cu, sb, se, tails, _inputs(76, tails), delim=delim), "delimiter round 0")
    assert [pair.ctx.get_live(b)[0] for b in range(3)] == [300 - 40 + 70 - 5, 200 + 40, 150 - 20 + 65 - 3]
    # a second round: everything after the delimiters' removal keeps working
    cu, sb, se = np.array([0, 1, 2, 3], np.int32), np.array([250, 0, 100], np.int32), np.array([260, 5, 101], np.int32)
    tails = [64, 64, 1]
    delim = (np.array([0, 1, 1, 1], np.int32), np.array([63], np.int32), np.array([64], np.int32))
    _ok(pair.run_round(cu, sb, se, tails, _inputs(77, tails), delim=delim), "delimiter round 1")


def test_bad_positions_and_delimiters_are_refused():
    import torch
    from harness import Pair
    from paper_2609_18935_gb300 import kvm
    pair = Pair(SHAPE, [100], [256], 64, seed_index=78)
    before = pair.snapshot_kv()
    tails = [8]
    ins = {l: {k: (torch.from_numpy(v).cuda() if v.dtype != np.uint16 else
                   torch.from_numpy(v.view(np.int16)).view(torch.bfloat16).cuda()) for k, v in x.items()}
           for l, x in _inputs(78, tails).items()}
    outs = {l: torch.empty((8, 16, 256) if SHAPE.layer_kind[l] == W.ATTN else (8, 4, 128), dtype=torch.bfloat16,
                           device="cuda") for l in range(4)}
    z = np.zeros(2, np.int32)
    with pytest.raises(kvm.KvmError) as ei:                 # a negative position id
        pair.ctx.update_round(z, [], [], np.array([0, 8]), ins, outs, tail_pos=np.array([1, 2, 3, -4, 5, 6, 7, 8]))
    assert ei.value.code == kvm.KVM_E_INVAL
    with pytest.raises(kvm.KvmError) as ei:                 # a delimiter outside the tail
        pair.ctx.update_round(z, [], [], np.array([0, 8]), ins, outs, delim=([0, 1], [6], [9]))
    assert ei.value.code == kvm.KVM_E_SPAN
    with pytest.raises(kvm.KvmError) as ei:                 # re-rotation outside the live entries
        pair.ctx.rerotate_keys(0, 90, 101, np.arange(11))
    assert ei.value.code == kvm.KVM_E_SPAN
    pair.ctx.check()
    after = pair.snapshot_kv()
    for key in before:
        for x, y in zip(before[key], after[key]):
            assert np.array_equal(x, y)
    assert pair.ctx.get_live(0) == (100, 100)
