"""Failure detection on the GPU without a fault (the library's bounded waits
and its host-side validation).

* A compaction whose blocks are made to wait on a device word that nothing
  sets gives up after a short, host-set number of polls, moves nothing, and
  kvm_check reports KVM_E_DEVICE naming the expired wait; the CUDA context
  stays usable, and the context works again after its state is restored from
  a root with kvm_fork.
* A round whose position ids would pass 2^31 - 1 is refused on the host
  before any launch, with live lengths, cursors, caches and states unchanged.
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


def test_expired_compaction_wait_is_reported_and_context_recovers():
    from harness import Pair
    from paper_2609_18935_gb300 import kvm
    w = W.make_workload("tiny")
    pair = Pair(w.shape, w.prefix_len, w.capacity(), 64, seed_index=w.index, prefix="refill")
    work = pair.fork()                          # the context that will fail; `pair` stays the root
    live = [work.ctx.get_live(0)[0]]
    span_cu, sb, se, tails = W.round_plan(w, 0, live)
    work.ctx.debug_compact_wait(polls=256, stall=True)
    work.ctx.kv_compact(span_cu, sb, se)        # accepted on the host; the device waits expire
    with pytest.raises(kvm.KvmError) as ei:
        work.ctx.check()
    assert ei.value.code == kvm.KVM_E_DEVICE
    assert "wait-timeout" in str(ei.value)
    work.ctx.check()                            # the check cleared the error word
    # restore the failed context from the root and run the round normally
    work.ctx.debug_compact_wait(polls=0, stall=False)
    work.ctx.fork_from(pair.ctx)
    work.oracle = [o.copy() for o in pair.oracle]
    errs = work.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails))
    bad = {k: v for k, v in errs.items() if not v <= TOL}
    assert not bad, bad


def test_position_overflow_is_refused_before_any_launch():
    import torch
    from harness import Pair
    from paper_2609_18935_gb300 import kvm
    shape = W.TINY
    M = 64
    pair = Pair(shape, [100], [512], M, seed_index=43, cursor_offset=2**31 - 1 - M - 100)
    w = W.Workload("edge-cursor", 43, shape, [100], 2)
    w.plan = [[(0.1, 2, M)], [(0.1, 2, 1)]]
    span_cu, sb, se, tails = W.round_plan(w, 0, [100])
    errs = pair.run_round(span_cu, sb, se, tails, W.tail_inputs(w, 0, tails))
    assert all(v <= TOL for v in errs.values()), errs
    assert pair.ctx.get_live(0)[1] == 2**31 - 1          # the cursor reached the last position id
    live0, cur0 = pair.ctx.get_live(0)
    kv0 = pair.snapshot_kv()
    S0 = pair.ctx.get_state(0).cpu()
    span_cu, sb, se, tails = W.round_plan(w, 1, [live0])
    assert len(sb) > 0
    ins = {l: {k: (torch.from_numpy(v).cuda() if v.dtype != np.uint16 else
                   torch.from_numpy(v.view(np.int16)).view(torch.bfloat16).cuda()) for k, v in x.items()}
           for l, x in W.tail_inputs(w, 1, tails).items()}
    outs = {0: torch.empty((1, shape.n_gdn_heads, shape.d_v), dtype=torch.bfloat16, device="cuda"),
            1: torch.empty((1, shape.n_q_heads, shape.head_dim), dtype=torch.bfloat16, device="cuda")}
    with pytest.raises(kvm.KvmError) as ei:
        pair.ctx.update_round(span_cu, sb, se, np.array([0, 1]), ins, outs)
    assert ei.value.code == kvm.KVM_E_CAPACITY
    pair.ctx.check()
    assert pair.ctx.get_live(0) == (live0, cur0)
    kv1 = pair.snapshot_kv()
    for key in kv0:
        for x, y in zip(kv0[key], kv1[key]):
            assert np.array_equal(x, y)
    assert torch.equal(S0, pair.ctx.get_state(0).cpu())
