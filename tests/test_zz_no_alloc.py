"""The allocation-free compaction entry point (kvm_kv_compact_noalloc).

It serves callers that cannot call cudaMalloc -- an engine that owns every
byte of device memory through its own arena, or a frame loop that must not
stall on an allocation -- by compacting KV buffers the caller owns, with its
bookkeeping in a fixed device array inside the library.  These tests drive it
through the C ABI and check that, on two calls in a row, it leaves exactly the
bytes the oracle's keep mask selects from the buffers before the call, and the
bytes the context-based kvm_kv_compact leaves (compaction is bit-exact, so the
tolerance is equality), and that its failure signal
(kvm_kv_compact_noalloc_check) reports nothing.  The file sorts last so that a
stop-at-first-failure run has already run every other test.
"""
import numpy as np
import pytest

from workload import synth as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_18935_gb300 import kvm
    kvm.load_library()


def _caller_buffers(pair, cap):
    """Copy the context's live KV into caller-owned [n_slabs][cap][D] slabs."""
    import torch
    s = pair.shape
    n_slabs = len(s.attn_layers) * s.n_kv_heads
    K = torch.zeros((n_slabs, cap, s.head_dim), dtype=torch.bfloat16, device="cuda")
    V = torch.zeros_like(K)
    live, _ = pair.ctx.get_live(0)
    for a, l in enumerate(s.attn_layers):
        k, v = pair.ctx.get_kv(l, 0)
        K[a * s.n_kv_heads:(a + 1) * s.n_kv_heads, :live] = k
        V[a * s.n_kv_heads:(a + 1) * s.n_kv_heads, :live] = v
    pos = torch.zeros(cap, dtype=torch.int32, device="cuda")
    pos[:live] = pair.ctx.get_positions(0)
    return K, V, pos


@pytest.mark.parametrize("shape,prefix", [(W.npc_shape(8), 3000), (W.TINY, 700)])
def test_noalloc_compaction_matches_context_compaction(shape, prefix):
    import torch
    from harness import Pair
    from oracle import kvm_oracle as O
    from paper_2609_18935_gb300 import kvm
    cap = prefix + 64
    pair = Pair(shape, [prefix], [cap], 64, seed_index=61)
    K, V, pos = _caller_buffers(pair, cap)
    live = prefix
    for call, (frac, n_sp) in enumerate([(0.06, 4), (0.03, 2)]):      # two calls in a row
        total = int(round(frac * live))
        sb, se = W.removal_spans((61, call, 1), live, total, n_sp)
        keep = torch.from_numpy(np.nonzero(O.keep_mask(live, sb, se))[0]).cuda()
        K0, V0, pos0 = K[:, :live].clone(), V[:, :live].clone(), pos[:live].clone()
        pair.ctx.kv_compact(np.array([0, len(sb)]), sb, se)
        new_live = kvm.kv_compact_noalloc(K, V, pos, live, sb, se)
        kvm.kv_compact_noalloc_check()                 # raises KvmError on a reported failure
        torch.cuda.synchronize()
        assert new_live == pair.ctx.get_live(0)[0] == live - total == keep.numel()
        # against the oracle's keep mask applied to the bytes before the call
        assert torch.equal(K[:, :new_live].view(torch.int16), K0.index_select(1, keep).view(torch.int16))
        assert torch.equal(V[:, :new_live].view(torch.int16), V0.index_select(1, keep).view(torch.int16))
        assert torch.equal(pos[:new_live], pos0.index_select(0, keep))
        for a, l in enumerate(shape.attn_layers):
            k, v = pair.ctx.get_kv(l, 0)
            sl = slice(a * shape.n_kv_heads, (a + 1) * shape.n_kv_heads)
            assert torch.equal(K[sl, :new_live].view(torch.int16), k.view(torch.int16)), f"K call {call} layer {l}"
            assert torch.equal(V[sl, :new_live].view(torch.int16), v.view(torch.int16)), f"V call {call} layer {l}"
        assert torch.equal(pos[:new_live], pair.ctx.get_positions(0))
        live = new_live
    pair.ctx.check()


def test_noalloc_rejects_requests_beyond_its_scratch():
    import torch
    from paper_2609_18935_gb300 import kvm
    K = torch.zeros((600, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvm.KvmError) as ei:          # more slabs than the scratch has tickets for
        kvm.kv_compact_noalloc(K, K, None, 8, [0], [1])
    assert ei.value.code == kvm.KVM_E_CAPACITY
    K = torch.zeros((2, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvm.KvmError) as ei:          # overlapping spans
        kvm.kv_compact_noalloc(K, K, None, 8, [0, 1], [3, 4])
    assert ei.value.code == kvm.KVM_E_SPAN


def test_noalloc_rejects_mismatched_buffers():
    """Buffers that do not match K's shape are refused before any launch."""
    import torch
    from paper_2609_18935_gb300 import kvm
    K = torch.zeros((4, 64, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ValueError):                   # V smaller than K
        kvm.kv_compact_noalloc(K, K[:2].contiguous(), None, 32, [0], [1])
    with pytest.raises(ValueError):                   # positions shorter than slab_rows
        kvm.kv_compact_noalloc(K, K.clone(), torch.zeros(16, dtype=torch.int32, device="cuda"), 32, [0], [1])
    with pytest.raises(ValueError):                   # a host tensor
        kvm.kv_compact_noalloc(K, K.cpu(), None, 32, [0], [1])
    kvm.kv_compact_noalloc_check()
