"""GPU parity of the attention probe (§5.3; Appendix C) against the fp64
oracle: after maintenance rounds (so the live cache has holes in position
space), the float32 reference softmax of the last n_q query tokens over the
live entries, averaged over queries and heads, and its per-group mass, with
the effective group count and the total variation distance computed from
them.  Bar: relative L2 5e-3 on the distribution and the group masses (fp32
against fp64; the measured error is far below it)."""
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


@pytest.mark.parametrize("head_dim,n_q_heads,n_q", [(256, 16, 8), (128, 8, 1), (64, 16, 16)])
def test_probe_after_maintenance_matches_oracle(head_dim, n_q_heads, n_q):
    import torch
    from harness import Pair, rel_l2, to_torch_bf16
    from oracle import kvm_oracle as O
    from paper_2609_18935_gb300 import kvm
    shape = W.ModelShape([W.GDN, W.ATTN, W.ATTN], n_q_heads, 2, head_dim, 64, 1e4, 4, 64, 64)
    prefix = [1000, 333]
    w = W.Workload("probe", 81, shape, prefix, 2)
    w.plan = [[(0.05, 3, 96), (0.1, 2, 40)], [(0.03, 2, 70), (0.0, 0, 17)]]
    pair = Pair(shape, prefix, w.capacity(), 96 + 40, seed_index=81)
    last = None
    for r in range(2):
        live = [pair.ctx.get_live(b)[0] for b in range(2)]
        cu, sb, se, tails = W.round_plan(w, r, live)
        last = (tails, W.tail_inputs(w, r, tails))
        errs = pair.run_round(cu, sb, se, tails, last[1])
        assert all(v <= TOL for v in errs.values()), errs
    tails, ins = last
    tail_cu = np.concatenate([[0], np.cumsum(tails)])
    rng = np.random.default_rng(5)
    for layer in shape.attn_layers:
        for b in range(2):
            L = pair.ctx.get_live(b)[0]
            qb = ins[layer]["q"][tail_cu[b]:tail_cu[b + 1]][-n_q:]       # queries of the last n_q entries
            cache = pair.oracle[b].caches[layer]
            ref = O.attention_probe(cache, O.bf16_to_f64(qb), shape.rotary_dim, shape.rope_theta)
            n_groups = 7
            group_of = rng.integers(-1, n_groups, size=L).astype(np.int32)
            probs, mass = pair.ctx.attn_probe(layer, b, to_torch_bf16(qb).cuda(),
                                              group_of=torch.from_numpy(group_of).cuda(), n_groups=n_groups)
            pair.ctx.check()
            got = probs.cpu().numpy().astype(np.float64)
            assert abs(got.sum() - 1.0) < 1e-4
            assert rel_l2(got, ref) <= TOL, (layer, b, rel_l2(got, ref))
            ref_mass = O.group_mass(ref, group_of, n_groups)
            got_mass = mass.cpu().numpy().astype(np.float64)
            assert rel_l2(got_mass, ref_mass) <= TOL
            assert abs(kvm.effective_group_count(got_mass) - O.effective_group_count(ref_mass)) <= \
                TOL * O.effective_group_count(ref_mass)
            assert kvm.total_variation(got, ref) <= TOL


def test_probe_rejects_bad_requests():
    import torch
    from harness import Pair
    from paper_2609_18935_gb300 import kvm
    pair = Pair(W.TINY, [20], [128], 64, seed_index=82)
    q = torch.zeros((4, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvm.KvmError):                 # a delta-rule layer
        pair.ctx.attn_probe(0, 0, q)
    with pytest.raises(kvm.KvmError):                 # more probe queries than the limit
        pair.ctx.attn_probe(1, 0, torch.zeros((17, 8, 64), dtype=torch.bfloat16, device="cuda"))
    with pytest.raises(kvm.KvmError):                 # a group id past n_groups is caught on the device
        pair.ctx.attn_probe(1, 0, q, group_of=torch.full((20,), 3, dtype=torch.int32, device="cuda"), n_groups=2)
        pair.ctx.check()
    pair.ctx.check()
