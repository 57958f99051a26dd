"""Parity at the full workload sizes, through the same C ABI call the
benchmark times (kvm_update_round), checked on sampled outputs.

Compaction and the tail append are checked bit-exactly for every attention
layer and character.  Attention outputs are checked on sampled (token, head)
rows, each recomputed by the oracle over the full surviving cache; delta-rule
outputs and carried states are checked on sampled (layer, character, head)
recurrences that the oracle runs token by token.  Layers that are not checked
get device-drawn inputs of the same distributions, so that the oracle only
draws what it checks.
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


class Sampled:
    """A GPU context plus oracle shadows of the sampled parts of its state."""

    def __init__(self, w, check_layers, check_chars, check_heads, max_tail):
        import torch
        from harness import to_torch_bf16
        from oracle import kvm_oracle as O
        from paper_2609_18935_gb300 import kvm
        self.O, self.w, self.s = O, w, w.shape
        s = self.s
        self.ctx = kvm.Context(s.layer_kind, s.n_q_heads, s.n_kv_heads, s.head_dim, s.rotary_dim, s.rope_theta,
                               s.n_gdn_heads, s.d_k, s.d_v, w.capacity(), max_tail)
        self.check_layers, self.check_chars, self.check_heads = check_layers, check_chars, check_heads
        self.caches = {}     # (layer, b) -> oracle AttnCache
        self.states = {}     # (layer, b, h) -> fp64 state of one head
        B = w.n_chars
        S_all = {l: np.zeros((B, s.n_gdn_heads, s.d_v, s.d_k), np.float32) for l in s.gdn_layers}
        for b, n in enumerate(w.prefix_len):
            pos = np.arange(n, dtype=np.int32)
            self.ctx.load_prefix(b, n, n, pos)
            for l in s.attn_layers:
                K, V, _ = W.prefix_cache(w, b, l, n)
                self.ctx.set_kv(l, b, to_torch_bf16(K).cuda(), to_torch_bf16(V).cuda())
                if l in check_layers and b in check_chars:
                    self.caches[(l, b)] = O.AttnCache(O.bf16_to_f64(K), O.bf16_to_f64(V), pos)
            for l in s.gdn_layers:
                S_all[l][b] = W.prefix_state(w, b, l)
                if l in check_layers and b in check_chars:
                    for h in check_heads:
                        self.states[(l, b, h)] = O.f32_to_f64(S_all[l][b, h])
        for l in s.gdn_layers:
            self.ctx.set_state(l, torch.from_numpy(S_all[l]).cuda())
        self.cursor = list(w.prefix_len)
        torch.cuda.synchronize()

    def round(self, rnd, rng):
        import torch
        from harness import to_torch_bf16, torch_bf16_to_f64, rel_l2
        O, s, w = self.O, self.s, self.w
        B = w.n_chars
        live = [self.ctx.get_live(b)[0] for b in range(B)]
        cu, sb, se, tails = W.round_plan(w, rnd, live)
        tail_cu = np.concatenate([[0], np.cumsum(tails)]).astype(np.int32)
        T = int(tail_cu[-1])
        dev = W.device_round_inputs(w, 50_000 + rnd, tails)
        host = W.tail_inputs(w, rnd, tails, layers=self.check_layers)
        for l, x in host.items():
            d = {k: to_torch_bf16(x[k]).cuda() for k in ("q", "k", "v")}
            if s.layer_kind[l] == W.GDN:
                d["alpha"] = torch.from_numpy(x["alpha"]).cuda()
                d["beta"] = torch.from_numpy(x["beta"]).cuda()
            dev[l] = d
        outs = {l: torch.empty((T, s.n_q_heads, s.head_dim) if k == W.ATTN else (T, s.n_gdn_heads, s.d_v),
                               dtype=torch.bfloat16, device="cuda") for l, k in enumerate(s.layer_kind)}
        # device copies of every cache before the round (compared byte for byte on the GPU)
        pre = {}
        for l in s.attn_layers:
            for b in range(B):
                k, v = self.ctx.get_kv(l, b)
                pre[(l, b)] = (k.view(torch.int16), v.view(torch.int16), self.ctx.get_positions(b))
        self.ctx.update_round(cu, sb, se, tail_cu, dev, outs)
        self.ctx.check()
        torch.cuda.synchronize()
        for b in range(B):
            bb, ee = sb[cu[b]:cu[b + 1]], se[cu[b]:cu[b + 1]]
            keep = torch.from_numpy(np.nonzero(O.keep_mask(live[b], bb, ee))[0]).cuda()
            Ln, p0 = int(keep.numel()), self.cursor[b]
            for l in s.attn_layers:
                k0, v0, pos0 = pre[(l, b)]
                k1, v1 = self.ctx.get_kv(l, b)
                pos1 = self.ctx.get_positions(b)
                assert torch.equal(k1.view(torch.int16)[:, :Ln], k0.index_select(1, keep)), f"K compaction {l} {b}"
                assert torch.equal(v1.view(torch.int16)[:, :Ln], v0.index_select(1, keep)), f"V compaction {l} {b}"
                assert torch.equal(pos1[:Ln], pos0.index_select(0, keep)), f"positions char {b}"
                tail_pos = torch.arange(p0, p0 + tails[b], dtype=torch.int32, device="cuda")
                assert torch.equal(pos1[Ln:], tail_pos), f"tail positions char {b}"
        errs = {}
        g = s.n_q_heads // s.n_kv_heads
        for l in self.check_layers:
            x = host[l]
            got = torch_bf16_to_f64(outs[l])
            S_gpu = self.ctx.get_state(l).cpu().numpy().astype(np.float64) if s.layer_kind[l] == W.GDN else None
            for b in self.check_chars:
                t0, t1 = int(tail_cu[b]), int(tail_cu[b + 1])
                M, p0 = t1 - t0, self.cursor[b]
                if M == 0:
                    continue
                if s.layer_kind[l] == W.ATTN:
                    c = self.caches[(l, b)]
                    bb, ee = sb[cu[b]:cu[b + 1]], se[cu[b]:cu[b + 1]]
                    K, V, pos, _ = O.kv_compact(c.K, c.V, c.pos, bb, ee)
                    positions = p0 + np.arange(M)
                    krot = O.rope(O.bf16_to_f64(x["k"][t0:t1]), positions, s.rotary_dim, s.rope_theta)
                    vnew = O.bf16_to_f64(x["v"][t0:t1])
                    toks = sorted(set([0, M - 1] + [int(t) for t in rng.integers(0, M, size=min(6, M))]))
                    qrot = O.rope(O.bf16_to_f64(x["q"][t0:t1][toks]), positions[toks], s.rotary_dim, s.rope_theta)
                    ref, gpu = [], []
                    for ti, tok in enumerate(toks):
                        for hq in range(s.n_q_heads):
                            kv = hq // g
                            keys = np.concatenate([K[kv], krot[:tok + 1, kv]])
                            vals = np.concatenate([V[kv], vnew[:tok + 1, kv]])
                            ref.append(O.attend_row(qrot[ti, hq], keys, vals))
                            gpu.append(got[t0 + tok, hq])
                    errs[("attn", l, b)] = rel_l2(np.array(gpu), np.array(ref))
                    self.caches[(l, b)] = O.AttnCache(np.concatenate([K, np.transpose(krot, (1, 0, 2))], axis=1),
                                                      np.concatenate([V, np.transpose(vnew, (1, 0, 2))], axis=1),
                                                      np.concatenate([pos, positions]))
                else:
                    for h in self.check_heads:
                        sl = np.s_[t0:t1, h:h + 1]
                        o, S = O.gdn_recurrent(O.bf16_to_f64(x["q"][sl]), O.bf16_to_f64(x["k"][sl]),
                                               O.bf16_to_f64(x["v"][sl]), O.f32_to_f64(x["alpha"][sl]),
                                               O.f32_to_f64(x["beta"][sl]), self.states[(l, b, h)][None])
                        self.states[(l, b, h)] = S[0]
                        errs[("gdn_out", l, b, h)] = rel_l2(got[t0:t1, h], o[:, 0])
                        errs[("S", l, b, h)] = rel_l2(S_gpu[b, h], S[0])
        for b in range(B):
            self.cursor[b] += tails[b]
        return errs


def _check(errs, what):
    assert errs, f"{what}: nothing was checked"
    bad = {k: v for k, v in errs.items() if not v <= TOL}
    assert not bad, f"{what}: rel-L2 above {TOL}: {bad}"


def test_npc_full_size_eight_rounds():
    """npc: 4 layers 3:1, prefix 8192, 8 chained rounds of 1-4 spans (~5 %), tail 256."""
    w = W.make_workload("npc")
    smp = Sampled(w, check_layers=[0, 2, 3], check_chars=[0], check_heads=[0, 9], max_tail=256)
    rng = np.random.default_rng(7)
    for r in range(8):
        _check(smp.round(r, rng), f"npc round {r}")


def test_long_lived_full_size_round():
    """long: 48 layers 3:1, prefix 32768, 10 spans = 3 % removed, tail 1024."""
    w = W.make_workload("long")
    smp = Sampled(w, check_layers=[0, 3, 46, 47], check_chars=[0], check_heads=[5], max_tail=1024)
    _check(smp.round(0, np.random.default_rng(8)), "long")


def test_population_full_size_round():
    """pop: 32 characters varlen-packed, prefixes U[2048,16384], 2-8 % in 1-6 spans, tails U[64,512]."""
    w = W.make_workload("pop")
    max_tail = sum(p[2] for p in w.plan[0])
    smp = Sampled(w, check_layers=[1, 3, 11], check_chars=[0, 7, 31], check_heads=[3], max_tail=max_tail)
    _check(smp.round(0, np.random.default_rng(9)), "pop")


def test_refill_equivalence_full_size():
    """refill: with nothing removed, a 512-token tail update on a 16384-token
    prefix equals the last 512 rows of a from-scratch prefill of 16896 tokens
    (outputs, final states, cache bytes), both computed on the GPU; and both
    arms match the fp64 oracle run over the whole 16896-token sequence from an
    empty state: attention rows of sampled tail tokens (every head) over the
    full cache, and sampled delta-rule heads token by token from zero
    (outputs of the tail and the final state)."""
    import torch
    from harness import to_torch_bf16, torch_bf16_bits, torch_bf16_to_f64, rel_l2
    from oracle import kvm_oracle as O
    from paper_2609_18935_gb300 import kvm
    w = W.make_workload("refill")
    s = w.shape
    N, M = 16384, 512
    check_attn, check_gdn, heads = 3, 0, [0, 9]
    ins = W.device_round_inputs(w, 424242, [N + M])
    host = W.tail_inputs(w, 0, [N + M], layers=[check_gdn, check_attn])   # the layers the oracle checks
    for l, x in host.items():
        d = {k: to_torch_bf16(x[k]).cuda() for k in ("q", "k", "v")}
        if s.layer_kind[l] == W.GDN:
            d["alpha"] = torch.from_numpy(x["alpha"]).cuda()
            d["beta"] = torch.from_numpy(x["beta"]).cuda()
        ins[l] = d
    mk = lambda mt: kvm.Context(s.layer_kind, s.n_q_heads, s.n_kv_heads, s.head_dim, s.rotary_dim,
                                s.rope_theta, s.n_gdn_heads, s.d_k, s.d_v, [N + M], mt)
    shape = lambda l, T: (T, s.n_q_heads, s.head_dim) if s.layer_kind[l] == W.ATTN else (T, s.n_gdn_heads, s.d_v)
    zero = np.zeros(2, np.int32)
    n_layers = len(s.layer_kind)
    full = mk(N + M)
    o_full = {l: torch.empty(shape(l, N + M), dtype=torch.bfloat16, device="cuda") for l in range(n_layers)}
    full.update_round(zero, [], [], np.array([0, N + M]), ins, o_full)
    tail = mk(N)
    head_in = {l: {k: v[:N].contiguous() for k, v in x.items()} for l, x in ins.items()}
    tail_in = {l: {k: v[N:].contiguous() for k, v in x.items()} for l, x in ins.items()}
    o_head = {l: torch.empty(shape(l, N), dtype=torch.bfloat16, device="cuda") for l in range(n_layers)}
    tail.update_round(zero, [], [], np.array([0, N]), head_in, o_head)
    o_tail = {l: torch.empty(shape(l, M), dtype=torch.bfloat16, device="cuda") for l in range(n_layers)}
    tail.update_round(zero, [], [], np.array([0, M]), tail_in, o_tail)
    full.check()
    tail.check()
    for l in range(n_layers):
        e = rel_l2(torch_bf16_to_f64(o_tail[l]), torch_bf16_to_f64(o_full[l][N:]))
        assert e <= TOL, (l, e)
        if s.layer_kind[l] == W.GDN:
            a = tail.get_state(l).cpu().numpy().astype(np.float64)
            b = full.get_state(l).cpu().numpy().astype(np.float64)
            assert rel_l2(a, b) <= TOL, l
        else:
            ka, va = tail.get_kv(l, 0)
            kb, vb = full.get_kv(l, 0)
            assert np.array_equal(torch_bf16_bits(ka), torch_bf16_bits(kb))
            assert np.array_equal(torch_bf16_bits(va), torch_bf16_bits(vb))
    assert tail.get_live(0) == full.get_live(0) == (N + M, N + M)
    # ---- the oracle over the whole sequence from an empty state
    errs = {}
    x = host[check_attn]
    positions = np.arange(N + M)
    krot = O.rope(O.bf16_to_f64(x["k"]), positions, s.rotary_dim, s.rope_theta)
    vv = O.bf16_to_f64(x["v"])
    g = s.n_q_heads // s.n_kv_heads
    toks = sorted(set([0, 1, M - 1] + [int(t) for t in np.random.default_rng(12).integers(0, M, 5)]))
    got_tail, got_full = torch_bf16_to_f64(o_tail[check_attn]), torch_bf16_to_f64(o_full[check_attn][N:])
    for t in toks:
        qrot = O.rope(O.bf16_to_f64(x["q"][N + t:N + t + 1]), positions[N + t:N + t + 1], s.rotary_dim, s.rope_theta)
        ref = np.stack([O.attend_row(qrot[0, hq], krot[:N + t + 1, hq // g], vv[:N + t + 1, hq // g])
                        for hq in range(s.n_q_heads)])
        errs[("attn tail", t)] = rel_l2(got_tail[t], ref)
        errs[("attn refill", t)] = rel_l2(got_full[t], ref)
    x = host[check_gdn]
    S_tail = tail.get_state(check_gdn).cpu().numpy().astype(np.float64)
    got = torch_bf16_to_f64(o_tail[check_gdn])
    for h in heads:
        sl = np.s_[:, h:h + 1]
        o, S = O.gdn_recurrent(O.bf16_to_f64(x["q"][sl]), O.bf16_to_f64(x["k"][sl]), O.bf16_to_f64(x["v"][sl]),
                               O.f32_to_f64(x["alpha"][sl]), O.f32_to_f64(x["beta"][sl]),
                               np.zeros((1, s.d_v, s.d_k)))
        errs[("gdn tail out", h)] = rel_l2(got[:, h], o[N:, 0])
        errs[("gdn S", h)] = rel_l2(S_tail[0, h], S[0])
    _check(errs, "refill vs oracle")
