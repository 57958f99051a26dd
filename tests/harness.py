"""Drive the CUDA library and the fp64 oracle on the same seeded inputs.

Used by the GPU parity tests and by the smoke check.  The oracle never sees
anything the CUDA path produced except through explicit comparisons.
"""
from __future__ import annotations

import numpy as np

from oracle import kvm_oracle as O
from workload import synth as W


def rel_l2(x, ref) -> float:
    x = np.asarray(x, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.linalg.norm(ref)
    return float(np.linalg.norm(x - ref) / (den if den > 0 else 1.0))


def to_torch_bf16(bits: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16)


def torch_bf16_to_f64(t) -> np.ndarray:
    import torch
    u = t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return O.bf16_to_f64(u)


def torch_bf16_bits(t) -> np.ndarray:
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


class Pair:
    """A GPU context and per-character oracle states holding the same prefix."""

    def __init__(self, shape: W.ModelShape, prefix_len, capacity, max_tail, seed_index=0,
                 prefix="random", cursor_offset=0, conv=False):
        import torch
        from paper_2609_18935_gb300 import kvm
        self.shape = shape
        s = shape
        ck = 4 if conv else 0
        self._new_ctx = lambda: kvm.Context(s.layer_kind, s.n_q_heads, s.n_kv_heads, s.head_dim, s.rotary_dim,
                                            s.rope_theta, s.n_gdn_heads, s.d_k, s.d_v, capacity, max_tail,
                                            conv_kernel=ck)
        self.ctx = self._new_ctx()
        # short convolution: taps per delta-rule layer and a random carried
        # state (the last three pre-convolution inputs of an earlier round)
        self.conv_w = None
        conv_state = {}
        if conv:
            C_ = s.n_gdn_heads * (2 * s.d_k + s.d_v)
            self.conv_w = {l: W.conv_weights((seed_index, 996, l), C_) for l in s.gdn_layers}
            for l in s.gdn_layers:
                bits = W.normal_bf16((seed_index, 995, l), (len(prefix_len), 3, C_))
                conv_state[l] = bits
                self.ctx.set_conv_weights(l, torch.from_numpy(self.conv_w[l]).cuda())
                self.ctx.set_conv_state(l, to_torch_bf16(bits).cuda())
        self.B = len(prefix_len)
        self.oracle = []
        w = W.Workload("custom", seed_index, shape, list(prefix_len), 1)
        S_all = {l: np.zeros((self.B, s.n_gdn_heads, s.d_v, s.d_k), np.float32) for l in s.gdn_layers}
        for b, n in enumerate(prefix_len):
            caches, states = {}, {}
            pos = np.arange(n, dtype=np.int32) + np.int32(cursor_offset)
            cursor = n + cursor_offset
            self.ctx.load_prefix(b, n, cursor, pos)
            for l in s.attn_layers:
                if prefix == "refill":
                    toks = W.prefix_tokens(w, b, l, n)
                    kr = O.rope(O.bf16_to_f64(toks["k"]), pos, s.rotary_dim, s.rope_theta)
                    K = W.f64_to_bf16_bits(np.transpose(kr, (1, 0, 2)))
                    V = np.ascontiguousarray(np.transpose(toks["v"], (1, 0, 2)))
                else:
                    K, V, _ = W.prefix_cache(w, b, l, n)
                if n > 0:
                    self.ctx.set_kv(l, b, to_torch_bf16(K).cuda(), to_torch_bf16(V).cuda())
                caches[l] = O.AttnCache(O.bf16_to_f64(K), O.bf16_to_f64(V), pos.astype(np.int64))
            for l in s.gdn_layers:
                if prefix == "empty":
                    S32 = np.zeros((s.n_gdn_heads, s.d_v, s.d_k), np.float32)
                elif prefix == "refill" and n > 0:
                    toks = W.prefix_tokens(w, b, l, n)
                    _, S = O.gdn_recurrent(O.bf16_to_f64(toks["q"]), O.bf16_to_f64(toks["k"]),
                                           O.bf16_to_f64(toks["v"]), O.f32_to_f64(toks["alpha"]),
                                           O.f32_to_f64(toks["beta"]), np.zeros((s.n_gdn_heads, s.d_v, s.d_k)))
                    S32 = S.astype(np.float32)
                else:
                    S32 = W.prefix_state(w, b, l)
                S_all[l][b] = S32
                states[l] = O.f32_to_f64(S32)
            self.oracle.append(O.CharacterState(caches, states, cursor,
                                                {l: O.bf16_to_f64(conv_state[l][b]) for l in conv_state}))
        for l in s.gdn_layers:
            self.ctx.set_state(l, torch.from_numpy(S_all[l]).cuda())
        torch.cuda.synchronize()

    # ------------------------------------------------------------------
    def snapshot_kv(self):
        """Device bytes of every live cache: {(layer, b): (K bits, V bits, pos)}."""
        snap = {}
        for l in self.shape.attn_layers:
            for b in range(self.B):
                k, v = self.ctx.get_kv(l, b)
                snap[(l, b)] = (torch_bf16_bits(k), torch_bf16_bits(v), self.ctx.get_positions(b).cpu().numpy())
        return snap

    def fork(self) -> "Pair":
        """A second pair holding the same state: a new GPU context filled by
        kvm_fork from this one and a copy of the oracle states (a per-task
        root branching from a maintained one, §4.2)."""
        import copy
        other = object.__new__(Pair)
        other.__dict__.update(self.__dict__)
        other.ctx = self._new_ctx()
        other.ctx.fork_from(self.ctx)
        other.oracle = copy.deepcopy(self.oracle)
        return other

    def rerotate(self, b, begin, end, new_pos):
        """Tail-and-relocate on both sides: stored keys of live entries
        [begin, end) of character b turned to position ids new_pos.  Returns
        rel-L2 errors of the turned keys per attention layer; positions are
        checked exactly."""
        s = self.shape
        self.ctx.rerotate_keys(b, begin, end, new_pos)
        self.ctx.check()
        st = self.oracle[b]
        errs = {}
        for l in s.attn_layers:
            st.caches[l] = O.rerotate_keys(st.caches[l], begin, end, new_pos, s.rotary_dim, s.rope_theta)
            k1, _ = self.ctx.get_kv(l, b)
            errs[("rerotated_k", l, b)] = rel_l2(O.bf16_to_f64(torch_bf16_bits(k1))[:, begin:end],
                                                 st.caches[l].K[:, begin:end])
            assert np.array_equal(self.ctx.get_positions(b).cpu().numpy(), st.caches[l].pos.astype(np.int32))
        st.cursor = max(st.cursor, int(np.max(new_pos)) + 1) if len(new_pos) else st.cursor
        assert self.ctx.get_live(b)[1] == st.cursor
        return errs

    def run_round(self, span_cu, sb, se, tails, inputs, check_bitexact=True, via="update_round",
                  tail_pos=None, delim=None):
        """One round on both sides.  Returns dict of rel-L2 errors and raises on
        any bit-exactness violation.  tail_pos: optional int32 [sum M] position
        ids of the tail (placement variants); delim: optional (cu, begins,
        ends) of maintenance delimiters (update_round only)."""
        import torch
        s = self.shape
        B = self.B
        tail_cu = np.concatenate([[0], np.cumsum(tails)]).astype(np.int32)
        if delim is not None:
            assert via == "update_round", "delimiters are a field of kvm_update_round"
        pre = self.snapshot_kv() if check_bitexact else None
        L_before = [self.ctx.get_live(b)[0] for b in range(B)]
        cur_before = [self.ctx.get_live(b)[1] for b in range(B)]
        # ---- GPU
        dev_in, dev_out = {}, {}
        total = int(tail_cu[-1])
        for l, kind in enumerate(s.layer_kind):
            x = inputs[l]
            d = {"q": to_torch_bf16(x["q"]).cuda(), "k": to_torch_bf16(x["k"]).cuda(),
                 "v": to_torch_bf16(x["v"]).cuda()}
            if kind == W.GDN:
                d["alpha"] = torch.from_numpy(x["alpha"]).cuda()
                d["beta"] = torch.from_numpy(x["beta"]).cuda()
                dev_out[l] = torch.empty((total, s.n_gdn_heads, s.d_v), dtype=torch.bfloat16, device="cuda")
            else:
                dev_out[l] = torch.empty((total, s.n_q_heads, s.head_dim), dtype=torch.bfloat16, device="cuda")
            dev_in[l] = d
        gather = torch.full((max(1, sum(L_before)),), -1, dtype=torch.int32, device="cuda")
        if via == "update_round":
            self.ctx.update_round(span_cu, sb, se, tail_cu, dev_in, dev_out, gather_out=gather, tail_pos=tail_pos,
                                  delim=delim)
        else:
            self.ctx.kv_compact(span_cu, sb, se, gather_out=gather)
            for l, kind in enumerate(s.layer_kind):
                d = dev_in[l]
                if kind == W.ATTN:
                    self.ctx.tail_attn_prefill(l, tail_cu, d["q"], d["k"], d["v"], dev_out[l], tail_pos=tail_pos)
                else:
                    self.ctx.gdn_chunk_scan_from_state(l, tail_cu, d["q"], d["k"], d["v"], d["alpha"],
                                                       d["beta"], dev_out[l])
            self.ctx.advance(tail_cu, tail_pos=tail_pos)
        self.ctx.check()
        torch.cuda.synchronize()
        # ---- oracle, per character
        errs = {}
        gpu_out = {l: torch_bf16_to_f64(dev_out[l]) for l in dev_out}
        ora_out = {l: np.zeros_like(gpu_out[l]) for l in dev_out}
        gather_np = gather.cpu().numpy()
        g_off = 0
        for b in range(B):
            bb, ee = sb[span_cu[b]:span_cu[b + 1]], se[span_cu[b]:span_cu[b + 1]]
            t0, t1 = tail_cu[b], tail_cu[b + 1]
            ins = {}
            for l, kind in enumerate(s.layer_kind):
                x = inputs[l]
                ins[l] = {"q": O.bf16_to_f64(x["q"][t0:t1]), "k": O.bf16_to_f64(x["k"][t0:t1]),
                          "v": O.bf16_to_f64(x["v"][t0:t1])}
                if kind == W.GDN:
                    ins[l]["alpha"] = O.f32_to_f64(x["alpha"][t0:t1])
                    ins[l]["beta"] = O.f32_to_f64(x["beta"][t0:t1])
            pos_b = None if tail_pos is None else np.asarray(tail_pos[t0:t1], np.int64)
            dl_b = None
            if delim is not None:
                dcu, dbg, den = delim
                dl_b = (list(dbg[dcu[b]:dcu[b + 1]]), list(den[dcu[b]:dcu[b + 1]]))
            n_delim = 0 if dl_b is None else int(sum(e - a for a, e in zip(*dl_b)))
            outs, new = O.maintenance_round(self.oracle[b], s.layer_kind, bb, ee, ins, s.rotary_dim,
                                            s.rope_theta, positions=pos_b, delimiters=dl_b,
                                            conv_weights=self.conv_w)
            for l in outs:
                ora_out[l][t0:t1] = outs[l]
            self.oracle[b] = new
            # bookkeeping
            L_new = L_before[b] - int(np.sum(np.asarray(ee) - np.asarray(bb)))
            live, cur = self.ctx.get_live(b)
            assert live == L_new + (t1 - t0) - n_delim, (b, live, L_new)
            if tail_pos is None:
                assert cur == cur_before[b] + (t1 - t0)
            assert new.cursor == cur
            keep_idx = np.nonzero(O.keep_mask(L_before[b], bb, ee))[0]
            assert np.array_equal(gather_np[g_off:g_off + L_new], keep_idx), f"gather map char {b}"
            g_off += L_new
            if check_bitexact:
                for l in s.attn_layers:
                    k0, v0, p0 = pre[(l, b)]
                    k1, v1 = self.ctx.get_kv(l, b)
                    k1, v1 = torch_bf16_bits(k1), torch_bf16_bits(v1)
                    p1 = self.ctx.get_positions(b).cpu().numpy()
                    assert np.array_equal(k1[:, :L_new], k0[:, keep_idx]), f"K compaction layer {l} char {b}"
                    assert np.array_equal(v1[:, :L_new], v0[:, keep_idx]), f"V compaction layer {l} char {b}"
                    assert np.array_equal(p1[:L_new], p0[keep_idx]), f"positions layer {l} char {b}"
                    if tail_pos is None and delim is None:
                        assert np.array_equal(p1[L_new:], np.arange(cur_before[b], cur_before[b] + t1 - t0)), \
                            f"tail positions char {b}"
                    assert np.array_equal(p1, new.caches[l].pos.astype(np.int32)), f"positions char {b}"
                    # appended rotated keys and values against the oracle's fp64 ones
                    if new.caches[l].live > L_new:
                        errs[("append_k", l, b)] = rel_l2(O.bf16_to_f64(k1[:, L_new:]), new.caches[l].K[:, L_new:])
                        assert np.array_equal(O.bf16_to_f64(v1[:, L_new:]), new.caches[l].V[:, L_new:])
        # the bar holds per (layer, character) for outputs and per (layer,
        # character, head) for states, so that one wrong character or head
        # cannot hide under the others' norm
        for l in dev_out:
            for b in range(B):
                t0, t1 = tail_cu[b], tail_cu[b + 1]
                if t1 > t0:
                    errs[("out", l, b)] = rel_l2(gpu_out[l][t0:t1], ora_out[l][t0:t1])
        if self.conv_w is not None:
            # the carried conv state holds raw bf16 inputs: bit-exact
            for l in s.gdn_layers:
                cs = O.bf16_to_f64(torch_bf16_bits(self.ctx.get_conv_state(l)))
                for b in range(B):
                    assert np.array_equal(cs[b], self.oracle[b].conv[l]), f"conv state layer {l} char {b}"
        for l in s.gdn_layers:
            S_gpu = self.ctx.get_state(l).cpu().numpy().astype(np.float64)
            for b in range(B):
                for h in range(s.n_gdn_heads):
                    errs[("S", l, b, h)] = rel_l2(S_gpu[b, h], self.oracle[b].states[l][h])
        return errs
