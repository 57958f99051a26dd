"""The bench's algorithmic-work accounting, on CPU.

Every roofline fraction the bench reports divides one of these counts by a
measured time, so each formula is checked against a count made the long way
(explicit loops over tokens, heads and keys) and against the per-round
figures of the npc workload (attention ~33 GFLOP and ~21 MB per attention
layer, delta rule 0.4 GFLOP and 6.3 MB per layer, a full compaction rewrite
~34 MB).
"""
from types import SimpleNamespace

import pytest

import bench

NPC = SimpleNamespace(head_dim=256, n_q_heads=16, n_kv_heads=2, d_k=128, d_v=128, n_gdn_heads=16,
                      attn_layers=[3], gdn_layers=[0, 1, 2])


def test_attention_flops_counts_every_score_and_weighted_value():
    s = SimpleNamespace(head_dim=8, n_q_heads=4, n_kv_heads=2)
    Lp, tails = [5, 0, 3], [3, 2, 0]
    brute = 0
    for l, m in zip(Lp, tails):
        for i in range(m):                       # tail token i sees l survivors and tokens 0..i
            for _ in range(s.n_q_heads):
                keys = l + i + 1
                brute += keys * 2 * s.head_dim   # q . k for every visible key
                brute += keys * 2 * s.head_dim   # sum of p_j v_j over the same keys
    assert bench.attention_flops(s, Lp, tails) == brute


def test_attention_bytes_reads_each_survivor_once_per_kv_head():
    s = SimpleNamespace(head_dim=8, n_q_heads=4, n_kv_heads=2)
    Lp, tails = [5, 7, 3], [3, 0, 1]
    brute = 0
    for l, m in zip(Lp, tails):
        if m:
            brute += l * s.n_kv_heads * s.head_dim * 2 * 2          # K and V of the survivors, bf16
        brute += m * s.n_q_heads * s.head_dim * 2 * 2              # q in, output out
        brute += m * s.n_kv_heads * s.head_dim * 2 * 2             # k_new, v_new appended
    assert bench.attention_bytes(s, Lp, tails) == brute


def test_gdn_accounting_by_token_and_head():
    s = SimpleNamespace(d_k=4, d_v=6, n_gdn_heads=3)
    tails = [2, 0, 5]
    flops = bytes_ = 0
    for m in tails:
        for _ in range(m):
            for _ in range(s.n_gdn_heads):
                flops += 6 * s.d_k * s.d_v                          # S k, the rank-1 update, S q
                bytes_ += (2 * s.d_k + 2 * s.d_v) * 2 + 2 * 4       # q, k, v, o bf16; alpha, beta fp32
        if m:
            bytes_ += s.n_gdn_heads * s.d_v * s.d_k * 4 * 2         # S read and written once
    assert bench.gdn_flops(s, tails) == flops
    assert bench.gdn_bytes(s, tails) == bytes_


def test_npc_round_figures():
    Lp, tails = [7782], [256]
    assert bench.attention_flops(NPC, Lp, tails) == pytest.approx(33.18e9, rel=1e-3)
    assert bench.attention_bytes(NPC, Lp, tails) == pytest.approx(20.66e6, rel=1e-3)
    assert bench.gdn_flops(NPC, tails) == pytest.approx(0.4027e9, rel=1e-3)
    assert bench.gdn_bytes(NPC, tails) == 6324224
    assert bench.rope_bytes(NPC, tails) == 256 * (16 + 4) * 256 * 2 * 2
    # a full rewrite of the 8192-entry cache of the one attention layer
    assert bench.compaction_bytes(NPC, 8192) == pytest.approx(33.6e6, rel=1e-3)
