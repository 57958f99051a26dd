"""The seeded generators produce valid, reproducible inputs of the stated shapes."""
import numpy as np
import pytest

from oracle import kvm_oracle as O
from workload import synth as W


@pytest.mark.parametrize("L,total,n", [(512, 64, 2), (8192, 410, 4), (32768, 983, 10), (100, 1, 1),
                                       (10, 9, 1), (10, 5, 5), (2048, 0, 3)])
def test_removal_spans_valid(L, total, n):
    b, e = W.removal_spans((5, L, n), L, total, n)
    O.validate_spans(L, b, e)
    assert int((e - b).sum()) == total
    b2, e2 = W.removal_spans((5, L, n), L, total, n)
    np.testing.assert_array_equal(b, b2)
    np.testing.assert_array_equal(e, e2)


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1 + 2 ** -8, 1 + 3 * 2 ** -8, 1 + 2 ** -8 + 2 ** -30, -3.0e-3, 0.0])
    back = W.bf16_bits_to_f32(W.f64_to_bf16_bits(x)).astype(np.float64)
    np.testing.assert_array_equal(back[:4], [1.0, 1.0, 1 + 2 ** -6, 1 + 2 ** -7])
    assert abs(back[4] + 3.0e-3) <= 3.0e-3 * 2 ** -8


def test_workload_shapes():
    for name in ["tiny", "npc", "long", "pop", "refill"]:
        w = W.make_workload(name)
        assert len(w.plan) == w.rounds
        caps = w.capacity()
        assert all(c >= n for c, n in zip(caps, w.prefix_len))
    w = W.make_workload("tiny")
    ins = W.tail_inputs(w, 0, [64])
    assert ins[1]["q"].shape == (64, 8, 64) and ins[1]["k"].shape == (64, 2, 64)
    k = W.bf16_bits_to_f32(ins[0]["k"]).astype(np.float64)
    np.testing.assert_allclose(np.linalg.norm(k, axis=-1), 1.0, atol=1e-2)
    assert ins[0]["alpha"].dtype == np.float32 and ins[0]["alpha"].shape == (64, 8)
