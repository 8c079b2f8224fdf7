"""The seeded input generator: published SplitMix64 outputs, value distribution,
special-pattern rate, determinism and the workload shapes."""
import numpy as np

import synth

GOLDEN = 0x9E3779B97F4A7C15


def test_splitmix64_published_outputs():
    # First five outputs of SplitMix64 seeded with 1234567 (Vigna's reference
    # implementation, as quoted alongside the xoshiro generators), and the first
    # output from state 0.
    lib = synth.host_lib()
    want = [6457827717110365317, 3203168211198807973, 9817491932198370423,
            4593380528125082431, 16408922859458223821]
    got = [lib.synth_splitmix64((1234567 + i * GOLDEN) % (1 << 64)) for i in range(5)]
    assert got == want
    assert lib.synth_splitmix64(0) == 0xE220A8397B1DCDAF


def test_distribution():
    v = synth.values_host(4_000_000, 4, seed=3).view(np.float32).astype(np.float64)
    assert abs(v.mean()) < 1e-4
    assert abs(v.std() - 0.02) < 2e-4
    # Irwin-Hall of 4 is bounded: |x| <= 131070 * scale ~ 3.46 sd.
    assert np.abs(v).max() <= 131070 * np.float32(0.02 / 37837) * 1.0000001


def test_specials_rate_and_table():
    table = synth.special_table()
    n = 3_000_000
    v = synth.values_host(n, 4, seed=1, specials=True)
    frac = np.isin(v, table).mean()
    # 1% target; binomial sd at n = 3e6 is ~6e-5 (a normal value equal to a table
    # entry is essentially impossible).
    assert abs(frac - 0.01) < 5e-4
    # Each pattern shows up.
    assert set(np.unique(v[np.isin(v, table)])) == set(table)


def test_bf16_is_upper_half_and_deterministic():
    a = synth.values_host(100_000, 4, seed=9, first_idx=12345)
    b = synth.values_host(100_000, 2, seed=9, first_idx=12345)
    np.testing.assert_array_equal(b, (a >> 16).astype(np.uint16))
    np.testing.assert_array_equal(a, synth.values_host(100_000, 4, seed=9, first_idx=12345))
    idx = np.array([12345, 12346, 99999 + 12345], np.int64)
    np.testing.assert_array_equal(synth.gather_host(idx, 4, seed=9), a[[0, 1, 99999]])
    assert not np.array_equal(a, synth.values_host(100_000, 4, seed=10, first_idx=12345))


def _count(shape):
    H, hd = shape.hidden, shape.head_dim
    attn = (shape.n_q * hd * H) * 2 + (shape.n_kv * hd * H) * 2 + 2 * hd
    mlp = (shape.n_experts * 3 * shape.moe_intermediate * H + shape.n_experts * H
           if shape.moe else 3 * shape.intermediate * H)
    per_layer = attn + mlp + 2 * H
    return shape.vocab * H * (1 if shape.tied else 2) + shape.layers * per_layer + H


def test_workload_parameter_counts():
    # Exact parameter counts of the five model shapes.
    assert _count(synth.TINY) == 1_975_808
    assert _count(synth.QWEN3_0_6B) == 596_049_920
    assert _count(synth.QWEN3_8B) == 8_190_735_360
    assert _count(synth.QWEN3_30B_A3B) == 30_532_122_624
