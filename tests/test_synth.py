"""The seeded generator: published SplitMix64 outputs, moments, layouts."""

import numpy as np

from synth import workload, WORKLOADS
from synth.gen import splitmix64, normal_bf16_bits, bf16_bits_to_f32, f32_to_bf16_bits


def test_splitmix64_published_sequence():
    # Reference outputs of the SplitMix64 generator seeded with 1234567
    # (state advanced by the golden gamma before each mix).
    expect = [6457827717110365317, 3203168211198807973, 9817491932198370423,
              4593380528125082431, 16408922859458223821]
    gamma = 0x9E3779B97F4A7C15
    got = [int(splitmix64(np.uint64((1234567 + i * gamma) % 2 ** 64))) for i in range(5)]
    assert got == expect


def test_normal_moments_and_chunk_independence():
    a = bf16_bits_to_f32(normal_bf16_bits(7, 2001, 0, 1 << 20)).astype(np.float64)
    assert abs(a.mean()) < 5e-3 and abs(a.var() - 1.0) < 1e-2
    assert np.abs(a).max() <= 3.47
    b = normal_bf16_bits(7, 2001, 1000, 5000, chunk=333)
    np.testing.assert_array_equal(b, normal_bf16_bits(7, 2001, 0, 6000)[1000:])


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e-3], np.float32)
    # 1 + 2^-8 is a tie -> even (1.0); 1 + 3*2^-8 is a tie -> 1 + 2^-6
    np.testing.assert_array_equal(bf16_bits_to_f32(f32_to_bf16_bits(x))[:4],
                                  np.array([1.0, 1.0, 1.015625, -2.5], np.float32))


def test_workload_layouts():
    w = workload("tiny")
    m = w.modality()
    assert m.size == 1298 and (m == 1).sum() == 250 and (m == 2).sum() == 1000
    assert w.cu_qlens().tolist() == [0, 32]
    assert workload("7b_10min").total_tokens == 135272
    assert workload("3b_60s").total_tokens == 16 + 1500 + 7200 + 64
    r = workload("7b_ragged16")
    assert r.num_seqs == 16
    for s, (ra, rv) in zip(r.seqs, r.ratios[0]):
        assert 30 <= s.duration_s <= 300 and s.duration_s % 2 == 0 and 16 <= s.n_q <= 256
        assert 0.2 <= ra <= 0.6 and 0.2 <= rv <= 0.6
    assert len(WORKLOADS) == 7 and WORKLOADS['7b_10min_1l'].total_tokens == 135272
    p = WORKLOADS['7b_10min_paper']
    assert p.prune_layers == list(range(14, 28)) and p.seqs[0].n_q == 1 and p.joint_step_keep == 0.85
