"""Pins of the decode-attention oracle (one new query token attending to a
cache, Sec. 3.2 last sentence).  Each check targets a plausible slip: a
missing 1/sqrt(D), a sign or operand swap, the wrong KV head for a query head,
a softmax over the wrong axis, a missing normalisation."""

import math

import numpy as np
import pytest

import oracle
from synth.gen import f32_to_bf16_bits


def bf(x):
    return f32_to_bf16_bits(np.asarray(x, np.float32))


def rand_bits(rng, shape, scale=1.0):
    return bf(rng.standard_normal(shape) * scale)


def test_single_key_returns_its_value():
    rng = np.random.default_rng(0)
    q, k, v = rand_bits(rng, (1, 2, 128)), rand_bits(rng, (1, 1, 128)), rand_bits(rng, (1, 1, 128))
    out = oracle.decode_attention(q, k, v, [0, 1], 2, 1)
    np.testing.assert_array_equal(out[0, 0], oracle.bf16_to_f64(v[0, 0]))
    np.testing.assert_array_equal(out[0, 1], oracle.bf16_to_f64(v[0, 0]))


def test_two_keys_closed_form_pins_scale_and_sign():
    # q = 2 e0, k1 = 3 e0, k2 = 0: logits 6/sqrt(128) and 0, so the weight of
    # v1 is the logistic 1 / (1 + exp(-6/sqrt(128))) = 0.6295...
    D = 128
    q = np.zeros((1, 1, D)); q[0, 0, 0] = 2.0
    k = np.zeros((2, 1, D)); k[0, 0, 0] = 3.0
    rng = np.random.default_rng(1)
    v = rand_bits(rng, (2, 1, D))
    out = oracle.decode_attention(bf(q), bf(k), v, [0, 2], 1, 1)[0, 0]
    w = 1.0 / (1.0 + math.exp(-6.0 / math.sqrt(D)))
    vv = oracle.bf16_to_f64(v)
    np.testing.assert_allclose(out, w * vv[0, 0] + (1 - w) * vv[1, 0], rtol=1e-12, atol=1e-15)
    # swapping the keys swaps the weights
    out2 = oracle.decode_attention(bf(q), bf(k[::-1].copy()), v, [0, 2], 1, 1)[0, 0]
    np.testing.assert_allclose(out2, (1 - w) * vv[0, 0] + w * vv[1, 0], rtol=1e-12, atol=1e-15)


def test_uniform_cases_give_the_mean_value():
    rng = np.random.default_rng(2)
    v = rand_bits(rng, (7, 2, 128))
    mean = oracle.bf16_to_f64(v).mean(axis=0)
    q = rand_bits(rng, (1, 4, 128))
    k_same = np.repeat(rand_bits(rng, (1, 2, 128)), 7, axis=0)
    out = oracle.decode_attention(q, k_same, v, [0, 7], 4, 2)
    np.testing.assert_allclose(out[0, 0], mean[0], rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(out[0, 3], mean[1], rtol=1e-12, atol=1e-14)
    out0 = oracle.decode_attention(np.zeros_like(q), rand_bits(rng, (7, 2, 128)), v, [0, 7], 4, 2)
    np.testing.assert_allclose(out0[0, 1], mean[0], rtol=1e-12, atol=1e-14)


def test_invariances():
    rng = np.random.default_rng(3)
    q, k, v = rand_bits(rng, (1, 4, 128)), rand_bits(rng, (9, 2, 128)), rand_bits(rng, (9, 2, 128))
    k[:, :, 5] = 0                     # so that the shift below is exact in bf16
    base = oracle.decode_attention(q, k, v, [0, 9], 4, 2)
    perm = rng.permutation(9)
    np.testing.assert_allclose(oracle.decode_attention(q, k[perm], v[perm], [0, 9], 4, 2), base, rtol=1e-12,
                               atol=1e-14)
    # the same shift of every key moves all logits of a head by one constant
    kf = oracle.bf16_to_f64(k)
    shift = np.zeros(128); shift[5] = 4.0
    k_shift = bf((kf + shift[None, None, :]).astype(np.float32))
    assert np.array_equal(oracle.bf16_to_f64(k_shift), kf + shift[None, None, :])
    np.testing.assert_allclose(oracle.decode_attention(q, k_shift, v, [0, 9], 4, 2), base, rtol=1e-10, atol=1e-12)
    # linear in V
    v2 = rand_bits(rng, (9, 2, 128))
    vs = bf(oracle.bf16_to_f64(v) * 0.5)
    lin = oracle.decode_attention(q, k, vs, [0, 9], 4, 2) + oracle.decode_attention(q, k, v2, [0, 9], 4, 2)
    both = oracle.bf16_to_f64(vs) + oracle.bf16_to_f64(v2)
    assert np.all(np.isfinite(both))
    # attention of the summed values equals the sum of attentions (sum computed exactly in fp64 here)
    q64, k64 = oracle.bf16_to_f64(q), oracle.bf16_to_f64(k)
    x = k64[:, 0, :] @ q64[0, 1] / math.sqrt(128)
    p = np.exp(x - x.max()); p /= p.sum()
    np.testing.assert_allclose(lin[0, 1], p @ both[:, 0, :], rtol=1e-10, atol=1e-12)


def test_grouped_query_heads_read_contiguous_kv_groups():
    rng = np.random.default_rng(4)
    q, k, v = rand_bits(rng, (1, 4, 128)), rand_bits(rng, (6, 2, 128)), rand_bits(rng, (6, 2, 128))
    gqa = oracle.decode_attention(q, k, v, [0, 6], 4, 2)
    mha = oracle.decode_attention(q, k[:, [0, 0, 1, 1]], v[:, [0, 0, 1, 1]], [0, 6], 4, 4)
    np.testing.assert_allclose(gqa, mha, rtol=1e-12)
    inter = oracle.decode_attention(q, k[:, [0, 1, 0, 1]], v[:, [0, 1, 0, 1]], [0, 6], 4, 4)
    assert not np.allclose(gqa, inter)


def test_brute_force_ragged_batch():
    # explicit loops with math.exp and math.fsum, no max subtraction
    rng = np.random.default_rng(5)
    lens = [3, 0, 5]
    cu = np.concatenate([[0], np.cumsum(lens)])
    D, hq, hkv = 8, 2, 1
    q, k, v = rand_bits(rng, (3, hq, D)), rand_bits(rng, (8, hkv, D)), rand_bits(rng, (8, hkv, D))
    got = oracle.decode_attention(q, k, v, cu, hq, hkv)
    qf, kf, vf = oracle.bf16_to_f64(q), oracle.bf16_to_f64(k), oracle.bf16_to_f64(v)
    for b in range(3):
        for h in range(hq):
            if lens[b] == 0:
                assert np.all(got[b, h] == 0)
                continue
            ws = [math.exp(math.fsum(qf[b, h, d] * kf[j, 0, d] for d in range(D)) / math.sqrt(D))
                  for j in range(cu[b], cu[b + 1])]
            z = math.fsum(ws)
            for d in range(D):
                ref = math.fsum(w * vf[j, 0, d] for w, j in zip(ws, range(cu[b], cu[b + 1]))) / z
                assert got[b, h, d] == pytest.approx(ref, rel=1e-12, abs=1e-14)
