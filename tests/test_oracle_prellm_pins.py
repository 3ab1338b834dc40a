"""Pins of the pre-LLM alignment oracle (Sec. 3.1, Eq. cka and Eq. gate).

Each check targets a plausible slip: a missing centring, a transposed product,
a wrong norm in the denominator, the wrong window, a reversed gate or blend
weight, an unnormalised distance."""

import numpy as np
import pytest

import oracle
from synth.gen import f32_to_bf16_bits


def bf(x):
    return f32_to_bf16_bits(np.asarray(x, np.float32))


def test_two_row_windows_score_one_and_a_three_row_closed_form():
    # Linear CKA compares the sample (time) Gram structure: two centred rows
    # are +-(x1 - x2)/2 in both streams, so any two-row window scores exactly 1.
    rng = np.random.default_rng(0)
    a, v = rng.standard_normal((2, 16)), rng.standard_normal((2, 16))
    np.testing.assert_allclose(oracle.window_cka(a, v, window=3), [1.0, 1.0], rtol=1e-12)
    # Three rows, worked by hand: a = (1,0), (0,0), (-1,0) (already centred), so
    # K_A = [[1,0,-1],[0,0,0],[-1,0,1]]; v = (1,0), (0,1), (0,0) centres to
    # (2,-1)/3, (-1,2)/3, (-1,-1)/3, so 9 K_V = [[5,-4,-1],[-4,5,-1],[-1,-1,2]].
    # <K_A, K_V> = (5 + 2 + 2)/9 = 1, ||K_A|| = 2, ||K_V|| = sqrt(90)/9.
    a3 = np.array([[1.0, 0.0], [0.0, 0.0], [-1.0, 0.0]])
    v3 = np.array([[1.0, 0.0], [0.0, 1.0], [0.0, 0.0]])
    assert oracle.window_cka(a3, v3, window=3)[1] == pytest.approx(9.0 / (2.0 * np.sqrt(90.0)), rel=1e-12)


def test_identical_streams_give_one_and_invariances_hold():
    rng = np.random.default_rng(1)
    a = rng.standard_normal((9, 32))
    np.testing.assert_allclose(oracle.window_cka(a, a), 1.0, rtol=1e-12)
    v = rng.standard_normal((9, 32))
    base = oracle.window_cka(a, v)
    assert np.all((base >= 0) & (base <= 1 + 1e-12))
    np.testing.assert_allclose(oracle.window_cka(a, 3.0 * v), base, rtol=1e-10)   # isotropic scaling
    qm, _ = np.linalg.qr(rng.standard_normal((32, 32)))
    np.testing.assert_allclose(oracle.window_cka(a @ qm, v @ qm), base, rtol=1e-9)  # orthogonal map
    np.testing.assert_allclose(oracle.window_cka(a + 5.0, v - 2.0), base, rtol=1e-9)  # centring


def test_gram_form_agrees_with_the_feature_form():
    # ||V^T A||_F^2 = <A A^T, V V^T>_F: an independent formula on the same windows
    rng = np.random.default_rng(2)
    a, v = rng.standard_normal((7, 20)), rng.standard_normal((7, 20))
    c = oracle.window_cka(a, v, window=5)
    for f in range(7):
        lo, hi = max(0, f - 2), min(7, f + 3)
        A = a[lo:hi] - a[lo:hi].mean(0)
        V = v[lo:hi] - v[lo:hi].mean(0)
        ka, kv = A @ A.T, V @ V.T
        assert c[f] == pytest.approx((ka * kv).sum() / (np.linalg.norm(ka) * np.linalg.norm(kv)), rel=1e-10)


def test_degenerate_windows_score_zero():
    a = np.ones((4, 8))
    v = np.random.default_rng(3).standard_normal((4, 8))
    assert np.all(oracle.window_cka(a, v) == 0.0)
    assert oracle.window_cka(a[:1], v[:1]).tolist() == [0.0]


def test_gate_branches_weights_and_distance_normalisation():
    rng = np.random.default_rng(4)
    v, a = rng.standard_normal((5, 6)), rng.standard_normal((5, 6))
    c = np.array([0.9, 0.8, 0.95, 0.85, 0.9])            # mean 0.88 >= 0.78: CKA only
    s, dn, cbar = oracle.gate(c, v, a)
    np.testing.assert_array_equal(s, c)
    assert cbar == pytest.approx(0.88)
    d = np.linalg.norm(v - a, axis=1)
    assert dn[np.argmin(d)] == 0.0 and dn[np.argmax(d)] == 1.0
    c2 = np.array([0.1, 0.2, 0.3, 0.4, 0.5])              # mean 0.3 < 0.78: blend
    s2, dn2, _ = oracle.gate(c2, v, a, tau=0.78, beta=0.9)
    np.testing.assert_allclose(s2, 0.1 * c2 + 0.9 * (1.0 - dn2))
    s3, _, _ = oracle.gate(np.full(5, 0.78), v, a)        # equality keeps the CKA branch
    np.testing.assert_array_equal(s3, np.full(5, 0.78))


def test_frame_pooling_and_audio_resampling():
    F, tpf, d = 4, 3, 8
    vis = np.arange(F * tpf * d, dtype=np.float32).reshape(F * tpf, d) / 64
    aud = np.arange(10 * d, dtype=np.float32).reshape(10, d) / 64      # 10 audio tokens over 4 frames
    v, a = oracle.frame_embeddings(bf(vis), bf(aud), F, tpf)
    np.testing.assert_allclose(v[1], vis[3:6].mean(0))
    # floor(j * 4 / 10): frames get audio tokens {0,1,2}, {3,4}, {5,6,7}, {8,9}
    np.testing.assert_allclose(a[0], aud[0:3].mean(0))
    np.testing.assert_allclose(a[1], aud[3:5].mean(0))
    np.testing.assert_allclose(a[3], aud[8:10].mean(0))
    with pytest.raises(ValueError):
        oracle.frame_embeddings(bf(vis), bf(aud[:3]), F, tpf)
