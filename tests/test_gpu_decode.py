"""Decode-step attention over a KV cache on the GPU against the fp64 oracle
(one decode token per sequence, Sec. 3.2 last sentence).

Tolerance: logits are fp32 dot products of 128 exactly widened bf16 products
(error ~1e-6), probabilities use the hardware exp2 (relative error ~1e-7), and
the weighted sums of up to 1.4e5 values run in fp32 in chunks of a few hundred
keys before an fp32 merge; |gpu - oracle| <= 2e-4 + 2e-3 |oracle| covers that
with margin, while leaving out one key of a few thousand (a change of order
1e-3 of the output scale) fails it."""

import numpy as np
import pytest
import torch

import oracle
from synth.gen import f32_to_bf16_bits

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ap():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_08794_gb300 as ap
    return ap


def bits(rng, shape, scale=1.0):
    return f32_to_bf16_bits((rng.standard_normal(shape) * scale).astype(np.float32))


def run(ap, cu, q, k, v, hq, hkv, pad_heads=0):
    """k, v: uint16 [T, Hkv, 128]; pad_heads > 0 places them in wider token rows."""
    T = k.shape[0]
    row = (hkv + pad_heads) * 128
    kd = torch.zeros(max(T, 1), row, dtype=torch.int16, device="cuda")
    vd = torch.zeros_like(kd)
    if T:
        kd[:, :hkv * 128] = torch.from_numpy(k.reshape(T, -1).view(np.int16)).cuda()
        vd[:, :hkv * 128] = torch.from_numpy(v.reshape(T, -1).view(np.int16)).cuda()
    qd = torch.from_numpy(q.view(np.int16)).cuda()
    out = torch.full((len(cu) - 1, hq, 128), float("nan"), dtype=torch.float32, device="cuda")
    ws = torch.zeros(max(256, ap.apack_decode_workspace_size(cu, hq, hkv)), dtype=torch.uint8, device="cuda")
    ap.apack_decode_attention(cu, qd, kd, vd, row * 2, hq, hkv, out, ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    return out.cpu().numpy()


def check(got, ref):
    np.testing.assert_allclose(got, ref, atol=2e-4, rtol=2e-3)


CASES = [
    ([1], 28, 4),
    ([7, 64, 65, 1000, 0, 4099], 28, 4),      # ragged, one empty cache
    ([5000, 333], 16, 2),                    # 3B heads
    ([2000], 8, 8),                          # one query head per KV head
    ([3000], 8, 1),                          # 8 query heads share one KV head
    ([100, 200, 300], 12, 4),                # 3 rows per group
]


@pytest.mark.parametrize("lens,hq,hkv", CASES)
def test_decode_attention_matches_oracle(ap, lens, hq, hkv):
    rng = np.random.default_rng(sum(lens) + hq)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    q = bits(rng, (len(lens), hq, 128))
    k = bits(rng, (T, hkv, 128), 1.5)        # peaky softmax
    v = bits(rng, (T, hkv, 128))
    got = run(ap, cu, q, k, v, hq, hkv)
    ref = oracle.decode_attention(q, k, v, cu, hq, hkv)
    check(got, ref)
    again = run(ap, cu, q, k, v, hq, hkv)
    if hkv in (2, 4) and hq // hkv <= 8:
        # tensor-core path: tiles are claimed as the CTAs go, so two calls may group the keys'
        # partial sums differently; both meet the rule and agree to fp32 rounding
        check(again, ref)
        np.testing.assert_allclose(again, got, rtol=1e-4, atol=1e-6)
    else:                                    # CUDA-core path: a fixed split and merge order
        assert got.tobytes() == again.tobytes()


def test_decode_attention_strided_rows_and_uniform_keys(ap):
    rng = np.random.default_rng(7)
    cu = np.array([0, 777, 1500], np.int32)
    q = bits(rng, (2, 28, 128))
    k = np.repeat(bits(rng, (1, 4, 128)), 1500, axis=0)     # identical keys: plain mean of V
    v = bits(rng, (1500, 4, 128))
    got = run(ap, cu, q, k, v, 28, 4, pad_heads=3)
    ref = oracle.decode_attention(q, k, v, cu, 28, 4)
    check(got, ref)
    vf = oracle.bf16_to_f64(v)
    np.testing.assert_allclose(ref[1, 27], vf[777:1500, 3].mean(axis=0), rtol=1e-12, atol=1e-14)


def test_decode_attention_full_ten_minute_cache(ap):
    # the uncompressed 10-minute 7B cache (135272 tokens) and its final compacted length
    rng = np.random.default_rng(8)
    for T in (135272, 22772):
        cu = np.array([0, T], np.int32)
        q = bits(rng, (1, 28, 128))
        k = bits(rng, (T, 4, 128))
        v = bits(rng, (T, 4, 128))
        check(run(ap, cu, q, k, v, 28, 4), oracle.decode_attention(q, k, v, cu, 28, 4))


def test_decode_attention_rejects_unsupported_groups(ap):
    rng = np.random.default_rng(9)
    cu = np.array([0, 10], np.int32)
    with pytest.raises(ap.ApackError):
        ap.apack_decode_workspace_size(cu, 32, 2)            # 16 query rows per KV head
    with pytest.raises(ap.ApackError):
        ap.apack_decode_workspace_size(np.array([0, 5, 3], np.int32), 28, 4)   # decreasing offsets


def test_decode_attention_batch_beyond_one_launch(ap):
    # 70 sequences: the chunk and combine kernels run in two launches
    rng = np.random.default_rng(70)
    lens = [int(x) for x in rng.integers(0, 700, 70)]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    q = bits(rng, (70, 28, 128))
    k = bits(rng, (T, 4, 128), 1.5)
    v = bits(rng, (T, 4, 128))
    check(run(ap, cu, q, k, v, 28, 4), oracle.decode_attention(q, k, v, cu, 28, 4))


@pytest.mark.parametrize("hq,hkv", [(28, 4), (16, 2)])
def test_decode_attention_rising_and_falling_maxima(ap, hq, hkv):
    # Row j of every head group reads feature j of the keys (q = 8 e_j, so a key value x gives
    # a logit of about 1.02 x in log2 units).  Feature j steps by 12 every 128 keys with period
    # 5 blocks: up for even rows (a new maximum about 2^12 above the previous one at every
    # block of a chunk), down for odd rows (the first block holds the maximum), plus one spike
    # late in row 1.  Long sequences, so that every chunk of keys spans several blocks.
    G = hq // hkv
    rng = np.random.default_rng(11 + hq)
    lens = [40000, 9001]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    qf = np.zeros((len(lens), hq, 128), np.float32)
    for h in range(hq):
        qf[:, h, h % G] = 8.0
    kf = rng.standard_normal((T, hkv, 128)).astype(np.float32) * 0.25
    for b, n in enumerate(lens):
        step = (np.arange(n) // 128) % 5
        for j in range(G):
            kf[cu[b]:cu[b + 1], :, j] = (12.0 * step if j % 2 == 0 else 12.0 * (4 - step))[:, None]
        kf[cu[b] + n - 5, :, 1] = 70.0
    q = f32_to_bf16_bits(qf)
    k = f32_to_bf16_bits(kf)
    v = bits(rng, (T, hkv, 128))
    got = run(ap, cu, q, k, v, hq, hkv)
    check(got, oracle.decode_attention(q, k, v, cu, hq, hkv))


def test_decode_attention_repeated_calls_on_one_workspace(ap):
    # On the tensor-core path the CTAs of a sequence claim its tiles from counters at the end of
    # the workspace, and the combine kernel zeroes them again: after every call they must read
    # zero, and every call must meet the rule (the tiles' split over CTAs varies between calls).
    rng = np.random.default_rng(2024)
    lens = [30011, 0, 4097, 1, 129]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    q = bits(rng, (len(lens), 28, 128))
    k = bits(rng, (T, 4, 128), 1.5)
    v = bits(rng, (T, 4, 128))
    ref = oracle.decode_attention(q, k, v, cu, 28, 4)
    kd = torch.from_numpy(k.reshape(T, -1).view(np.int16)).cuda()
    vd = torch.from_numpy(v.reshape(T, -1).view(np.int16)).cuda()
    qd = torch.from_numpy(q.view(np.int16)).cuda()
    n_ws = ap.apack_decode_workspace_size(cu, 28, 4)
    ws = torch.zeros(n_ws, dtype=torch.uint8, device="cuda")
    cl0 = n_ws - (len(lens) * 4 + 255) // 256 * 256          # the claim counters: the last region
    for _ in range(12):
        out = torch.full((len(lens), 28, 128), float("nan"), dtype=torch.float32, device="cuda")
        ap.apack_decode_attention(cu, qd, kd, vd, 4 * 256, 28, 4, out, ws)
        torch.cuda.synchronize()
        assert ap.apack_device_error(ws) == ap.APACK_OK
        assert not ws[cl0:cl0 + 4 * len(lens)].any()
        check(out.cpu().numpy(), ref)


RANDOM_HEADS = [(28, 4), (16, 2), (12, 4), (32, 4), (8, 2), (8, 8), (8, 1), (4, 4)]


@pytest.mark.parametrize("seed", range(16))
def test_random_decode_matches_oracle(ap, seed):
    # random batches: one to eight sequences of 0 to 20000 cached tokens (some empty, some shorter
    # than one 128-key tile), every supported head layout (the tensor-core path for Hkv 2 or 4,
    # the CUDA-core path otherwise), key scales from flat to peaky softmax, and a token-row
    # stride wider than the heads in half the cases
    rng = np.random.default_rng(9000 + seed)
    hq, hkv = RANDOM_HEADS[seed % len(RANDOM_HEADS)]
    B = int(rng.integers(1, 9))
    lens = [0 if rng.random() < 0.1 else int(rng.choice([rng.integers(1, 130), rng.integers(1, 20000)]))
            for _ in range(B)]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    q = bits(rng, (B, hq, 128))
    k = bits(rng, (T, hkv, 128), float(rng.choice([0.3, 1.0, 2.0])))
    v = bits(rng, (T, hkv, 128))
    got = run(ap, cu, q, k, v, hq, hkv, pad_heads=int(rng.integers(0, 2)))
    check(got, oracle.decode_attention(q, k, v, cu, hq, hkv))
