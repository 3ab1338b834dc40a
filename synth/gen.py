"""Counter-based generator: value = f(seed, tensor id, element index).

Definition (so that a CUDA twin produces the same bits, see ``fill.cu``):

* ``splitmix64(x)`` is the SplitMix64 finaliser of Steele, Lea and Flood
  ("Fast splittable pseudorandom number generators", OOPSLA 2014), the same
  mixing function Vigna publishes for seeding xoshiro generators:
  ``z = x + 0x9E3779B97F4A7C15; z = (z ^ z>>30) * 0xBF58476D1CE4E5B9;
  z = (z ^ z>>27) * 0x94D049BB133111EB; return z ^ z>>31`` (mod 2^64).
* the stream key of a tensor is ``key = splitmix64(splitmix64(seed) ^ tid)``;
  element ``i`` draws ``h = splitmix64(key ^ splitmix64(i))``.
* a standard-normal-like bf16 value is the Irwin-Hall sum of the four 16-bit
  words of ``h``: ``s = sum(words) - 131070`` (an exact integer), scaled in
  float32 by ``1/sqrt((2^32-1)/3)`` (unit variance) and rounded to bf16 with
  round-to-nearest-even.  Integer steps plus one correctly rounded float32
  multiply make the result bit-identical on any IEEE machine and on the GPU.
  The distribution has mean 0, variance 1 and support of +-3.46.

Tensor ids keep distinct streams apart: ``tid = kind * 1000 + layer``.
"""

import numpy as np

TID_Q = 1000        # query rows of layer l: TID_Q + l
TID_K = 2000        # key cache of layer l
TID_V = 3000        # value cache of layer l
TID_HIDDEN = 4000   # hidden states
TID_PLANT = 5000    # which tokens are planted
TID_RAGGED = 6000   # per-sequence draws of the ragged batch
TID_POS = 7000      # position ids
TID_VIS_EMB = 8000  # visual encoder embeddings (pre-LLM alignment)
TID_AUD_EMB = 8001  # audio encoder embeddings (pre-LLM alignment)

_M64 = np.uint64(0xFFFFFFFFFFFFFFFF)
_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_MUL1 = np.uint64(0xBF58476D1CE4E5B9)
_MUL2 = np.uint64(0x94D049BB133111EB)

# float32(1 / sqrt((2**32 - 1) / 3)); the scale that gives the Irwin-Hall sum
# of four 16-bit uniforms unit variance.
NORMAL_SCALE_F32 = np.float32(1.0 / np.sqrt((2.0 ** 32 - 1.0) / 3.0))


def splitmix64(x):
    """SplitMix64 finaliser on uint64 scalars or arrays (wrapping arithmetic)."""
    with np.errstate(over="ignore"):
        z = np.asarray(x, dtype=np.uint64) + _GOLDEN
        z = (z ^ (z >> np.uint64(30))) * _MUL1
        z = (z ^ (z >> np.uint64(27))) * _MUL2
        return z ^ (z >> np.uint64(31))


def stream_key(seed, tid):
    return splitmix64(splitmix64(np.uint64(seed)) ^ np.uint64(tid))


def hash_stream(seed, tid, index):
    """64-bit hash of element ``index`` (array of uint64) of stream (seed, tid)."""
    key = stream_key(seed, tid)
    return splitmix64(key ^ splitmix64(np.asarray(index, dtype=np.uint64)))


def uniform_u32(seed, tid, index):
    """Upper 32 bits of the element hash (uniform integers)."""
    return (hash_stream(seed, tid, index) >> np.uint64(32)).astype(np.uint32)


def f32_to_bf16_bits(x):
    """float32 -> bf16 bit pattern (uint16), round to nearest even (finite input)."""
    b = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))
    return (b >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b):
    """bf16 bit pattern (uint16) -> float32 (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16_bits(seed, tid, start, count, chunk=1 << 22):
    """``count`` bf16 values (as uint16 bits) of stream (seed, tid) from ``start``."""
    out = np.empty(count, dtype=np.uint16)
    for c0 in range(0, count, chunk):
        c1 = min(count, c0 + chunk)
        idx = np.arange(start + c0, start + c1, dtype=np.uint64)
        h = hash_stream(seed, tid, idx)
        s = ((h & np.uint64(0xFFFF)) + ((h >> np.uint64(16)) & np.uint64(0xFFFF))
             + ((h >> np.uint64(32)) & np.uint64(0xFFFF)) + (h >> np.uint64(48)))
        z = (s.astype(np.int64) - 131070).astype(np.float32) * NORMAL_SCALE_F32
        out[c0:c1] = f32_to_bf16_bits(z)
    return out
