"""Analytic prefill cost of a pruning schedule (A-PACK App. G, "FLOPs Accounting").

One decoder layer at sequence length n costs (Eq. perlayer)

    phi(n) = 4 n d^2 + 2 n^2 d + 2 n d m

(the four attention projections, the quadratic attention, the feed-forward
block; d = hidden size, m = FFN width).  Prefill sums phi over the actual
per-layer lengths n_1 .. n_T (Eq. prefill) and the FLOPs ratio divides by T
layers at the uncompressed length n_0 (Eq. ratio).

A pruning step at layer l uses that layer's attention to score the tokens, so
layer l itself still runs at the length it entered with and layers after it
run at the pruned length.  Host arithmetic only; no device code.
"""

from dataclasses import dataclass
from typing import Iterable, List, Sequence, Tuple


@dataclass(frozen=True)
class Thinker:
    layers: int     # T
    hidden: int     # d
    ffn: int        # m


# The constants App. G gives for the Qwen2.5-Omni thinker.
QWEN25_OMNI_7B = Thinker(layers=28, hidden=3584, ffn=18944)
QWEN25_OMNI_3B = Thinker(layers=36, hidden=2048, ffn=11008)


def phi(n: float, model: Thinker) -> float:
    """FLOPs of one decoder layer at length n (Eq. perlayer)."""
    d, m = model.hidden, model.ffn
    return 4.0 * n * d * d + 2.0 * n * n * d + 2.0 * n * d * m


def layer_schedule(n0: int, steps: Iterable[Tuple[int, int]], model: Thinker) -> List[int]:
    """Lengths n_1 .. n_T entering each layer (layers numbered 0 .. T-1 here).

    steps: (layer l, tokens after the step) for every pruning step, ascending.
    Layers up to and including l run at the length before the step."""
    n = [n0] * model.layers
    for layer, after in sorted(steps):
        for i in range(layer + 1, model.layers):
            n[i] = after
    return n


def prefill_flops(schedule: Sequence[int], model: Thinker) -> float:
    """F_pre = sum over layers of phi(n_i) (Eq. prefill)."""
    if len(schedule) != model.layers:
        raise ValueError("one length per layer expected")
    return float(sum(phi(n, model) for n in schedule))


def flops_ratio(schedule: Sequence[int], n0: int, model: Thinker) -> float:
    """rho = F_pre / (T phi(n_0)) (Eq. ratio)."""
    return prefill_flops(schedule, model) / (model.layers * phi(n0, model))
