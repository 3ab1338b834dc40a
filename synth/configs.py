"""The five audio-video workloads of the prune step, as token layouts and shapes.

Everything here is input description: sequence layouts, model shapes, the
pruning schedule and the keep ratios a caller passes in.  Turning ratios into
keep counts and everything after that belongs to the method (the library and
the oracle each do it on their own).

Token layout of one sequence (stated choice; the paper fixes none):
``[n_sys system tokens] [chunk 0] ... [chunk C-1] [n_q text-query tokens]``
where each 2-second chunk holds its video frames first (``fps * 2`` frames of
``tpf`` visual tokens) and then its audio (25 tokens/s * 2 s = 50 tokens).
Audio runs at 25 tokens per second, the rate the paper reports for the
Qwen2.5-Omni audio encoder (Sec. D).  Modality codes: 0 = system/text/query
(never pruned), 1 = audio, 2 = visual.
"""

from dataclasses import dataclass, field
from typing import List, Tuple

import numpy as np

from .gen import uniform_u32, TID_RAGGED

MOD_OTHER, MOD_AUDIO, MOD_VISUAL = 0, 1, 2
AUDIO_RATE = 25          # tokens per second
CHUNK_S = 2              # seconds per interleave chunk


@dataclass(frozen=True)
class SeqLayout:
    duration_s: int
    fps: int               # video frames per second after pre-LLM compression
    tpf: int               # visual tokens per frame
    n_q: int               # text-query tokens (the query span, at the end)
    n_sys: int = 16

    @property
    def n_audio(self) -> int:
        return AUDIO_RATE * self.duration_s

    @property
    def n_visual(self) -> int:
        return self.fps * self.duration_s * self.tpf

    @property
    def length(self) -> int:
        return self.n_sys + self.n_audio + self.n_visual + self.n_q

    def modality(self) -> np.ndarray:
        assert self.duration_s % CHUNK_S == 0
        parts = [np.zeros(self.n_sys, np.uint8)]
        vis = np.full(self.fps * CHUNK_S * self.tpf, MOD_VISUAL, np.uint8)
        aud = np.full(AUDIO_RATE * CHUNK_S, MOD_AUDIO, np.uint8)
        for _ in range(self.duration_s // CHUNK_S):
            parts.append(vis)
            parts.append(aud)
        parts.append(np.zeros(self.n_q, np.uint8))
        m = np.concatenate(parts)
        assert m.size == self.length
        return m


@dataclass(frozen=True)
class Plant:
    """Shift ``count`` keys of one modality by ``amp * sqrt(D)`` along the
    unit mean query direction of their KV-head group (on every pruning layer)."""
    modality: int
    count: int
    amp: float


@dataclass
class Workload:
    name: str
    seed: int
    num_layers: int          # decoder layers L
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    hidden: int
    seqs: List[SeqLayout]
    prune_layers: List[int]  # pruning layers, ascending
    # ratios[step][seq] = (audio keep, visual keep), cumulative w.r.t. the
    # counts entering the first step
    ratios: List[List[Tuple[float, float]]]
    plants: List[List[Plant]] = field(default_factory=list)  # per sequence
    # joint selection over S with a per-step keep fraction of the current |S|
    # (the paper's form); when set, `ratios` is unused
    joint_step_keep: float = None

    @property
    def num_seqs(self) -> int:
        return len(self.seqs)

    def modality(self) -> np.ndarray:
        return np.concatenate([s.modality() for s in self.seqs])

    def cu_seqlens(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum([s.length for s in self.seqs])]).astype(np.int32)

    def cu_qlens(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum([s.n_q for s in self.seqs])]).astype(np.int32)

    def compact_layers(self, step: int) -> int:
        """KV layers compacted at a step: layers [l, L) of the pruning layer l."""
        return self.num_layers - self.prune_layers[step]

    @property
    def total_tokens(self) -> int:
        return int(sum(s.length for s in self.seqs))

    @property
    def total_mm(self) -> int:
        return int(sum(s.n_audio + s.n_visual for s in self.seqs))


def _qwen7b(**kw):
    return dict(num_layers=28, num_q_heads=28, num_kv_heads=4, head_dim=128, hidden=3584, **kw)


def _qwen3b(**kw):
    return dict(num_layers=36, num_q_heads=16, num_kv_heads=2, head_dim=128, hidden=2048, **kw)


def _ragged_seqs(seed: int, n: int):
    """Ragged batch draws: duration an even number of seconds uniform in
    [30, 300]; query length uniform in [16, 256]; keep ratios per (sequence,
    modality) uniform in [0.2, 0.6] on a 1e-3 grid."""
    seqs, ratios = [], []
    for b in range(n):
        u = uniform_u32(seed, TID_RAGGED, np.arange(4 * b, 4 * b + 4, dtype=np.uint64)).astype(np.int64)
        dur = 30 + 2 * int(u[0] % 136)              # 30, 32, ..., 300
        n_q = 16 + int(u[1] % 241)                  # 16 .. 256
        ra = (200 + int(u[2] % 401)) / 1000.0       # 0.200 .. 0.600
        rv = (200 + int(u[3] % 401)) / 1000.0
        seqs.append(SeqLayout(duration_s=dur, fps=2, tpf=100, n_q=n_q))
        ratios.append((ra, rv))
    return seqs, ratios


def _build() -> dict:
    w = {}
    # 1: tiny single-layer step, 7B heads, 10 s at 1 fps x 100 tokens/frame.
    s1 = SeqLayout(duration_s=10, fps=1, tpf=100, n_q=32)
    w["tiny"] = Workload(
        name="tiny", seed=0, **{**_qwen7b(), "num_layers": 1}, seqs=[s1],
        prune_layers=[0], ratios=[[(0.5, 0.3)]],
        plants=[[Plant(1, 8, 0.5), Plant(2, 20, 0.5)]])
    # 2: 3B-shaped 60-s clip, 2 fps x 60 tokens/frame, prune at layer 10.
    s2 = SeqLayout(duration_s=60, fps=2, tpf=60, n_q=64)
    w["3b_60s"] = Workload(
        name="3b_60s", seed=1, **_qwen3b(), seqs=[s2], prune_layers=[10],
        ratios=[[(0.5, 0.25)]],
        plants=[[Plant(1, 15, 0.5), Plant(2, 72, 0.5)]])
    # 3: 7B-shaped 2-min clip, progressive at layers 4/12/20.
    s3 = SeqLayout(duration_s=120, fps=2, tpf=100, n_q=128)
    w["7b_2min"] = Workload(
        name="7b_2min", seed=2, **_qwen7b(), seqs=[s3], prune_layers=[4, 12, 20],
        ratios=[[(0.7, 0.4)], [(0.5, 0.25)], [(0.3, 0.15)]],
        plants=[[Plant(1, 30, 0.5), Plant(2, 240, 0.5)]])
    # 4: 7B-shaped 10-min video, heavy-tailed plants (5% at +1.0, 0.1% at +3.0).
    s4 = SeqLayout(duration_s=600, fps=2, tpf=100, n_q=256)
    w["7b_10min"] = Workload(
        name="7b_10min", seed=3, **_qwen7b(), seqs=[s4], prune_layers=[4, 12, 20],
        ratios=[[(0.7, 0.4)], [(0.5, 0.25)], [(0.3, 0.15)]],
        plants=[[Plant(1, 750, 1.0), Plant(2, 6000, 1.0),
                 Plant(1, 15, 3.0), Plant(2, 120, 3.0)]])
    # 4 on one layer: the 10-minute sequence pruned once at the last layer (one
    # compacted K/V layer); same scoring and selection work as the first step of
    # 7b_10min with a device footprint of about 2 GB (profiling captures).
    w["7b_10min_1l"] = Workload(
        name="7b_10min_1l", seed=3, **_qwen7b(), seqs=[s4], prune_layers=[27],
        ratios=[[(0.7, 0.4)]],
        plants=[[Plant(1, 750, 1.0), Plant(2, 6000, 1.0),
                 Plant(1, 15, 3.0), Plant(2, 120, 3.0)]])
    # The paper's own inner-LLM setting on the 10-minute sequence: the last query
    # token only, one top-k over all of S, pruning at every layer from L_mid = 14
    # (depth / 2) to 27 with P = 15% of the current |S| per layer (25% tier).
    s4q = SeqLayout(duration_s=600, fps=2, tpf=100, n_q=1)
    w["7b_10min_paper"] = Workload(
        name="7b_10min_paper", seed=5, **_qwen7b(), seqs=[s4q], prune_layers=list(range(14, 28)),
        ratios=[], joint_step_keep=0.85,
        plants=[[Plant(1, 750, 1.0), Plant(2, 6000, 1.0),
                 Plant(1, 15, 3.0), Plant(2, 120, 3.0)]])
    # 5: ragged batch of 16 7B-shaped sequences, prune at layer 8.
    seqs5, r5 = _ragged_seqs(4, 16)
    w["7b_ragged16"] = Workload(
        name="7b_ragged16", seed=4, **_qwen7b(), seqs=seqs5, prune_layers=[8],
        ratios=[r5],
        plants=[[Plant(1, s.n_audio // 100, 0.5), Plant(2, s.n_visual // 100, 0.5)] for s in seqs5])
    return w


WORKLOADS = _build()


def workload(name: str) -> Workload:
    return WORKLOADS[name]


def scaled_copy(wl: Workload, duration_s: int, n_q: int = None, name: str = None) -> Workload:
    """The same model shapes and schedule on one shorter sequence (used for
    bounded CPU samples and small parity cases).  Plant counts scale with the
    number of tokens of each modality."""
    base = wl.seqs[0]
    s = SeqLayout(duration_s=duration_s, fps=base.fps, tpf=base.tpf,
                  n_q=base.n_q if n_q is None else n_q, n_sys=base.n_sys)
    plants = []
    for p in wl.plants[0]:
        n_m = base.n_audio if p.modality == MOD_AUDIO else base.n_visual
        n_s = s.n_audio if p.modality == MOD_AUDIO else s.n_visual
        plants.append(Plant(p.modality, max(1, (p.count * n_s) // n_m), p.amp))
    return Workload(name=name or f"{wl.name}@{duration_s}s", seed=wl.seed, num_layers=wl.num_layers,
                    num_q_heads=wl.num_q_heads, num_kv_heads=wl.num_kv_heads, head_dim=wl.head_dim,
                    hidden=wl.hidden, seqs=[s], prune_layers=list(wl.prune_layers),
                    ratios=[[r[0]] for r in wl.ratios], plants=[plants], joint_step_keep=wl.joint_step_keep)


def sequence_subset(wl: Workload, seq_ids, name: str = None) -> Workload:
    """The workload restricted to the sequences ``seq_ids`` (ascending), with their own
    layouts, plants and keep ratios: one rank's share of a batch split by sequence."""
    ids = [int(i) for i in seq_ids]
    return Workload(name=name or f"{wl.name}[{','.join(map(str, ids))}]", seed=wl.seed, num_layers=wl.num_layers,
                    num_q_heads=wl.num_q_heads, num_kv_heads=wl.num_kv_heads, head_dim=wl.head_dim,
                    hidden=wl.hidden, seqs=[wl.seqs[i] for i in ids], prune_layers=list(wl.prune_layers),
                    ratios=[[r[i] for i in ids] for r in wl.ratios],
                    plants=[wl.plants[i] for i in ids] if wl.plants else [],
                    joint_step_keep=wl.joint_step_keep)
