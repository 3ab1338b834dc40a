"""CPU oracle of A-PACK's pre-LLM frame alignment score (test infrastructure only).

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` leg of ``bench.py`` may use it; it shares no code with the
CUDA path.

Sec. 3.1, "Coarse pass" and "Gated fine pass" (Eq. cka, Eq. gate; Algorithm 1,
the first five steps), in fp64 from exactly widened bf16 embeddings:

* v_f: mean of the visual tokens of frame f; a_f: the audio sequence resampled
  onto the frame axis.  Reading taken: audio token j belongs to frame
  floor(j * F / N_a) and a_f is the mean of the audio tokens of frame f
  (requires N_a >= F so that every frame has one).
* Window W_f = {f - w//2, ..., f + w//2} cut to the clip [0, F) at its ends
  (reading); A_f, V_f stack the window's a and v rows, each centred by its
  mean over the window rows.
* c_f = ||V_f^T A_f||_F^2 / (||A_f^T A_f||_F ||V_f^T V_f||_F)  (Eq. cka, linear
  CKA), computed literally with the d x d products; a window whose centred rows
  are all zero has no defined CKA and scores 0 (reading).
* d_f = ||v_f - a_f||_2, the direct distance of the frame's visual tokens to the
  audio tokens (reading: Euclidean distance of the pooled embeddings);
  d^_f = (d_f - min d) / (max d - min d) over the clip (0 when all are equal).
* c-bar = mean of c_f; s_f = c_f if c-bar >= tau, else (1 - beta) c_f +
  beta (1 - d^_f)  (Eq. gate; Algorithm 1 writes the comparison as c-bar <= tau,
  the equation's strict form is taken).  Defaults tau = 0.78, beta = 0.90
  (Table S-hparams).
"""

import numpy as np

from .apack_oracle import bf16_to_f64

TAU_DEFAULT = 0.78
BETA_DEFAULT = 0.90
WINDOW_DEFAULT = 3


def frame_embeddings(visual_bits, audio_bits, n_frames, tokens_per_frame):
    """(v [F, d], a [F, d]) fp64 frame embeddings from bf16 token rows."""
    v_tok = bf16_to_f64(visual_bits).reshape(n_frames, tokens_per_frame, -1)
    a_tok = bf16_to_f64(audio_bits)
    n_a = a_tok.shape[0]
    if n_a < n_frames:
        raise ValueError("fewer audio tokens than frames")
    v = v_tok.mean(axis=1)
    frame_of = (np.arange(n_a) * n_frames) // n_a
    a = np.stack([a_tok[frame_of == f].mean(axis=0) for f in range(n_frames)])
    return v, a


def window_cka(a, v, window=WINDOW_DEFAULT):
    """c_f of Eq. cka for every frame (literal d x d products)."""
    F = a.shape[0]
    half = window // 2
    c = np.zeros(F)
    for f in range(F):
        lo, hi = max(0, f - half), min(F, f + half + 1)
        A = a[lo:hi] - a[lo:hi].mean(axis=0, keepdims=True)
        V = v[lo:hi] - v[lo:hi].mean(axis=0, keepdims=True)
        den = np.linalg.norm(A.T @ A) * np.linalg.norm(V.T @ V)
        c[f] = np.linalg.norm(V.T @ A) ** 2 / den if den > 0 else 0.0
    return c


def gate(c, v, a, tau=TAU_DEFAULT, beta=BETA_DEFAULT):
    """(s_f of Eq. gate, d^_f, c-bar)."""
    d = np.linalg.norm(v - a, axis=1)
    span = d.max() - d.min()
    dn = (d - d.min()) / span if span > 0 else np.zeros_like(d)
    cbar = float(c.mean())
    s = c.copy() if cbar >= tau else (1.0 - beta) * c + beta * (1.0 - dn)
    return s, dn, cbar


def frame_alignment(visual_bits, audio_bits, n_frames, tokens_per_frame, window=WINDOW_DEFAULT,
                    tau=TAU_DEFAULT, beta=BETA_DEFAULT):
    v, a = frame_embeddings(visual_bits, audio_bits, n_frames, tokens_per_frame)
    c = window_cka(a, v, window)
    s, dn, cbar = gate(c, v, a, tau, beta)
    return dict(c=c, s=s, dnorm=dn, cbar=cbar, v=v, a=a)
