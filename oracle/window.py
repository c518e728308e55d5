"""Re-anchored audio window of the draft's cross-attention (float64, numpy).

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and the CPU legs of ``bench.py`` may import it.

What it computes (App. "Attention conditions" and "Window geometry"): the
restricted arms let the draft attend to a fixed-width window of encoder frames
that differ only in its centre.  The half-width is 400 ms; the shifted centre
moves 500 ms forward and is clipped to the valid audio grid; the random centre
is uniform over that grid with seed 0.  The deployed correction takes the
centre from verification attention: the anchor frame the verify step returns
(Sec. 5 "Verification-Attention Correction").

Reading (the paper's grid is the 80 ms one of its Qwen and Voxtral analyses;
this decoder's encoder frames are Whisper's, 30 s / 1500 = 20 ms): a half-width
of 20 frames and a shift of 25 frames; the window [c - 20, c + 20] (41 frames)
clipped to [0, T); the clipped shifted centre min(c + 25, T - 1).
"""
from __future__ import annotations

import numpy as np

from oracle.decoder import softmax

FRAME_MS = 20.0
HALF_WIDTH_MS = 400.0
SHIFT_MS = 500.0
RANDOM_SEED = 0


def frames(ms: float) -> int:
    """Milliseconds on the encoder grid, in whole frames."""
    return int(round(ms / FRAME_MS))


def window_center(kind: str, anchor: int, T: int, rng: np.random.Generator = None) -> int:
    """Centre of the window for one draft round: "anchor" (the verification
    anchor), "shifted" (500 ms later, clipped to the grid) or "random" (uniform
    over the grid, from `rng`, seeded with 0 by default)."""
    if T < 1:
        raise ValueError("no encoder frames")
    if kind == "anchor":
        return int(min(max(anchor, 0), T - 1))
    if kind == "shifted":
        return int(min(max(anchor, 0) + frames(SHIFT_MS), T - 1))
    if kind == "random":
        rng = rng if rng is not None else np.random.default_rng(RANDOM_SEED)
        return int(rng.integers(0, T))
    raise ValueError(kind)


def window(center: int, T: int) -> tuple:
    """Frames [lo, hi) the restricted cross-attention may read: the centre plus
    and minus the half-width, clipped to [0, T)."""
    h = frames(HALF_WIDTH_MS)
    return max(center - h, 0), min(center + h + 1, T)


def windowed_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray, n_heads: int, lo: int, hi: int) -> np.ndarray:
    """Multi-head attention of one query over the encoder frames [lo, hi) only
    (q [d]; K, V [T, d], head h in columns h*hd:(h+1)*hd).  Returns [d]."""
    Kw, Vw = K[lo:hi], V[lo:hi]
    n, d = Kw.shape
    hd = d // n_heads
    s = np.einsum("hc,nhc->hn", q.reshape(n_heads, hd), Kw.reshape(n, n_heads, hd)) / np.sqrt(hd)
    return np.einsum("hn,nhc->hc", softmax(s), Vw.reshape(n, n_heads, hd)).reshape(d)
