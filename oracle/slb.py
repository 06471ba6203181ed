"""Plain model of the semantic lookaside buffer's INT8 scan and margin gate
(Sec. IV-A; the 0.0136 threshold and the ~20 % escalation rate are given
there, the latencies in Table III).

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU baseline may use it.

The paper states that tool embeddings are INT8-quantized and scanned with an
integer dot product, that the two best candidates are compared, and that a
margin above the calibrated threshold routes to the best one while a smaller
margin escalates to a cross-encoder (not modelled: it needs trained weights).
Readings where it is silent (listed in the design notes):

* quantization is symmetric and per vector: scale = max|x| / 127, code =
  round-half-even(x / scale), in [-127, 127]; an all-zero vector has scale 0
  and zero codes. The query is quantized the same way.
* score(q, t) = float32(dot of the codes) * (scale_q * scale_t), the product of
  the scales formed first, all in float32. Floating point here decides an
  integer (which tool ranks first), so the oracle takes those decisions in the
  kernel's precision, float32; the dot itself is exact (|dot| < 2^24).
* candidates are ordered by score, higher first, then by lower tool index.
* margin = top-1 score - top-2 score in float32; the decision routes to the
  top-1 tool when margin > tau, else escalates. With a single tool there is no
  runner-up: it always routes.
"""
from __future__ import annotations

from typing import List, Tuple

import numpy as np

__all__ = ["slb_quantize", "slb_scores", "slb_top2", "slb_route"]

TAU = np.float32(0.0136)


def slb_quantize(x) -> Tuple[np.ndarray, np.ndarray]:
    """Rows of x [n][dim] -> (int8 codes [n][dim], float32 scales [n])."""
    x = np.asarray(x, dtype=np.float32)
    n = x.shape[0]
    codes = np.zeros(x.shape, dtype=np.int8)
    scales = np.zeros(n, dtype=np.float32)
    for i in range(n):
        amax = np.float32(np.max(np.abs(x[i]))) if x.shape[1] else np.float32(0)
        if amax == 0:
            continue
        s = np.float32(amax / np.float32(127.0))
        q = np.rint(x[i] / s)                 # float32 division, round half to even
        codes[i] = np.clip(q, -127, 127).astype(np.int8)
        scales[i] = s
    return codes, scales


def slb_scores(q_codes, q_scales, t_codes, t_scales) -> np.ndarray:
    """float32 scores [n_queries][n_tools] of the rule above."""
    # Integer dot products: every product and partial sum is an integer of
    # magnitude at most 4096 * 128^2 = 2^26, far below 2^53, so a float64 matrix
    # product computes them exactly.
    qc = np.asarray(q_codes, dtype=np.float64)
    tc = np.asarray(t_codes, dtype=np.float64)
    dots = qc @ tc.T
    c = (np.asarray(q_scales, dtype=np.float32)[:, None] *
         np.asarray(t_scales, dtype=np.float32)[None, :])   # float32 products of the scales
    return dots.astype(np.float32) * c


def slb_top2(scores_row) -> List[Tuple[int, np.float32]]:
    """The two best (index, score) pairs of one query; fewer if fewer tools."""
    order = sorted(range(len(scores_row)), key=lambda j: (-float(scores_row[j]), j))
    return [(j, np.float32(scores_row[j])) for j in order[:2]]


def slb_route(q_codes, q_scales, t_codes, t_scales, tau=TAU):
    """Per query: (top-1 index, top-2 index or -1, top-1 score, top-2 score or
    -inf, routed tool or -1 when the margin gate escalates)."""
    s = slb_scores(q_codes, q_scales, t_codes, t_scales)
    out = []
    for a in range(s.shape[0]):
        top = slb_top2(s[a])
        i1, s1 = top[0]
        if len(top) > 1:
            i2, s2 = top[1]
        else:
            i2, s2 = -1, np.float32(-np.inf)
        margin = np.float32(s1 - s2)
        out.append((i1, i2, s1, s2, i1 if margin > np.float32(tau) else -1))
    return out
