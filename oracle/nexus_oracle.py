"""Plain fp64 CPU oracle for the Nexus KV-cache splicing hot path.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline / reference arm of ``bench.py`` may import this module. The product
path (the CUDA library and its Python binding) never imports, links or calls
it, and this module imports nothing from the product.

Every function is the plain definition from the paper written out in NumPy
float64, slow and obvious on purpose. Inputs are the same bf16 bit patterns
the GPU receives, widened exactly to float64.

Sources (the paper: "Nexus: Depth-Adaptive KV-Cache Splicing and
Retrieval-Decoupled Tool Routing for Agentic LLMs on Unified Memory"):

* RoPE and its base frequencies theta_i = b^(-2i/d), b = 1e6 ......... Sec. III-B
* phase drift Delta theta_i = (n_past - m0) theta_i ................. Sec. III-B, Eq. 1
* reanchoring: rotate each transplanted key by delta = n_past - m0 ... Sec. III-B
* anchored splice (delta = 0) is output-exact ....................... Sec. IV-A
* depth-adaptive recompute fraction R(n_past) ....................... Sec. III-C, Eq. 2
* redecoded suffix length ceil(S * R / 100) ......................... Sec. V-A
* scaled dot-product attention softmax(QK^T / sqrt(d)) V ............ Sec. III-A
* R = 100 % is numerically a full prefill ........................... Sec. III-C
* attention-logit soft-capping (models with token-innermost V) ....... Sec. V-B
* the re-decoded suffix tokens' fresh Q, K, V (projection, RoPE) ..... Sec. V-A, Sec. III-B

Readings taken where the paper is silent (each is listed in the design
notes): NeoX half-split pairs (i, i + d/2) by default with GPT-J interleaved
pairs as an option; rotation by +delta; delta = 0 is a pure copy; a block
inserted at depth p displaces the later rows, which move by +L and are
re-rotated by +L; query t of a suffix of R sits at position T - R + t and sees
keys j <= its position; query head h reads KV head floor(h / group).
"""
from __future__ import annotations

import math
from fractions import Fraction

import numpy as np

__all__ = [
    "bf16_bits_to_f64",
    "rope_inv_freq",
    "rope_rotate",
    "rerotate",
    "recompute_pct",
    "redecode_len",
    "splice_sequence",
    "paged_gather",
    "attention",
    "suffix_positions",
    "qkv_recompute",
]


# --------------------------------------------------------------------------
# dtype plumbing: bf16 bit patterns -> float64 (exact widening)
# --------------------------------------------------------------------------
def bf16_bits_to_f64(bits) -> np.ndarray:
    """Widen bf16 bit patterns (uint16 / int16 array) exactly to float64.

    A bf16 number is the upper 16 bits of an IEEE float32, so shifting the
    pattern left by 16 gives the float32 with the same value.
    """
    b = np.asarray(bits).astype(np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------
# RoPE (Sec. III-B)
# --------------------------------------------------------------------------
def rope_inv_freq(head_dim: int, theta_base: float = 1.0e6,
                  freq_scale: float = 1.0) -> np.ndarray:
    """theta_i = freq_scale * b^(-2i/d) for i = 0 .. d/2 - 1 (Sec. III-B).

    ``freq_scale`` is the linear position-scaling parameter a compiled block
    header records; the runtime model uses 1.0.
    """
    i = np.arange(head_dim // 2, dtype=np.float64)
    return freq_scale * np.power(np.float64(theta_base), -2.0 * i / head_dim)


def rope_rotate(x, pos, theta_base: float = 1.0e6, freq_scale: float = 1.0,
                rope_type: str = "neox") -> np.ndarray:
    """Rotate every feature pair i of ``x[..., d]`` by the angle pos * theta_i.

    ``pos`` broadcasts against ``x.shape[:-1]``. For pair (a, b) and angle t the
    result is (a cos t - b sin t, a sin t + b cos t) (Sec. III-B). ``neox`` pairs
    feature i with i + d/2; ``gptj`` pairs 2i with 2i + 1.
    """
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    ang = np.asarray(pos, dtype=np.float64)[..., None] * rope_inv_freq(d, theta_base, freq_scale)
    c, s = np.cos(ang), np.sin(ang)
    out = np.empty(np.broadcast_shapes(x.shape, ang.shape[:-1] + (d,)), dtype=np.float64)
    if rope_type == "neox":
        a, b = x[..., :half], x[..., half:]
        out[..., :half] = a * c - b * s
        out[..., half:] = a * s + b * c
    elif rope_type == "gptj":
        a, b = x[..., 0::2], x[..., 1::2]
        out[..., 0::2] = a * c - b * s
        out[..., 1::2] = a * s + b * c
    else:
        raise ValueError(f"unknown rope_type {rope_type!r}")
    return out


def rerotate(k, delta: int, theta_base: float = 1.0e6, freq_scale: float = 1.0,
             rope_type: str = "neox") -> np.ndarray:
    """Reanchor keys compiled at m0 to m0 + delta (Sec. III-B, Eq. 1).

    Rotating by +delta undoes the phase error (n_past - m0) theta_i of Eq. 1.
    delta = 0 is the anchored splice, which the paper states is output-exact
    (Sec. IV-A): it is a plain copy of the bits, with no arithmetic at all.
    """
    k = np.asarray(k, dtype=np.float64)
    if int(delta) == 0:
        return k.copy()
    return rope_rotate(k, int(delta), theta_base, freq_scale, rope_type)


# --------------------------------------------------------------------------
# Depth-adaptive recompute policy (Sec. III-C, Eq. 2; Sec. V-A)
# --------------------------------------------------------------------------
def recompute_pct(n_past: int, M: int = 256, R_base=5, K: int = 4) -> Fraction:
    """R(n_past) of Eq. 2 in exact rational arithmetic, clamped to 100 %.

    R = R_base for n_past <= M, else R_base + (n_past - M) / (M (K - 1)) *
    (100 - R_base). M is the splice threshold P, K the multiple of M at which
    recompute reaches 100 %.
    """
    if K < 2 or M < 1:
        raise ValueError("Eq. 2 needs K >= 2 and M >= 1")
    R_base = Fraction(R_base)
    if n_past <= M:
        return R_base
    r = R_base + Fraction(n_past - M, M * (K - 1)) * (100 - R_base)
    return min(r, Fraction(100))


def redecode_len(S: int, n_past: int, M: int = 256, R_base=5, K: int = 4) -> int:
    """Number of trailing tokens invalidated and re-decoded: ceil(S R / 100) (Sec. V-A)."""
    r = recompute_pct(n_past, M, R_base, K)
    return min(int(S), math.ceil(Fraction(int(S)) * r / 100))


# --------------------------------------------------------------------------
# Splice (Sec. III-B reanchoring, Sec. V-A splice at the cursor)
# --------------------------------------------------------------------------
def splice_sequence(live_k, live_v, inserts, theta_base: float = 1.0e6,
                    freq_scale: float = 1.0, rope_type: str = "neox"):
    """Logical post-splice K and V of one sequence.

    ``live_k``/``live_v``: [n_layers][n_past][H][d]; ``inserts``: a list of
    (p, block_k, block_v, m0) with p the depth in the original sequence
    (0 <= p <= n_past, non-decreasing), block arrays [n_layers][L][H][d] and m0
    the block's compile anchor. The result is live[0:p1] ++ block1 ++
    live[p1:p2] ++ block2 ++ ... ++ live[pk:n_past]. Block rows are reanchored
    by delta = (new position) - m0; displaced live rows are re-rotated by the
    number of block rows inserted before them. V rows are copied unchanged.
    """
    live_k = np.asarray(live_k, dtype=np.float64)
    live_v = np.asarray(live_v, dtype=np.float64)
    n_past = live_k.shape[1]
    ks, vs = [], []
    cursor = 0          # next unread live row
    shift = 0           # block rows inserted so far
    for p, bk, bv, m0 in inserts:
        if p < cursor or p > n_past:
            raise ValueError("insert depths must be non-decreasing and <= n_past")
        ks.append(rerotate(live_k[:, cursor:p], shift, theta_base, freq_scale, rope_type))
        vs.append(live_v[:, cursor:p].copy())
        new_pos = p + shift
        ks.append(rerotate(bk, new_pos - m0, theta_base, freq_scale, rope_type))
        vs.append(np.asarray(bv, dtype=np.float64).copy())
        shift += np.asarray(bk).shape[1]
        cursor = p
    ks.append(rerotate(live_k[:, cursor:n_past], shift, theta_base, freq_scale, rope_type))
    vs.append(live_v[:, cursor:n_past].copy())
    return np.concatenate(ks, axis=1), np.concatenate(vs, axis=1)


def paged_gather(pool, page_table, n_tokens: int, page_size: int = 16,
                 token_innermost: bool = False) -> np.ndarray:
    """Read a logical [n_layers][n_tokens][H][d] sequence out of a paged pool.

    Row-major pool: [n_layers][n_pages][H][page_size][d]; token-innermost
    (transposed-V) pool: [n_layers][n_pages][H][d][page_size]. Position t lives
    in page ``page_table[t // page_size]`` at slot ``t % page_size``.
    """
    pool = np.asarray(pool)
    pt = np.asarray(page_table)
    pos = np.arange(n_tokens)
    pages = pt[pos // page_size]
    slots = pos % page_size
    if token_innermost:
        g = pool[:, pages, :, :, slots]          # [n_tokens][n_layers][H][d]
    else:
        g = pool[:, pages, :, slots, :]          # [n_tokens][n_layers][H][d]
    return np.moveaxis(g, 0, 1)


# --------------------------------------------------------------------------
# Attention (Sec. III-A) over a suffix of queries (Sec. III-C, Sec. V-A)
# --------------------------------------------------------------------------
def suffix_positions(T: int, R: int) -> np.ndarray:
    """Positions of the last R tokens of a T-token cache: T - R + t."""
    return np.arange(T - R, T, dtype=np.int64)


def attention(q, k, v, q_pos, group: int, softcap=None):
    """Causal GQA attention, the plain definition softmax(QK^T / sqrt(d)) V.

    q [R][Hq][d]; k, v [T][Hkv][d]; query t sees keys j <= q_pos[t]; query head
    h reads KV head h // group. Returns (o [R][Hq][d], lse [R][Hq]) with
    lse = log sum_j exp(s_j) over the visible keys, s_j = q.k_j / sqrt(d).

    ``softcap`` (attention-logit soft-capping of the models whose V cache is
    token-innermost, Sec. V-B): the scaled score s is replaced by
    softcap * tanh(s / softcap) before the softmax.
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    q_pos = np.asarray(q_pos, dtype=np.int64)
    R, Hq, d = q.shape
    T = k.shape[0]
    visible = np.arange(T)[None, :] <= q_pos[:, None]          # [R][T]
    o = np.zeros((R, Hq, d))
    lse = np.zeros((R, Hq))
    for h in range(Hq):
        kv = h // group
        s = (q[:, h, :] @ k[:, kv, :].T) / math.sqrt(d)       # [R][T]
        if softcap is not None:
            s = softcap * np.tanh(s / softcap)
        s = np.where(visible, s, -np.inf)
        m = s.max(axis=1, keepdims=True)
        e = np.exp(s - m)
        z = e.sum(axis=1, keepdims=True)
        o[:, h, :] = (e / z) @ v[:, kv, :]
        lse[:, h] = m[:, 0] + np.log(z[:, 0])
    return o, lse


# --------------------------------------------------------------------------
# Re-decoding the suffix: fresh Q, K, V of the invalidated tokens (Sec. V-A)
# --------------------------------------------------------------------------
def qkv_recompute(x, w_qkv, b_qkv, positions, n_q_heads: int, n_kv_heads: int,
                  theta_base: float = 1.0e6, freq_scale: float = 1.0, rope_type: str = "neox"):
    """Q, K, V of re-decoded tokens at the given positions (Sec. V-A, Sec. III-B).

    x [R][hidden]; w_qkv [(Hq + 2 Hkv) d][hidden] (output features, input
    features); b_qkv [(Hq + 2 Hkv) d] or None. y = x w_qkv^T + b is split, in
    this order, into Q (Hq heads), K (Hkv heads) and V (Hkv heads) of d = 128
    features; Q and K are rotated at each token's position, V is not.
    Returns q [R][Hq][d], k [R][Hkv][d], v [R][Hkv][d].
    """
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(w_qkv, dtype=np.float64)
    y = x @ w.T
    if b_qkv is not None:
        y = y + np.asarray(b_qkv, dtype=np.float64)[None, :]
    R = x.shape[0]
    d = w.shape[0] // (n_q_heads + 2 * n_kv_heads)
    q = y[:, : n_q_heads * d].reshape(R, n_q_heads, d)
    k = y[:, n_q_heads * d: (n_q_heads + n_kv_heads) * d].reshape(R, n_kv_heads, d)
    v = y[:, (n_q_heads + n_kv_heads) * d:].reshape(R, n_kv_heads, d)
    pos = np.asarray(positions, dtype=np.float64)[:, None]
    q = rope_rotate(q, pos, theta_base, freq_scale, rope_type)
    k = rope_rotate(k, pos, theta_base, freq_scale, rope_type)
    return q, k, v
