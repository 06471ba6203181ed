"""Pins of the fp64 oracle against facts the paper and mathematics fix.

Each ``pin_*`` takes the oracle routine it checks as an argument and raises
AssertionError when the routine is wrong. ``test_oracle_pins.py`` runs them on
the real oracle; ``test_oracle_mutants.py`` runs them on copies with planted
mistakes (a dropped term, a wrong sign, a wrong index, a transposed operand)
and requires some pin to fail for each.
"""
from __future__ import annotations

import math
import os
from fractions import Fraction

import numpy as np
import torch

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _rs(seed):
    return np.random.default_rng(seed)


# ----------------------------------------------------------------- policy
def load_table1():
    rows = []
    with open(os.path.join(GOLDEN, "table1_recompute_pct.txt")) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if line:
                K, n, r = line.split()
                rows.append((int(K), int(n), r))
    assert len(rows) == 8
    return rows


def pin_table1(recompute_pct):
    """Table I's printed R(%) column, one decimal (Sec. VI-A)."""
    for K, n, printed in load_table1():
        r = recompute_pct(n, M=256, R_base=5, K=K)
        assert f"{float(r):.1f}" == printed, (K, n, float(r), printed)


def pin_eq2_shape(recompute_pct):
    """Eq. 2 boundary facts: flat R_base up to M, reaches exactly 100 at n = K M, clamped after."""
    for K in (2, 3, 4, 16):
        M = 256
        assert recompute_pct(0, M, 5, K) == 5
        assert recompute_pct(M, M, 5, K) == 5
        assert recompute_pct(M + 1, M, 5, K) > 5
        assert recompute_pct(K * M, M, 5, K) == 100
        assert recompute_pct(K * M + 1, M, 5, K) == 100
        assert recompute_pct(10 * K * M, M, 5, K) == 100
        prev = Fraction(0)
        for n in range(0, K * M + 64, 7):
            r = recompute_pct(n, M, 5, K)
            assert r >= prev
            prev = r
        # linear between M and K M: the midpoint gives the midpoint percentage
        mid = M + (K - 1) * M // 2
        if (K - 1) * M % 2 == 0:
            assert recompute_pct(mid, M, 5, K) == Fraction(5 + 100, 2)


def pin_redecode_len(redecode_len, recompute_pct):
    """ceil(S R / 100) (Sec. V-A), checked by searching for the smallest m with 100 m >= S R."""
    for K in (4, 16):
        for n in (0, 100, 256, 257, 300, 511, 512, 513, 700, 1024, 2048, 5000):
            R = recompute_pct(n, 256, 5, K)
            for S in (0, 1, 2, 7, 19, 64, 100, 127, 128, 129, 500, 2192):
                m = 0
                while 100 * m < S * R:
                    m += 1
                assert redecode_len(S, n, 256, 5, K) == min(S, m), (S, n, K)
    # R = 100 % re-decodes everything (the full re-prefill point of Sec. III-C)
    assert redecode_len(2192, 4 * 256, 256, 5, 4) == 2192


# ------------------------------------------------------------------- RoPE
def pin_rope_inv_freq(rope_inv_freq):
    """theta_i = b^(-2i/d): theta_0 = 1, constant ratio b^(-2/d), last = b^(-(d-2)/d)."""
    th = rope_inv_freq(128, 1.0e6, 1.0)
    assert th.shape == (64,)
    assert th[0] == 1.0
    ratio = th[1:] / th[:-1]
    assert np.allclose(ratio, 1.0e6 ** (-2.0 / 128), rtol=1e-13, atol=0)
    assert math.isclose(th[-1], 1.0e6 ** (-126.0 / 128), rel_tol=1e-13)
    th2 = rope_inv_freq(128, 1.0e6, 0.5)
    assert np.allclose(th2, 0.5 * th, rtol=1e-15, atol=0)


def pin_rope_complex(rope_rotate):
    """A rotation of pair (a, b) by t is the complex product (a + i b) e^(i t)."""
    r = _rs(11)
    for d in (2, 8, 128):
        x = r.standard_normal((5, d))
        pos = np.array([0, 1, 7, 300, 30000])
        th = 1.0e6 ** (-2.0 * np.arange(d // 2) / d)
        e = np.exp(1j * pos[:, None] * th[None, :])
        z = (x[:, : d // 2] + 1j * x[:, d // 2:]) * e
        y = rope_rotate(x, pos, 1.0e6, 1.0, "neox")
        assert np.allclose(y[:, : d // 2], z.real, rtol=0, atol=1e-12)
        assert np.allclose(y[:, d // 2:], z.imag, rtol=0, atol=1e-12)
        zg = (x[:, 0::2] + 1j * x[:, 1::2]) * e
        yg = rope_rotate(x, pos, 1.0e6, 1.0, "gptj")
        assert np.allclose(yg[:, 0::2], zg.real, rtol=0, atol=1e-12)
        assert np.allclose(yg[:, 1::2], zg.imag, rtol=0, atol=1e-12)


def pin_rope_2x2(rope_rotate):
    """d = 2: theta_0 = 1 and the map is the textbook matrix [[cos, -sin], [sin, cos]]."""
    for t in (0.0, 1.0, -3.0, 12.0):
        x = np.array([0.3, -1.7])
        c, s = math.cos(t), math.sin(t)
        want = np.array([[c, -s], [s, c]]) @ x
        got = rope_rotate(x[None], np.array([t]), 1.0e6, 1.0, "neox")[0]
        assert np.allclose(got, want, rtol=0, atol=1e-15)


def pin_rope_group(rope_rotate):
    """R(a) R(b) = R(a + b), R(0) = I, pair norms kept, dot products depend on t - s only."""
    r = _rs(12)
    x = r.standard_normal((64, 128))
    a = r.integers(-2000, 2000, size=64)
    b = r.integers(-2000, 2000, size=64)
    lhs = rope_rotate(rope_rotate(x, a), b)
    rhs = rope_rotate(x, a + b)
    assert np.max(np.abs(lhs - rhs)) < 1e-12
    big_a = r.integers(0, 40000, size=64)
    big_b = r.integers(-40000, 40000, size=64)
    assert np.max(np.abs(rope_rotate(rope_rotate(x, big_a), big_b) - rope_rotate(x, big_a + big_b))) < 1e-10
    assert np.array_equal(rope_rotate(x, np.zeros(64, dtype=np.int64)), x)
    y = rope_rotate(x, big_a)
    assert np.allclose(x[:, :64] ** 2 + x[:, 64:] ** 2, y[:, :64] ** 2 + y[:, 64:] ** 2, rtol=1e-12, atol=1e-12)
    q, k = r.standard_normal((2, 128))
    for t, s, c in ((5, 3, 100), (700, 12, 31000), (9000, 8999, -4000)):
        d1 = rope_rotate(q[None], np.array([t]))[0] @ rope_rotate(k[None], np.array([s]))[0]
        d2 = rope_rotate(q[None], np.array([t + c]))[0] @ rope_rotate(k[None], np.array([s + c]))[0]
        assert abs(d1 - d2) < 1e-10


def pin_rerotate(rerotate, rope_rotate):
    """Reanchoring (Sec. III-B): a key compiled at m0 and rotated by p - m0 is the key at p;
    delta = 0 keeps every bit, including -0.0, NaN payloads and infinities (Sec. IV-A)."""
    r = _rs(13)
    raw = r.standard_normal((10, 8, 128))
    for m0, p in ((0, 300), (17, 6000), (4096, 100), (0, 30000)):
        j = np.arange(10)[:, None]
        compiled = rope_rotate(raw, m0 + j)
        assert np.max(np.abs(rerotate(compiled, p - m0) - rope_rotate(raw, p + j))) < 1e-10
    odd = np.array([[-0.0, np.nan, np.inf, -np.inf, 1e-40, -2.5] * 2])
    odd = np.concatenate([odd, np.zeros((1, 116))], axis=1)
    out = rerotate(odd, 0)
    assert np.array_equal(out.view(np.uint64), odd.view(np.uint64))


# ----------------------------------------------------------------- splice
def _raw_session(seed, n_layers, n_past, H=2, d=8):
    r = _rs(seed)
    return r.standard_normal((n_layers, n_past, H, d)), r.standard_normal((n_layers, n_past, H, d))


def pin_splice_closed_form(splice_sequence, rope_rotate):
    """Whatever the insert depths, the spliced cache equals the cache a prefill of the
    spliced token sequence computes: every K row rotated at its final position, V unchanged."""
    r = _rs(14)
    for case in range(6):
        L_layers, H, d = 2, 2, 8
        n_past = int(r.integers(0, 90))
        n_ins = int(r.integers(1, 4))
        depths = np.sort(r.integers(0, n_past + 1, size=n_ins))
        if case == 0:
            depths[:] = n_past          # appended at the cursor, back to back
        raw_live = r.standard_normal((L_layers, n_past, H, d))
        v_live = r.standard_normal((L_layers, n_past, H, d))
        live_k = rope_rotate(raw_live, np.arange(n_past)[None, :, None])
        inserts, raws, vs = [], [], []
        for p in depths:
            L = int(r.integers(1, 40))
            m0 = int(r.integers(0, 50))
            raw_b = r.standard_normal((L_layers, L, H, d))
            v_b = r.standard_normal((L_layers, L, H, d))
            bk = rope_rotate(raw_b, (m0 + np.arange(L))[None, :, None])
            inserts.append((int(p), bk, v_b, m0))
            raws.append(raw_b)
            vs.append(v_b)
        k_out, v_out = splice_sequence(live_k, v_live, inserts)
        # expected: the spliced raw token sequence, rotated at its own positions
        parts_r, parts_v, cur = [], [], 0
        for (p, _, _, _), rb, vb in zip(inserts, raws, vs):
            parts_r += [raw_live[:, cur:p], rb]
            parts_v += [v_live[:, cur:p], vb]
            cur = p
        parts_r.append(raw_live[:, cur:])
        parts_v.append(v_live[:, cur:])
        raw_all = np.concatenate(parts_r, axis=1)
        T = raw_all.shape[1]
        want_k = rope_rotate(raw_all, np.arange(T)[None, :, None])
        assert k_out.shape == want_k.shape
        assert np.max(np.abs(k_out - want_k)) < 1e-10, case
        assert np.array_equal(v_out, np.concatenate(parts_v, axis=1))


def pin_anchored_splice_exact(splice_sequence, rope_rotate):
    """delta = 0 (block compiled at the splice position, appended at the cursor) gives
    a cache byte-identical to the one the prefix computes (Sec. IV-A)."""
    r = _rs(15)
    n_past, L = 37, 21
    raw = r.standard_normal((1, n_past + L, 4, 16))
    v = r.standard_normal((1, n_past + L, 4, 16))
    prefix_k = rope_rotate(raw, np.arange(n_past + L)[None, :, None])
    live_k = prefix_k[:, :n_past]
    block_k = rope_rotate(raw[:, n_past:], (n_past + np.arange(L))[None, :, None])
    k_out, v_out = splice_sequence(live_k, v[:, :n_past], [(n_past, block_k, v[:, n_past:], n_past)])
    assert np.array_equal(k_out.view(np.uint64), prefix_k.view(np.uint64))
    assert np.array_equal(v_out, v)


def pin_paged_gather(paged_gather):
    """Paged layout reading, checked against explicit loops."""
    r = _rs(16)
    nL, nP, H, P, d = 2, 7, 3, 4, 5
    pool = r.standard_normal((nL, nP, H, P, d))
    pt = r.permutation(nP)[:5]
    n = 18
    got = paged_gather(pool, pt, n, page_size=P)
    want = np.zeros((nL, n, H, d))
    for l in range(nL):
        for t in range(n):
            for h in range(H):
                want[l, t, h] = pool[l, pt[t // P], h, t % P]
    assert np.array_equal(got, want)
    poolT = r.standard_normal((nL, nP, H, d, P))
    gotT = paged_gather(poolT, pt, n, page_size=P, token_innermost=True)
    for l in range(nL):
        for t in range(n):
            for h in range(H):
                want[l, t, h] = poolT[l, pt[t // P], h, :, t % P]
    assert np.array_equal(gotT, want)


# -------------------------------------------------------------- attention
def _sdpa(q, k, v, q_pos, group):
    """torch's library scaled_dot_product_attention in float64 on the CPU."""
    R, Hq, d = q.shape
    T = k.shape[0]
    qt = torch.from_numpy(q).permute(1, 0, 2)                                # [Hq][R][d]
    kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(group, 0)     # [Hq][T][d]
    vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(group, 0)
    mask = torch.from_numpy(np.arange(T)[None, :] <= np.asarray(q_pos)[:, None])
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)
    return o.permute(1, 0, 2).numpy()


def pin_attention_library(attention):
    """Equals torch's scaled_dot_product_attention (float64, CPU) with the causal suffix mask,
    and, at R = T, its built-in causal mode (the full prefill of Sec. III-C)."""
    r = _rs(17)
    for R, T, Hkv, group, d in ((5, 9, 2, 3, 16), (1, 1, 1, 5, 8), (12, 12, 2, 2, 32), (7, 40, 3, 5, 128)):
        q = r.standard_normal((R, Hkv * group, d))
        k = r.standard_normal((T, Hkv, d))
        v = r.standard_normal((T, Hkv, d))
        pos = np.arange(T - R, T)
        o, _ = attention(q, k, v, pos, group)
        assert np.max(np.abs(o - _sdpa(q, k, v, pos, group))) < 1e-12
        if R == T:
            qt = torch.from_numpy(q).permute(1, 0, 2)
            kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(group, 0)
            vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(group, 0)
            oc = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
            assert np.max(np.abs(o - oc.permute(1, 0, 2).numpy())) < 1e-12


def pin_suffix_positions(suffix_positions):
    """The re-decoded suffix is the trailing R tokens of a T-token cache (Sec. III-C,
    Sec. V-A): one position per token, R = T is the whole prefill and R = 0 is empty.
    Through torch's library attention: the queries at these positions, each seeing the
    keys at or before its position, give the last R rows of the library's built-in
    causal prefill of all T tokens, which never sees the positions."""
    for T in (1, 2, 9, 300):
        assert np.array_equal(np.asarray(suffix_positions(T, T)), np.arange(T))
        assert len(suffix_positions(T, 0)) == 0
        for R in sorted({1, 2, T // 2, T - 1, T} - {0}):
            pos = np.asarray(suffix_positions(T, R))
            assert pos.shape == (R,)
            assert pos[-1] == T - 1
            assert np.all(np.diff(pos) == 1)
    r = _rs(22)
    T, Hkv, group, d = 23, 2, 3, 16
    q = r.standard_normal((T, Hkv * group, d))
    k = r.standard_normal((T, Hkv, d))
    v = r.standard_normal((T, Hkv, d))
    qt = torch.from_numpy(q).permute(1, 0, 2)
    kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(group, 0)
    vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(group, 0)
    full = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
    full = full.permute(1, 0, 2).numpy()
    for R in (1, 5, 22, 23):
        o = _sdpa(q[T - R:], k, v, suffix_positions(T, R), group)
        assert np.max(np.abs(o - full[T - R:])) < 1e-12


def pin_attention_special(attention):
    """Special cases: a lone visible key returns its value; equal keys give the mean of
    the visible values; one-hot values expose the softmax rows, which are >= 0, zero on
    masked keys and sum to 1; lse is the log-sum-exp of the scaled visible scores."""
    from scipy.special import logsumexp
    r = _rs(18)
    d, T = 16, 9
    q = r.standard_normal((T, 4, d))
    k = r.standard_normal((T, 2, d))
    v = r.standard_normal((T, 2, d))
    o, _ = attention(q[:1], k, v, [0], 2)
    assert np.allclose(o[0], v[0][[0, 0, 1, 1]], atol=1e-14, rtol=0)
    ke = np.repeat(r.standard_normal((1, 2, d)), T, axis=0)
    pos = np.arange(T)
    o, _ = attention(q, ke, v, pos, 2)
    for t in range(T):
        mean = v[: t + 1].mean(axis=0)
        assert np.allclose(o[t], mean[[0, 0, 1, 1]], atol=1e-12, rtol=0)
    # one-hot values: o[t, h, j] = P[t, h, j]
    v1 = np.zeros((T, 2, d))
    for j in range(T):
        v1[j, :, j] = 1.0
    pos = np.array([0, 3, 8])
    o, lse = attention(q[:3], k, v1, pos, 2)
    for t, pt in enumerate(pos):
        for h in range(4):
            row = o[t, h, :T]
            assert np.all(row >= 0)
            assert np.all(row[pt + 1:] == 0)
            assert abs(row.sum() - 1.0) < 1e-13
            s = q[t, h] @ k[: pt + 1, h // 2].T / math.sqrt(d)
            assert abs(lse[t, h] - logsumexp(s)) < 1e-12
            assert np.allclose(row[: pt + 1], np.exp(s - logsumexp(s)), atol=1e-14, rtol=0)


def pin_attention_shift(attention, rope_rotate):
    """Rotating every query and key by an extra c positions leaves attention unchanged:
    scores depend on relative position only (Sec. III-B)."""
    r = _rs(19)
    R, T, d = 4, 20, 128
    q = r.standard_normal((R, 10, d))
    k = r.standard_normal((T, 2, d))
    v = r.standard_normal((T, 2, d))
    pos = np.arange(T - R, T)
    qa = rope_rotate(q, pos[:, None])
    ka = rope_rotate(k, np.arange(T)[:, None])
    o1, l1 = attention(qa, ka, v, pos, 5)
    for c in (1, 999, 30000):
        qb = rope_rotate(q, (pos + c)[:, None])
        kb = rope_rotate(k, (np.arange(T) + c)[:, None])
        o2, l2 = attention(qb, kb, v, pos, 5)
        assert np.max(np.abs(o1 - o2)) < 1e-9
        assert np.max(np.abs(l1 - l2)) < 1e-9


def pin_attention_split(attention):
    """Splitting the visible keys into chunks and merging by log-sum-exp weights
    reproduces the whole: o = sum_s exp(lse_s - lse) o_s."""
    r = _rs(20)
    R, T, d = 6, 50, 32
    q = r.standard_normal((R, 4, d))
    k = r.standard_normal((T, 2, d))
    v = r.standard_normal((T, 2, d))
    pos = np.arange(T - R, T)
    o, lse = attention(q, k, v, pos, 2)
    acc = np.zeros_like(o)
    for a, b in ((0, 17), (17, 40), (40, 50)):
        # chunk [a, b): keys outside the chunk are hidden by shifting them past every query
        kk = k[a:b]
        vv = v[a:b]
        oc, lc = attention(q, kk, vv, pos - a, 2)
        acc += np.exp(lc - lse)[..., None] * oc
    assert np.max(np.abs(acc - o)) < 1e-12


def pin_attention_softcap(attention):
    """Soft-capped scores (Sec. V-B): a very large cap is plain attention; a key
    with an enormous score saturates at +cap, so its weight is the closed form
    e^cap / (e^cap + n_other); caps apply to the 1/sqrt(d)-scaled score."""
    r = _rs(21)
    R, T, d = 5, 30, 64
    q = r.standard_normal((R, 4, d))
    k = r.standard_normal((T, 2, d))
    v = r.standard_normal((T, 2, d))
    pos = np.arange(T - R, T)
    o1, l1 = attention(q, k, v, pos, 2)
    o2, l2 = attention(q, k, v, pos, 2, softcap=1.0e7)
    assert np.max(np.abs(o1 - o2)) < 1e-9 and np.max(np.abs(l1 - l2)) < 1e-9
    # saturation: key 0 aligned with an enormous query, the others orthogonal (score 0)
    cap = 3.0
    qq = np.zeros((1, 1, d)); qq[0, 0, 0] = 1.0e6
    kk = np.zeros((8, 1, d)); kk[0, 0, 0] = 1.0; kk[1:, 0, 1] = 1.0
    vv = np.zeros((8, 1, d)); vv[0, 0, 0] = 1.0
    o, lse = attention(qq, kk, vv, [7], 1, softcap=cap)
    w0 = math.exp(cap) / (math.exp(cap) + 7.0)
    assert abs(o[0, 0, 0] - w0) < 1e-12
    assert abs(lse[0, 0] - math.log(math.exp(cap) + 7.0)) < 1e-12
    # the cap sees the scaled score: s = 2 / sqrt(d) gives cap * tanh(s / cap)
    qq = np.zeros((1, 1, d)); qq[0, 0, 0] = 2.0
    o, lse = attention(qq, kk, vv, [7], 1, softcap=cap)
    s0 = cap * math.tanh((2.0 / math.sqrt(d)) / cap)
    assert abs(lse[0, 0] - math.log(math.exp(s0) + 7.0)) < 1e-12


def pin_qkv_recompute(qkv_recompute, rope_rotate):
    """The re-decoded tokens' projection (Sec. V-A): a one-hot input row picks
    column j of the weight plus the bias (at position 0, where RoPE is the
    identity); Q heads come first, then K, then V; the map is affine in x; Q and
    K at position p are the position-0 vectors rotated by p; V ignores position."""
    r = _rs(22)
    Hq, Hkv, d, hidden = 4, 2, 8, 6
    out = (Hq + 2 * Hkv) * d
    w = r.standard_normal((out, hidden))
    b = r.standard_normal(out)
    for j in range(hidden):
        x = np.zeros((1, hidden)); x[0, j] = 1.0
        q, k, v = qkv_recompute(x, w, b, [0], Hq, Hkv)
        col = w[:, j] + b
        assert np.allclose(q.reshape(-1), col[: Hq * d], atol=1e-14, rtol=0)
        assert np.allclose(k.reshape(-1), col[Hq * d: (Hq + Hkv) * d], atol=1e-14, rtol=0)
        assert np.allclose(v.reshape(-1), col[(Hq + Hkv) * d:], atol=1e-14, rtol=0)
    x1, x2 = r.standard_normal((2, 3, hidden))
    pos = np.array([5, 70, 3000])
    f = lambda x: qkv_recompute(x, w, None, pos, Hq, Hkv)
    for a, b2, c in zip(f(x1 + x2), f(x1), f(x2)):
        assert np.max(np.abs(a - b2 - c)) < 1e-11
    q0, k0, v0 = qkv_recompute(x1, w, b, [0, 0, 0], Hq, Hkv)
    qp, kp, vp = qkv_recompute(x1, w, b, pos, Hq, Hkv)
    assert np.max(np.abs(qp - rope_rotate(q0, pos[:, None]))) < 1e-11
    assert np.max(np.abs(kp - rope_rotate(k0, pos[:, None]))) < 1e-11
    assert np.array_equal(vp, v0)


def pin_common_prefix_len(common_prefix_len):
    """Exact-token common prefix (Sec. V-D): the library's os.path.commonprefix
    on lists, the whole sequence against itself or an extension, the index of
    the first changed token, symmetry and the empty sequence."""
    import os.path
    r = _rs(23)
    for _ in range(200):
        n = int(r.integers(0, 40))
        a = [int(t) for t in r.integers(0, 5, n)]
        b = a[: int(r.integers(0, n + 1))] + [int(t) for t in r.integers(0, 5, int(r.integers(0, 9)))]
        want = len(os.path.commonprefix([a, b]))
        assert common_prefix_len(a, b) == want == common_prefix_len(b, a)
        assert common_prefix_len(a, a) == len(a)
        assert common_prefix_len(a, a + [7, 8]) == len(a)
        if n:
            i = int(r.integers(0, n))
            c = list(a); c[i] = c[i] + 11
            assert common_prefix_len(a, c) == i
    assert common_prefix_len([], [1, 2]) == 0


def pin_warm_match(warm_match, common_prefix_len):
    """Best slot = the longest exact-token prefix, ties to the latest use, a
    miss when no slot shares the first token; empty slots are skipped."""
    r = _rs(24)
    for _ in range(300):
        n_slots = int(r.integers(1, 7))
        base = [int(t) for t in r.integers(0, 3, 12)]
        slots = []
        for _s in range(n_slots):
            if r.random() < 0.2:
                slots.append(None)
                continue
            cut = int(r.integers(0, 13))
            slots.append(base[:cut] + [int(t) for t in r.integers(0, 3, int(r.integers(0, 6)))])
        uses = [int(u) for u in r.permutation(n_slots) + 1]
        q = base[: int(r.integers(0, 13))] + [int(t) for t in r.integers(0, 3, 3)]
        s, m = warm_match(slots, uses, q)
        lens = [common_prefix_len(t, q) if t is not None else 0 for t in slots]
        assert m == max(lens + [0])
        if m == 0:
            assert s == -1
        else:
            ties = [i for i in range(n_slots) if slots[i] is not None and lens[i] == m]
            assert s == max(ties, key=lambda i: uses[i])
    # a hand-made tie: both slots share 3 tokens, slot 0 used later
    assert warm_match([[1, 2, 3, 9], [1, 2, 3, 8]], [5, 4], [1, 2, 3, 7]) == (0, 3)
    assert warm_match([[1, 2, 3, 9], [1, 2, 3, 8]], [4, 5], [1, 2, 3, 7]) == (1, 3)
    assert warm_match([[4, 5], None], [1, 0], [5, 4]) == (-1, 0)


def pin_warm_arena(WarmArenaModel):
    """The arena's decisions on hand-made scenarios: reuse of a stored prefix
    with its exact rows, LRU eviction, in-place extension of a slot, a stored
    prefix of a slot refreshes it, truncation at max_tokens, and forks are
    copies that later stores do not change."""
    def rows(tokens):   # K = V = one row per token holding the token value
        a = np.asarray(tokens, dtype=np.float64).reshape(1, -1, 1, 1)
        return a, -a
    A = list(range(100))
    arena = WarmArenaModel(n_slots=3, max_tokens=120)
    sa = arena.store(A, *rows(A))
    assert sa == 0 and arena.match(A) == (0, 100)
    assert arena.match(A[:50] + [999]) == (0, 50)
    assert arena.match([999] + A) == (-1, 0)
    k, v = arena.fork(0, 37)
    assert np.array_equal(k, rows(A)[0][:, :37]) and np.array_equal(v, rows(A)[1][:, :37])
    B, C, D = [1000 + t for t in A], [2000 + t for t in A], [3000 + t for t in A]
    assert arena.store(B, *rows(B)) == 1 and arena.store(C, *rows(C)) == 2
    arena.fork(0, 10)                        # A is now used after B and C
    assert arena.store(D, *rows(D)) == 1     # B, the least recently used, is evicted
    assert arena.match(B)[0] == -1 and arena.match(A) == (0, 100)
    A2 = A + [500, 501]
    assert arena.store(A2, *rows(A2)) == 0   # an extension replaces its prefix's slot
    assert arena.match(A2) == (0, 102)
    assert arena.store(A[:60], *rows(A[:60])) == 0 and arena.match(A2) == (0, 102)
    E = [4000 + t for t in range(200)]
    se = arena.store(E, *rows(E))
    assert arena.match(E) == (se, 120)       # only the first max_tokens tokens are kept
    k_before, _ = arena.fork(se, 120)
    F = [5000 + t for t in range(5)]
    arena.store(F, *rows(F))
    arena.store([6000], *rows([6000]))
    assert np.array_equal(k_before, rows(E)[0][:, :120])


def pin_slb_quantize(slb_quantize):
    """INT8 codes of the tool scan (Sec. IV-A): within [-127, 127], the largest
    magnitude at +-127, reconstruction within half a step, vectors already on the
    grid unchanged, halves rounded to even, a zero vector left at zero."""
    r = _rs(25)
    x = r.standard_normal((20, 96)).astype(np.float32)
    codes, scales = slb_quantize(x)
    assert codes.dtype == np.int8 and scales.dtype == np.float32
    assert np.all(np.abs(codes.astype(int)) <= 127)
    for i in range(20):
        j = int(np.argmax(np.abs(x[i])))
        assert abs(int(codes[i, j])) == 127 and np.sign(codes[i, j]) == np.sign(x[i, j])
        err = np.abs(x[i].astype(np.float64) - codes[i].astype(np.float64) * float(scales[i]))
        assert np.all(err <= 0.5 * float(scales[i]) * (1 + 1e-5))
    g = (r.integers(-127, 128, (5, 64)).astype(np.float32)) * np.float32(0.25)
    g[:, 0] = np.float32(127 * 0.25)
    c2, s2 = slb_quantize(g)
    assert np.all(s2 == np.float32(0.25)) and np.array_equal(c2.astype(np.float32) * 0.25, g)
    h = np.zeros((1, 4), np.float32)
    h[0] = [127.0, 2.5, 3.5, -2.5]                    # scale exactly 1
    c3, _ = slb_quantize(h)
    assert list(c3[0]) == [127, 2, 4, -2]
    c4, s4 = slb_quantize(np.zeros((1, 8), np.float32))
    assert s4[0] == 0 and not c4.any()


def pin_slb_scores(slb_scores, slb_quantize):
    """Scores: a one-hot query code reads one code of each tool times both scales;
    swapping query and tool changes nothing; for unit vectors the score is the
    cosine up to the quantization error, sqrt(d) (s_q + s_t) / 2 + s_q s_t d / 4."""
    r = _rs(26)
    tc = r.integers(-127, 128, (7, 32)).astype(np.int8)
    ts = (r.random(7).astype(np.float32) + np.float32(0.5)) * np.float32(0.01)
    for k in (0, 5, 31):
        qc = np.zeros((1, 32), np.int8)
        qc[0, k] = 1
        got = slb_scores(qc, np.array([1.0], np.float32), tc, ts)[0]
        want = np.array([np.float32(np.float32(tc[j, k]) * ts[j]) for j in range(7)])
        assert np.array_equal(got, want)
    a = slb_scores(tc[:3], ts[:3], tc[3:], ts[3:])
    b = slb_scores(tc[3:], ts[3:], tc[:3], ts[:3])
    assert np.array_equal(a, b.T)
    d = 768
    x = r.standard_normal((12, d))
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    y = x[:4] + 0.3 * r.standard_normal((4, d))
    y /= np.linalg.norm(y, axis=1, keepdims=True)
    xc, xs = slb_quantize(x)
    yc, ys = slb_quantize(y)
    s = slb_scores(yc, ys, xc, xs)
    cos = y @ x.T
    for a_ in range(4):
        for b_ in range(12):
            bound = (np.sqrt(d) * (ys[a_] + xs[b_]) / 2 + ys[a_] * xs[b_] * d / 4) * (1 + 1e-6)
            assert abs(float(s[a_, b_]) - cos[a_, b_]) <= bound


def pin_slb_route(slb_route):
    """The gate: the best two by score then index (brute force over a hand-made
    registry with a tie), routing only when the margin is strictly above tau,
    and a lone tool always routed."""
    one = np.array([1.0], np.float32)
    q = np.zeros((1, 4), np.int8)
    q[0, 0] = 1
    step = np.float32(1.0 / 1024)
    def registry(vals):
        t = np.zeros((len(vals), 4), np.int8)
        t[:, 0] = vals
        return t, np.full(len(vals), step, np.float32)
    tau = np.float32(3.0 / 1024)
    t, ts = registry([7, 10, 3, 10])               # tie at 10: index 1 before 3
    (i1, i2, s1, s2, route), = slb_route(q, one, t, ts, tau)
    assert (i1, i2) == (1, 3) and s1 == s2 == np.float32(10 / 1024) and route == -1
    t, ts = registry([7, 10, 3])                   # margin 3/1024 == tau: escalates
    assert slb_route(q, one, t, ts, tau)[0][4] == -1
    t, ts = registry([6, 10, 3])                   # margin 4/1024 > tau: routes to 1
    assert slb_route(q, one, t, ts, tau)[0][4] == 1
    t, ts = registry([-5])                         # a single tool: always routed
    (i1, i2, s1, s2, route), = slb_route(q, one, t, ts, tau)
    assert (i1, i2, route) == (0, -1, 0) and s2 == -np.inf
    r = _rs(27)
    for _ in range(20):
        vals = r.integers(-127, 128, 9)
        t, ts = registry(vals)
        (i1, i2, _, _, _), = slb_route(q, one, t, ts, tau)
        order = sorted(range(9), key=lambda j: (-int(vals[j]), j))
        assert (i1, i2) == (order[0], order[1])
