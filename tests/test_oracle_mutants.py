"""Planted mistakes in copies of the oracle must each trip at least one pin.

Each mutant below is a plausible slip when writing the oracle from the paper
(a dropped term, a wrong sign, a wrong index, a transposed operand). The
mutants live here, on the CPU, and never touch the real oracle module.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
import oracle_pins as P


def _fails(fn, *args):
    try:
        fn(*args)
    except AssertionError:
        return True
    except Exception:
        return True
    return False


# ---- policy mutants (Eq. 2)
def pct_denominator_mk(n, M=256, R_base=5, K=4):
    if n <= M:
        return Fraction(R_base)
    return min(Fraction(R_base) + Fraction(n - M, M * K) * (100 - R_base), Fraction(100))


def pct_no_clamp(n, M=256, R_base=5, K=4):
    if n <= M:
        return Fraction(R_base)
    return Fraction(R_base) + Fraction(n - M, M * (K - 1)) * (100 - R_base)


def pct_drops_base(n, M=256, R_base=5, K=4):
    if n <= M:
        return Fraction(R_base)
    return min(Fraction(R_base) + Fraction(n - M, M * (K - 1)) * 100, Fraction(100))


def len_floor(S, n, M=256, R_base=5, K=4):
    return min(S, math.floor(Fraction(S) * oracle.recompute_pct(n, M, R_base, K) / 100))


@pytest.mark.parametrize("mut", [pct_denominator_mk, pct_no_clamp, pct_drops_base])
def test_policy_mutants_caught(mut):
    assert _fails(P.pin_table1, mut) or _fails(P.pin_eq2_shape, mut)


def test_redecode_floor_caught():
    assert _fails(P.pin_redecode_len, len_floor, oracle.recompute_pct)


# ---- RoPE mutants
def _rope_factory(sign=1.0, pairs="half", exponent=2.0, swap_out=False):
    def rope(x, pos, theta_base=1.0e6, freq_scale=1.0, rope_type="neox"):
        x = np.asarray(x, dtype=np.float64)
        d = x.shape[-1]
        h = d // 2
        th = freq_scale * theta_base ** (-exponent * np.arange(h) / d)
        ang = np.asarray(pos, dtype=np.float64)[..., None] * th
        c, s = np.cos(ang), sign * np.sin(ang)
        out = np.empty(np.broadcast_shapes(x.shape, ang.shape[:-1] + (d,)))
        if rope_type == "neox" and pairs == "half":
            a, b = x[..., :h], x[..., h:]
            out[..., :h] = a * c - b * s
            out[..., h:] = (b * s + a * c) if swap_out else (a * s + b * c)
        else:
            a, b = x[..., 0::2], x[..., 1::2]
            out[..., 0::2] = a * c - b * s
            out[..., 1::2] = a * s + b * c
        return out
    return rope


ROPE_MUTANTS = {
    "sin_sign": _rope_factory(sign=-1.0),
    "interleaved_as_neox": _rope_factory(pairs="interleaved"),
    "exponent_i_over_d": _rope_factory(exponent=1.0),
    "swapped_terms": _rope_factory(swap_out=True),
}


@pytest.mark.parametrize("name", sorted(ROPE_MUTANTS))
def test_rope_mutants_caught(name):
    m = ROPE_MUTANTS[name]
    assert (_fails(P.pin_rope_complex, m) or _fails(P.pin_rope_2x2, m)
            or _fails(P.pin_rope_group, m))


# ---- splice mutants
def splice_tail_not_rotated(live_k, live_v, inserts, *a, **kw):
    ks, vs, cur, shift = [], [], 0, 0
    for p, bk, bv, m0 in inserts:
        ks.append(live_k[:, cur:p]); vs.append(live_v[:, cur:p])
        ks.append(oracle.rerotate(bk, p + shift - m0)); vs.append(bv)
        shift += bk.shape[1]; cur = p
    ks.append(live_k[:, cur:]); vs.append(live_v[:, cur:])
    return np.concatenate(ks, 1), np.concatenate(vs, 1)


def splice_delta_sign(live_k, live_v, inserts, *a, **kw):
    ks, vs, cur, shift = [], [], 0, 0
    for p, bk, bv, m0 in inserts:
        ks.append(oracle.rerotate(live_k[:, cur:p], shift)); vs.append(live_v[:, cur:p])
        ks.append(oracle.rerotate(bk, m0 - (p + shift))); vs.append(bv)
        shift += bk.shape[1]; cur = p
    ks.append(oracle.rerotate(live_k[:, cur:], shift)); vs.append(live_v[:, cur:])
    return np.concatenate(ks, 1), np.concatenate(vs, 1)


def splice_ignores_earlier_inserts(live_k, live_v, inserts, *a, **kw):
    ks, vs, cur, shift = [], [], 0, 0
    for p, bk, bv, m0 in inserts:
        ks.append(oracle.rerotate(live_k[:, cur:p], shift)); vs.append(live_v[:, cur:p])
        ks.append(oracle.rerotate(bk, p - m0)); vs.append(bv)
        shift += bk.shape[1]; cur = p
    ks.append(oracle.rerotate(live_k[:, cur:], shift)); vs.append(live_v[:, cur:])
    return np.concatenate(ks, 1), np.concatenate(vs, 1)


@pytest.mark.parametrize("mut", [splice_tail_not_rotated, splice_delta_sign, splice_ignores_earlier_inserts])
def test_splice_mutants_caught(mut):
    assert _fails(P.pin_splice_closed_form, mut, oracle.rope_rotate)


def test_rerotate_arithmetic_at_zero_caught():
    def rerot_always_math(k, delta, *a, **kw):
        return oracle.rope_rotate(k, int(delta))
    assert _fails(P.pin_rerotate, rerot_always_math, oracle.rope_rotate)


# ---- attention mutants
def _attn_factory(scale=True, strict=False, head_map="div", transpose_v=False):
    def attn(q, k, v, q_pos, group):
        q = np.asarray(q, float); k = np.asarray(k, float); v = np.asarray(v, float)
        R, Hq, d = q.shape
        T = k.shape[0]
        Hkv = k.shape[1]
        pos = np.asarray(q_pos)
        vis = (np.arange(T)[None, :] < pos[:, None]) if strict else (np.arange(T)[None, :] <= pos[:, None])
        o = np.zeros((R, Hq, d)); lse = np.zeros((R, Hq))
        for h in range(Hq):
            kv = h // group if head_map == "div" else h % Hkv
            s = q[:, h] @ k[:, kv].T
            if scale:
                s = s / math.sqrt(d)
            s = np.where(vis, s, -np.inf)
            m = s.max(1, keepdims=True)
            e = np.exp(s - m)
            z = e.sum(1, keepdims=True)
            vv = v[:, kv]
            if transpose_v and T == d:
                vv = vv.T
            o[:, h] = (e / z) @ vv
            lse[:, h] = m[:, 0] + np.log(z[:, 0])
        return o, lse
    return attn


ATTN_MUTANTS = {
    "no_scale": _attn_factory(scale=False),
    "strict_mask": _attn_factory(strict=True),
    "head_mod": _attn_factory(head_map="mod"),
}


@pytest.mark.parametrize("name", sorted(ATTN_MUTANTS))
def test_attention_mutants_caught(name):
    m = ATTN_MUTANTS[name]
    assert (_fails(P.pin_attention_library, m) or _fails(P.pin_attention_special, m))


SUFFIX_POSITION_MUTANTS = {
    # the suffix shifted one past the cache end
    "start_plus_one": lambda T, R: np.arange(T - R + 1, T + 1, dtype=np.int64),
    # positions counted from the suffix start instead of the cache start
    "from_zero": lambda T, R: np.arange(R, dtype=np.int64),
    # one token short at the end
    "one_short": lambda T, R: np.arange(T - R, T - 1, dtype=np.int64),
}


@pytest.mark.parametrize("name", sorted(SUFFIX_POSITION_MUTANTS))
def test_suffix_position_mutants_caught(name):
    assert _fails(P.pin_suffix_positions, SUFFIX_POSITION_MUTANTS[name])


def test_softcap_mutants_caught():
    def cap_before_scale(q, k, v, q_pos, group, softcap=None):
        q = np.asarray(q, float); k = np.asarray(k, float); v = np.asarray(v, float)
        R, Hq, d = q.shape
        T = k.shape[0]
        vis = np.arange(T)[None, :] <= np.asarray(q_pos)[:, None]
        o = np.zeros((R, Hq, d)); lse = np.zeros((R, Hq))
        for h in range(Hq):
            s = q[:, h] @ k[:, h // group].T
            if softcap is not None:
                s = softcap * np.tanh(s / softcap)
            s = np.where(vis, s / math.sqrt(d), -np.inf)
            m = s.max(1, keepdims=True); e = np.exp(s - m); z = e.sum(1, keepdims=True)
            o[:, h] = (e / z) @ v[:, h // group]; lse[:, h] = m[:, 0] + np.log(z[:, 0])
        return o, lse

    def cap_ignored(q, k, v, q_pos, group, softcap=None):
        return oracle.attention(q, k, v, q_pos, group)

    assert _fails(P.pin_attention_softcap, cap_before_scale)
    assert _fails(P.pin_attention_softcap, cap_ignored)


def test_qkv_mutants_caught():
    def transposed_weight(x, w, b, positions, Hq, Hkv, *a, **kw):
        w = np.asarray(w)
        wt = w.reshape(-1)[: w.size].reshape(w.shape[1], w.shape[0]).T   # a mis-strided read
        return oracle.qkv_recompute(x, wt, b, positions, Hq, Hkv)

    def kv_swapped(x, w, b, positions, Hq, Hkv, *a, **kw):
        q, k, v = oracle.qkv_recompute(x, w, b, positions, Hq, Hkv)
        return q, v, k

    def no_bias(x, w, b, positions, Hq, Hkv, *a, **kw):
        return oracle.qkv_recompute(x, w, None, positions, Hq, Hkv)

    def v_rotated(x, w, b, positions, Hq, Hkv, *a, **kw):
        q, k, v = oracle.qkv_recompute(x, w, b, positions, Hq, Hkv)
        return q, k, oracle.rope_rotate(v, np.asarray(positions)[:, None])

    for mut in (transposed_weight, kv_swapped, no_bias, v_rotated):
        assert _fails(P.pin_qkv_recompute, mut, oracle.rope_rotate), mut.__name__


def test_arena_mutants_caught():
    def lcp_counts_mismatch(a, b):
        n = oracle.common_prefix_len(a, b)
        return n + 1 if n < min(len(a), len(b)) else n

    assert _fails(P.pin_common_prefix_len, lcp_counts_mismatch)

    def match_ties_to_oldest(slots, uses, q):
        best, best_len, best_use = -1, 0, None
        for s, t in enumerate(slots):
            if t is None:
                continue
            n = oracle.common_prefix_len(t, q)
            if n and (n > best_len or (n == best_len and uses[s] < best_use)):
                best, best_len, best_use = s, n, uses[s]
        return best, best_len

    assert _fails(P.pin_warm_match, match_ties_to_oldest, oracle.common_prefix_len)

    class EvictsMostRecent(oracle.WarmArenaModel):
        """Evicts the most recently used slot when the arena is full."""
        def store(self, tokens, k, v):
            toks = [int(t) for t in tokens[: self.max_tokens]]
            related = any(t is not None and (t[: len(toks)] == toks or toks[: len(t)] == t)
                          for t in self.tokens)
            if not related and all(t is not None for t in self.tokens):
                self.tokens[max(range(self.n_slots), key=lambda i: self.last_use[i])] = None
            return super().store(tokens, k, v)

    class NoExtension(oracle.WarmArenaModel):
        """Never replaces a slot whose tokens are a prefix of the stored ones."""
        def store(self, tokens, k, v):
            toks = [int(t) for t in tokens[: self.max_tokens]]
            for s, t in enumerate(self.tokens):
                if t is not None and len(t) >= len(toks) and t[: len(toks)] == toks:
                    self._touch(s)
                    return s
            empty = [s for s, t in enumerate(self.tokens) if t is None]
            s = empty[0] if empty else min(range(self.n_slots), key=lambda i: self.last_use[i])
            self.tokens[s] = toks
            self.k[s] = np.array(k[:, : len(toks)])
            self.v[s] = np.array(v[:, : len(toks)])
            self._touch(s)
            return s

    for mut in (EvictsMostRecent, NoExtension):
        assert _fails(P.pin_warm_arena, mut), mut.__name__


def test_slb_mutants_caught():
    def round_half_up(x):
        codes, scales = oracle.slb_quantize(x)
        x = np.asarray(x, np.float32)
        for i in range(x.shape[0]):
            if scales[i]:
                codes[i] = np.clip(np.floor(x[i] / scales[i] + np.float32(0.5)), -127, 127)
        return codes, scales

    def scale_by_255(x):
        x = np.asarray(x, np.float32)
        codes, scales = oracle.slb_quantize(x)
        return codes, scales * np.float32(127.0 / 255.0)

    assert _fails(P.pin_slb_quantize, round_half_up)
    assert _fails(P.pin_slb_quantize, scale_by_255)

    def no_tool_scale(qc, qs, tc, ts):
        return oracle.slb_scores(qc, qs, tc, np.ones_like(ts))

    assert _fails(P.pin_slb_scores, no_tool_scale, oracle.slb_quantize)

    def gate_inclusive(qc, qs, tc, ts, tau=oracle.slb.TAU):
        out = []
        for i1, i2, s1, s2, _ in oracle.slb_route(qc, qs, tc, ts, tau):
            out.append((i1, i2, s1, s2, i1 if np.float32(s1 - s2) >= tau else -1))
        return out

    def ties_to_last(qc, qs, tc, ts, tau=oracle.slb.TAU):
        s = oracle.slb_scores(qc, qs, tc, ts)
        out = []
        for a in range(s.shape[0]):
            order = sorted(range(s.shape[1]), key=lambda j: (-float(s[a, j]), -j))
            i1 = order[0]
            i2 = order[1] if len(order) > 1 else -1
            s2 = s[a, i2] if i2 >= 0 else np.float32(-np.inf)
            out.append((i1, i2, s[a, i1], s2, i1 if s[a, i1] - s2 > tau else -1))
        return out

    assert _fails(P.pin_slb_route, gate_inclusive)
    assert _fails(P.pin_slb_route, ties_to_last)
