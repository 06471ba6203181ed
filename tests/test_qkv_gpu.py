"""Parity of the re-decoded suffix tokens' fresh Q, K, V (Sec. V-A) with the
oracle: projection, RoPE at the new positions (Sec. III-B) and the paged-cache
write, through the C ABI.

Tolerance: every output element within 2e-3 + half a bf16 ulp of the fp64
oracle (the bf16 store alone errs by up to half an ulp; float32 accumulation
of 5120 exact bf16 products and the float rotation add a few 1e-5). Cache slots
the call does not own stay bit-identical.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_k_close, f64
from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import HIDDEN, qkv_weights, randn_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return torch.device("cuda:0")


class QkvCase:
    """Sequences with their suffix positions in a randomly filled paged pool."""

    def __init__(self, dev, kv_len, q_len, hidden, n_q_heads=40, n_kv_heads=8, n_layers=2,
                 layer=1, vt=False, gptj=False, bias=True, seed=0, shuffle=True, theta=1.0e6):
        self.dev, self.layer, self.vt, self.gptj = dev, layer, vt, gptj
        self.kv_len, self.q_len = list(kv_len), list(q_len)
        self.Hq, self.Hkv, self.hidden = n_q_heads, n_kv_heads, hidden
        self.theta = theta
        self.max_pages = max(-(-k // 16) for k in kv_len) + 1
        r = np.random.default_rng(seed)
        # Only the pages holding suffix positions are distinct pool pages; the
        # rest of each table points at a shared spare page never written.
        used = [sorted({p // 16 for p in range(k - q, k)}) for k, q in zip(kv_len, q_len)]
        n_need = sum(len(u) for u in used)
        self.n_pages = n_need + 8
        order = r.permutation(self.n_pages) if shuffle else np.arange(self.n_pages)
        self.h_pt = np.full((len(kv_len), self.max_pages), int(order[-1]), np.int32)
        k = 0
        for s, u in enumerate(used):
            for pg in u:
                self.h_pt[s, pg] = order[k]
                k += 1
        self.d_pt = torch.as_tensor(self.h_pt, device=dev)
        shape = (n_layers, self.n_pages, n_kv_heads, 16, 128)
        self.kp = randn_bf16(shape, seed + 1, dev)
        vshape = (n_layers, self.n_pages, n_kv_heads, 128, 16) if vt else shape
        self.vp = randn_bf16(vshape, seed + 2, dev)
        self.k0, self.v0 = self.kp.clone(), self.vp.clone()
        self.cache = nexus.kv_cache(self.kp, self.vp, self.n_pages, n_layers, n_kv_heads, vt,
                                    rope_theta=theta,
                                    rope_type=nexus.ROPE_GPTJ if gptj else nexus.ROPE_NEOX)
        self.n_tok = sum(q_len)
        self.x = randn_bf16((self.n_tok, hidden), seed + 3, dev)
        self.n_heads = n_q_heads + 2 * n_kv_heads
        self.w, self.b = qkv_weights(self.n_heads, hidden, seed + 4, dev, bias)
        self.q = torch.full((self.n_tok, n_q_heads, 128), float("nan"), dtype=torch.bfloat16,
                            device=dev)

    def run(self, h_pt=True, stream=None):
        nexus.suffix_qkv(self.cache, self.d_pt, len(self.kv_len), self.max_pages, self.kv_len,
                         self.q_len, self.x, self.w, self.b, self.q, layer=self.layer,
                         n_q_heads=self.Hq, h_page_tables=self.h_pt if h_pt else None,
                         stream=stream)

    def positions(self):
        return np.concatenate([np.arange(k - q, k) for k, q in zip(self.kv_len, self.q_len)]
                              ).astype(np.int64)

    def slots(self):
        """(sequence row, page, slot) of every packed token."""
        rows = np.concatenate([np.full(q, s) for s, q in enumerate(self.q_len)]).astype(np.int64)
        pos = self.positions()
        return rows, self.h_pt[rows, pos // 16].astype(np.int64), pos % 16

    def written_kv(self):
        _, pg, sl = self.slots()
        pg = torch.as_tensor(pg, device=self.dev)
        sl = torch.as_tensor(sl, device=self.dev)
        k = self.kp[self.layer][pg, :, sl, :]
        v = self.vp[self.layer][pg, :, :, sl] if self.vt else self.vp[self.layer][pg, :, sl, :]
        return k, v

    def oracle(self, rows=None):
        sel = slice(None) if rows is None else rows
        pos = self.positions()[sel]
        x = f64(self.x[sel])
        b = None if self.b is None else self.b.double().cpu().numpy()
        return oracle.qkv_recompute(x, f64(self.w), b, pos, self.Hq, self.Hkv,
                                    theta_base=self.theta,
                                    rope_type="gptj" if self.gptj else "neox")

    def check(self, rows=None, what=""):
        q, k, v = self.oracle(rows)
        sel = slice(None) if rows is None else rows
        gk, gv = self.written_kv()
        assert_k_close(f64(self.q[sel]), q, what + " Q")
        assert_k_close(f64(gk[sel]), k, what + " K")
        assert_k_close(f64(gv[sel]), v, what + " V")

    def check_untouched(self):
        """Every pool element outside the written slots keeps its bits."""
        _, pg, sl = self.slots()
        pg = torch.as_tensor(pg, device=self.dev)
        sl = torch.as_tensor(sl, device=self.dev)
        k, v = self.kp.clone(), self.vp.clone()
        k[self.layer, pg, :, sl, :] = self.k0[self.layer, pg, :, sl, :]
        if self.vt:
            v[self.layer, pg, :, :, sl] = self.v0[self.layer, pg, :, :, sl]
        else:
            v[self.layer, pg, :, sl, :] = self.v0[self.layer, pg, :, sl, :]
        assert torch.equal(k.view(torch.int16), self.k0.view(torch.int16))
        assert torch.equal(v.view(torch.int16), self.v0.view(torch.int16))


@pytest.mark.parametrize("vt,gptj,bias", [(False, False, True), (True, False, True),
                                          (False, True, False), (True, True, True)])
def test_qkv_small_ragged(dev, vt, gptj, bias):
    # 150 tokens: a full 128-row tile and a ragged one; hidden 256: four stages
    c = QkvCase(dev, [300], [150], 256, vt=vt, gptj=gptj, bias=bias, seed=11)
    c.run()
    torch.cuda.synchronize()
    c.check(what=f"vt={vt} gptj={gptj}")
    c.check_untouched()


def test_qkv_varlen_sequences(dev):
    # several sequences, one empty, tokens of one 128-row tile from three of them
    c = QkvCase(dev, [40, 700, 1, 333, 129], [17, 90, 0, 333, 1], 512, vt=True, seed=12)
    c.run()
    torch.cuda.synchronize()
    c.check(what="varlen")
    c.check_untouched()


def test_qkv_odd_heads_and_hidden_tail(dev):
    # 3 + 2 * 1 = 5 heads: the last 256-feature tile holds one head; hidden 72
    # leaves 8 features in the last 64-wide stage
    c = QkvCase(dev, [64], [50], 72, n_q_heads=3, n_kv_heads=1, seed=13)
    c.run()
    torch.cuda.synchronize()
    c.check(what="odd")
    c.check_untouched()


def test_qkv_deep_positions(dev):
    # positions past 10^6: the angle reduction of the rotation
    c = QkvCase(dev, [1_000_003], [70], 128, seed=14, n_layers=1, layer=0)
    c.run()
    torch.cuda.synchronize()
    c.check(what="deep")


def test_qkv_single_token(dev):
    c = QkvCase(dev, [5], [1], HIDDEN, seed=15)
    c.run()
    torch.cuda.synchronize()
    c.check(what="single")
    c.check_untouched()


def test_qkv_full_size_redecode(dev):
    # The 100 % suffix of the 8192 + 1024 token session with token-innermost V:
    # 2192 re-decoded tokens, hidden 5120, 40 + 8 + 8 heads; every output checked.
    c = QkvCase(dev, [9216], [2192], HIDDEN, vt=True, seed=16, n_layers=2, layer=1)
    c.run()
    torch.cuda.synchronize()
    c.check(what="2192 tokens")
    c.check_untouched()


def test_qkv_full_size_many_tiles_sampled(dev):
    # 8 sequences of 1000 re-decoded tokens: 63 token tiles x 28 feature tiles,
    # several tiles per CTA; sampled rows against the oracle.
    kv = [5000 + 97 * i for i in range(8)]
    c = QkvCase(dev, kv, [1000] * 8, HIDDEN, seed=17)
    c.run()
    torch.cuda.synchronize()
    rows = np.random.default_rng(0).choice(c.n_tok, 300, replace=False)
    rows = np.sort(np.concatenate([rows, [0, 127, 128, c.n_tok - 1]]))
    c.check(rows=rows, what="8 x 1000")
    c.check_untouched()


def test_qkv_repeat_is_bitwise_deterministic(dev):
    c = QkvCase(dev, [2000], [700], 1024, vt=True, seed=18)
    c.run()
    q1 = c.q.clone()
    k1, v1 = (t.clone() for t in c.written_kv())
    c.run()
    torch.cuda.synchronize()
    k2, v2 = c.written_kv()
    assert torch.equal(q1.view(torch.int16), c.q.view(torch.int16))
    assert torch.equal(k1.view(torch.int16), k2.view(torch.int16))
    assert torch.equal(v1.view(torch.int16), v2.view(torch.int16))


def test_qkv_bad_page_is_skipped_and_reported(dev):
    # Without the host tables the kernel checks the page ids itself: a token
    # whose page lies outside the pool is not written and the call reports it.
    c = QkvCase(dev, [64], [32], 128, seed=19)
    bad = c.h_pt.copy()
    bad[0, 3] = c.n_pages + 5                                # positions 48..63
    c.d_pt = torch.as_tensor(bad, device=dev)
    assert nexus.device_status() == nexus.OK
    c.run(h_pt=False)
    assert nexus.device_status() == nexus.ERANGE
    assert nexus.device_status() == nexus.OK                 # the record is cleared
    q, k, v = c.oracle()
    assert_k_close(f64(c.q), q, "Q")
    c.d_pt = torch.as_tensor(c.h_pt, device=dev)
    gk, gv = c.written_kv()
    assert_k_close(f64(gk[:16]), k[:16], "K")               # positions 32..47 written
    assert torch.equal(gk[16:].view(torch.int16),
                       c.k0[c.layer][torch.as_tensor(c.h_pt[0, 3], device=dev)].permute(1, 0, 2)
                       .reshape(16, 8, 128).view(torch.int16))


def test_qkv_bench_size_32768_tokens_sampled(dev):
    # The bench's launch: all 32768 tokens of the c5 re-prefill, one layer, hidden
    # 5120, 40 + 8 + 8 heads; 256 sampled rows (every tile row position class and
    # the ragged ends) against the oracle, and no write outside the cache slots.
    c = QkvCase(dev, [32768], [32768], HIDDEN, seed=22, n_layers=1, layer=0)
    c.run()
    torch.cuda.synchronize()
    r = np.random.default_rng(1)
    rows = np.sort(np.unique(np.concatenate([r.choice(32768, 250, replace=False),
                                             [0, 1, 127, 128, 32767, 32640]])))
    c.check(rows=rows, what="32768 tokens")
    c.check_untouched()


@pytest.mark.parametrize("vt,gptj", [(False, False), (True, False), (True, True)])
def test_qkv_short_suffix_64_tokens(dev, vt, gptj):
    # 64 tokens or fewer take one-head tiles with 64 token rows per stage: the
    # c5 suffix shape (64 re-decoded tokens, hidden 5120, 40 + 8 + 8 heads).
    c = QkvCase(dev, [34816], [64], HIDDEN, vt=vt, gptj=gptj, seed=31, n_layers=1, layer=0)
    c.run()
    torch.cuda.synchronize()
    c.check(what=f"64 tokens vt={vt} gptj={gptj}")
    c.check_untouched()


def test_qkv_short_suffix_ragged_sequences(dev):
    # 63 tokens from four sequences (one empty), odd head counts, hidden 1000
    c = QkvCase(dev, [100, 40, 5000, 17], [30, 0, 32, 1], 1000, n_q_heads=5, n_kv_heads=1,
                vt=True, seed=32)
    c.run()
    torch.cuda.synchronize()
    c.check(what="short ragged")
    c.check_untouched()


@pytest.mark.parametrize("hidden,gptj", [(256, True), (448, False), (HIDDEN, True)])
def test_qkv_short_pair_split_hidden(dev, hidden, gptj):
    # Up to 64 tokens each head's tile is shared by a pair of CTAs that split the
    # hidden dimension and add their partial sums over distributed shared memory:
    # the smallest split (two stages, the second partly past the hidden size), an
    # odd stage count, and the bench's width with GPT-J pairs; varlen with a
    # one-token sequence; two runs bit-identical.
    c = QkvCase(dev, [700, 9000, 33], [1, 40, 23], hidden, gptj=gptj, seed=34 + hidden)
    c.run()
    torch.cuda.synchronize()
    c.check(what=f"pair split hidden {hidden} gptj={gptj}")
    c.check_untouched()
    q1 = c.q.clone()
    k1, v1 = c.kp.clone(), c.vp.clone()
    c.run()
    torch.cuda.synchronize()
    assert torch.equal(q1.view(torch.int16), c.q.view(torch.int16))
    assert torch.equal(k1.view(torch.int16), c.kp.view(torch.int16))
    assert torch.equal(v1.view(torch.int16), c.vp.view(torch.int16))
    assert nexus.device_status() == nexus.OK


def test_qkv_65_tokens_take_long_tiles(dev):
    c = QkvCase(dev, [300], [65], 512, seed=33)
    c.run()
    torch.cuda.synchronize()
    c.check(what="65 tokens")
    c.check_untouched()


def test_recompute_then_attention_back_to_back(dev):
    """The re-decode of a layer as a model runs it: fresh Q/K/V, then the suffix
    attention reading them, then the next recompute overwriting them, all on one
    stream with no synchronisation. The launches overlap their setup with the
    previous kernel (programmatic dependent launch) and must still read only
    completed inputs and not overwrite inputs still being read: the attention
    output equals the one of the same calls synchronised after each step, bit for
    bit, and the oracle's on the recomputed Q, K and V."""
    kv, ql = [3000], [64]
    c = QkvCase(dev, kv, ql, HIDDEN, seed=61, n_layers=2, layer=1)
    x1, x2 = c.x.clone(), randn_bf16(c.x.shape, 62, dev)
    need, _ = nexus.attention_workspace_size(kv, ql, 40, 8, 1, 0)
    ws = torch.empty(max(16, need), dtype=torch.uint8, device=dev)

    def attend(o, lse, stream=None):
        nexus.suffix_attention(c.cache, c.d_pt, 1, c.max_pages, kv, ql, c.q[None], o, lse, 40,
                               c.layer, c.layer + 1, split_kv=0, workspace=ws,
                               workspace_bytes=need, stream=stream)

    k0, v0 = c.kp.clone(), c.vp.clone()
    # synchronised after every step
    c.x = x1
    c.run()
    torch.cuda.synchronize()
    q1, kp1, vp1 = c.q.clone(), c.kp.clone(), c.vp.clone()
    o_ref = torch.empty((1, 64, 40, 128), dtype=torch.bfloat16, device=dev)
    l_ref = torch.empty((1, 64, 40), dtype=torch.float32, device=dev)
    attend(o_ref, l_ref)
    torch.cuda.synchronize()
    # back to back on one stream
    c.kp.copy_(k0)
    c.vp.copy_(v0)
    s = torch.cuda.Stream()
    o = torch.full_like(o_ref, float("nan"))
    l = torch.full_like(l_ref, float("nan"))
    torch.cuda.synchronize()
    with torch.cuda.stream(s):   # three library launches back to back, nothing between
        c.x = x1
        c.run(stream=s)
        attend(o, l, stream=s)
        c.x = x2
        c.run(stream=s)
    s.synchronize()
    assert nexus.device_status() == nexus.OK
    assert torch.equal(o.view(torch.int16), o_ref.view(torch.int16))
    assert torch.equal(l, l_ref)
    # and the oracle on the recomputed rows (sampled)
    rows = np.array([0, 1, 31, 62, 63])
    pos = np.arange(kv[0] - ql[0], kv[0])
    pg = torch.as_tensor(c.h_pt[0][np.arange(kv[0]) // 16], device=dev).long()
    sl = torch.arange(kv[0], device=dev) % 16
    k_all = kp1[c.layer][pg, :, sl, :]
    v_all = vp1[c.layer][pg, :, sl, :]
    want, want_l = oracle.attention(f64(q1[rows]), f64(k_all), f64(v_all), pos[rows], 5)
    from gpu_cases import assert_attn_close
    assert_attn_close(f64(o[0, rows]), want, f64(l[0, rows]), want_l, "recompute then attention")
