"""Suffix-redecode / re-prefill attention on the GPU against the fp64 oracle
(softmax(QK^T / sqrt(d)) V of Sec. III-A over the last R positions,
Sec. III-C / Sec. V-A)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import (SplicedCase, assert_attn_close, f64, new_pools, write_rows)
from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import randn_bf16, workload

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0") if torch.cuda.is_available() else None


def _direct_case(kv_lens, q_lens, Hq=40, H=8, L=1, vt=False, seed=0, shuffle=True,
                 garbage=True, vscale=1.0, order=None, k_edit=None):
    """Sequences written straight into a paged pool (no splice); slots past
    kv_len hold NaN so any leak of them into the output shows. vscale (a power
    of two, so exact in bf16) scales V. `order` (a permutation of the pool's
    pages) overrides `shuffle`. `k_edit(i, k)` may replace sequence i's K rows
    before they are written."""
    rng = np.random.default_rng(seed)
    max_pages = max(-(-k // 16) for k in kv_lens) + 1
    n_pages = sum(-(-k // 16) for k in kv_lens) + 8
    kp, vp = new_pools(L, n_pages, H, vt, DEV, float("nan") if garbage else 0.0)
    if order is None:
        order = rng.permutation(n_pages) if shuffle else np.arange(n_pages)
    assert sorted(order) == list(range(n_pages))
    h_pt = np.full((len(kv_lens), max_pages), -1, np.int32)
    ks, vs, cur = [], [], 0
    for i, T in enumerate(kv_lens):
        npg = -(-T // 16)
        h_pt[i, :npg] = order[cur:cur + npg]
        cur += npg
        k = randn_bf16((L, T, H, 128), seed * 100 + 2 * i, DEV)
        if k_edit is not None:
            k = k_edit(i, k)
        v = randn_bf16((L, T, H, 128), seed * 100 + 2 * i + 1, DEV)
        if vscale != 1.0:
            v = (v.float() * vscale).to(torch.bfloat16)
        write_rows(kp, vp, h_pt[i], k, v, vt)
        ks.append(k)
        vs.append(v)
    q = randn_bf16((L, sum(q_lens), Hq, 128), seed * 100 + 99, DEV)
    cache = nexus.kv_cache(kp, vp, n_pages, L, H, vt)
    return cache, torch.as_tensor(h_pt, device=DEV), max_pages, ks, vs, q


def _run(cache, d_pt, max_pages, kv_lens, q_lens, q, Hq, L, split_kv=1, rows=None):
    o = torch.full_like(q, float("nan"))
    lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=DEV)
    nbytes, _ = nexus.attention_workspace_size(kv_lens, q_lens, Hq, cache.n_kv_heads, L, split_kv)
    ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=DEV)
    nexus.suffix_attention(cache, d_pt, d_pt.shape[0], max_pages, kv_lens, q_lens, q, o, lse, Hq,
                           0, L, rows=rows, split_kv=split_kv, workspace=ws, workspace_bytes=nbytes)
    assert nexus.device_status() == nexus.OK
    return o, lse


def _check(ks, vs, q, o, lse, kv_lens, q_lens, group, layer=0, what="", softcap=None):
    off = 0
    for i, (T, R) in enumerate(zip(kv_lens, q_lens)):
        if R == 0:
            continue
        want_o, want_l = oracle.attention(f64(q[layer, off:off + R]), f64(ks[i][layer]),
                                          f64(vs[i][layer]), oracle.suffix_positions(T, R), group,
                                          softcap=softcap)
        assert_attn_close(f64(o[layer, off:off + R]), want_o, f64(lse[layer, off:off + R]), want_l,
                          f"{what} seq {i} T={T} R={R}")
        off += R


@pytest.mark.parametrize("T,R", [(1, 1), (2, 2), (15, 15), (16, 16), (17, 17), (130, 1),
                                 (640, 64), (300, 24), (301, 25), (302, 26), (1000, 127),
                                 (1001, 128), (1003, 129), (257, 257)])
def test_suffix_attention_shapes(T, R):
    cache, d_pt, mp, ks, vs, q = _direct_case([T], [R], seed=T * 7 + R)
    o, lse = _run(cache, d_pt, mp, [T], [R], q, 40, 1)
    _check(ks, vs, q, o, lse, [T], [R], 5, what="shape")


@pytest.mark.parametrize("Hq,H", [(8, 8), (16, 2), (32, 8), (12, 4)])
def test_gqa_groupings(Hq, H):
    cache, d_pt, mp, ks, vs, q = _direct_case([333], [200], Hq=Hq, H=H, seed=Hq + H)
    o, lse = _run(cache, d_pt, mp, [333], [200], q, Hq, 1)
    _check(ks, vs, q, o, lse, [333], [200], Hq // H, what=f"gqa {Hq}/{H}")


def test_transposed_v_layout():
    cache, d_pt, mp, ks, vs, q = _direct_case([777], [300], vt=True, seed=3)
    o, lse = _run(cache, d_pt, mp, [777], [300], q, 40, 1)
    _check(ks, vs, q, o, lse, [777], [300], 5, what="vT")


def test_varlen_batch_multi_layer():
    kv = [700, 33, 1500, 16, 900]
    ql = [100, 33, 7, 0, 450]
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, L=3, seed=5)
    o, lse = _run(cache, d_pt, mp, kv, ql, q, 40, 3)
    for layer in range(3):
        _check(ks, vs, q, o, lse, kv, ql, 5, layer, what=f"varlen layer {layer}")


@pytest.mark.parametrize("splits", [2, 5, 19, 32])
def test_split_kv_matches_oracle(splits):
    kv, ql = [5000], [64]
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, seed=11)
    o, lse = _run(cache, d_pt, mp, kv, ql, q, 40, 1, split_kv=splits)
    _check(ks, vs, q, o, lse, kv, ql, 5, what=f"split {splits}")


def test_split_kv_auto_varlen():
    kv, ql = [3000, 200, 4100], [40, 1, 64]
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, L=2, seed=12)
    _, splits = nexus.attention_workspace_size(kv, ql, 40, 8, 2, 0)
    assert splits > 1
    o, lse = _run(cache, d_pt, mp, kv, ql, q, 40, 2, split_kv=0)
    for layer in range(2):
        _check(ks, vs, q, o, lse, kv, ql, 5, layer, what="auto split")


def test_max_sequences_per_call():
    """512 sequences, the most one call takes: short ragged caches, some with no
    queries; every row against the oracle, without and with a split."""
    rng = np.random.default_rng(21)
    kv = [int(x) for x in rng.integers(1, 161, 512)]
    ql = [int(rng.integers(0, min(k, 40) + 1)) for k in kv]
    ql[0], ql[511] = 0, kv[511]
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, seed=21)
    for split in (1, 3):
        o, lse = _run(cache, d_pt, mp, kv, ql, q, 40, 1, split_kv=split)
        _check(ks, vs, q, o, lse, kv, ql, 5, what=f"512 sequences, split {split}")


def test_split_kv_uneven_pairs():
    """Automatic split over sequences whose tile pairs differ (full pairs, a
    sequence of one tile, pairs with a one-tile tail) and an empty sequence in
    between; every row against the oracle."""
    kv, ql = [9000, 5000, 7000, 300], [64, 0, 25, 50]
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, seed=17)
    _, splits = nexus.attention_workspace_size(kv, ql, 40, 8, 1, 0)
    assert splits > 1
    o, lse = _run(cache, d_pt, mp, kv, ql, q, 40, 1, split_kv=0)
    _check(ks, vs, q, o, lse, kv, ql, 5, what="uneven pairs")


# A tile pair holding one query tile, under a split plan, runs its key range in
# both tile slots (even key tiles in slot A, odd in slot B) and merges the two
# before writing its partial rows. Cases: the last CTA with key tiles 7 | 8,
# where rows 1016..1023 see no key of tile 8 (slot B empty for them); three
# tiles a CTA (the ragged tile in slot A); long ranges with a soft cap; a
# sequence holding only a one-tile pair; transposed V.
@pytest.mark.parametrize("kv,ql,split,vt,cap", [
    (1030, 64, 5, False, None), (1030, 64, 4, True, None), (5000, 64, 3, False, 30.0),
    (4100, 14, 2, True, None), (4100, 14, 7, False, 20.0), (2222, 110, 6, True, 50.0)])
def test_split_kv_one_tile_pair_both_slots(kv, ql, split, vt, cap):
    kv, ql = [kv], [ql]
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, vt=vt, seed=kv[0] + split)
    if cap is None:
        o, lse = _run(cache, d_pt, mp, kv, ql, q, 40, 1, split_kv=split)
    else:
        o = torch.full_like(q, float("nan"))
        lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=DEV)
        nbytes, _ = nexus.attention_workspace_size(kv, ql, 40, 8, 1, split)
        ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=DEV)
        nexus.suffix_attention_softcap(cache, d_pt, 1, mp, kv, ql, q, o, lse, 40, 0, 1,
                                       split_kv=split, workspace=ws, workspace_bytes=nbytes,
                                       softcap=cap)
        assert nexus.device_status() == nexus.OK
    _check(ks, vs, q, o, lse, kv, ql, 5, what=f"one-tile pair split {split}", softcap=cap)


def _runs_of_eight(n_pages, offset, seed):
    """Pages in runs of eight consecutive ids, the runs shuffled, the whole
    order rotated by `offset` so runs start off key-tile boundaries."""
    rng = np.random.default_rng(seed)
    runs = [list(range(i, min(i + 8, n_pages))) for i in range(0, n_pages, 8)]
    rng.shuffle(runs)
    order = [p for r in runs for p in r]
    return np.array(order[offset:] + order[:offset])


# A key tile whose eight page ids are consecutive is copied with one box per
# 64-column half (eight pages each); others page by page. Pages in order (every
# full tile takes the eight-page copies), and runs of eight shuffled and rotated
# (tiles of both kinds, runs starting inside a tile); both V layouts, split and
# unsplit plans, a ragged last tile.
@pytest.mark.parametrize("vt,split,layout", [
    (False, 1, "in order"), (True, 1, "in order"), (False, 4, "in order"), (True, 0, "in order"),
    (False, 1, "runs"), (True, 3, "runs"), (False, 0, "runs+3")])
def test_contiguous_page_runs(vt, split, layout):
    kv, ql = [3001, 1500], [300, 64]
    n_pages = sum(-(-k // 16) for k in kv) + 8
    order = None
    if layout == "in order":
        order = np.arange(n_pages)
    elif layout == "runs":
        order = _runs_of_eight(n_pages, 0, 5)
    else:
        order = _runs_of_eight(n_pages, 3, 6)
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, vt=vt, seed=31 + split, order=order)
    o, lse = _run(cache, d_pt, mp, kv, ql, q, 40, 1, split_kv=split)
    _check(ks, vs, q, o, lse, kv, ql, 5, what=f"pages {layout} split {split} vt {vt}")


def test_reprefill_equals_textbook_causal():
    T = 600
    cache, d_pt, mp, ks, vs, q = _direct_case([T], [T], seed=13)
    o = torch.empty_like(q)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
    nexus.reprefill(cache, d_pt, 1, mp, [T], q, o, lse, 40, 0, 1)
    assert nexus.device_status() == nexus.OK
    _check(ks, vs, q, o, lse, [T], [T], 5, what="reprefill")


# Keys planted along a direction u that every query shares (q = (q0 + u) / 2,
# |u|^2 = 128), so that a planted key's score a (64 +- 6) stands far above the
# others (std ~8): the running max jumps by more than 2^8 (log2 units, 62.7 in
# raw score) in the last 48 keys of key tile 1 (key 228: the part of P computed
# after the first 80 keys' P is released), in the first 80 keys of tile 3 (key
# 424), and by about the threshold in tile 4 (key 612: some rows move, some do
# not), for every row at or after the key. One key then carries nearly all of a
# row's weight, at up to 2^8 where the max stays, so its bf16 P alone is off by
# up to 2^-9 of |v|: V is scaled by 1/4 to keep the outputs where 1e-2 holds
# (a wrong rescale of O or l would miss by ~|v|).
_PLANTED = {228: 2.0, 424: 3.5, 612: 4.6}


@pytest.mark.parametrize("vt,split,cap", [(False, 1, None), (True, 1, None), (False, 3, None),
                                          (True, 3, None), (False, 1, 50.0), (True, 3, 50.0)])
def test_running_max_moves_inside_a_tile(vt, split, cap):
    T = 640
    g = torch.Generator().manual_seed(7)
    u = torch.randn(128, generator=g)
    u = u / u.norm() * 128 ** 0.5

    def plant(i, k):
        k = k.clone()
        for key, a in _PLANTED.items():
            k[:, key] = (a * u).to(k.dtype).to(k.device)
        return k

    cache, d_pt, mp, ks, vs, q = _direct_case([T], [T], vt=vt, seed=41 + split, k_edit=plant,
                                              vscale=0.25)
    q = (0.5 * q.float() + 0.5 * u.to(DEV)).to(torch.bfloat16)
    if cap is None:
        o, lse = _run(cache, d_pt, mp, [T], [T], q, 40, 1, split_kv=split)
    else:
        o = torch.full_like(q, float("nan"))
        lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=DEV)
        nbytes, _ = nexus.attention_workspace_size([T], [T], 40, 8, 1, split)
        ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=DEV)
        nexus.suffix_attention_softcap(cache, d_pt, 1, mp, [T], [T], q, o, lse, 40, 0, 1,
                                       split_kv=split, workspace=ws, workspace_bytes=nbytes,
                                       softcap=cap)
        assert nexus.device_status() == nexus.OK
    _check(ks, vs, q, o, lse, [T], [T], 5, what=f"planted maxima vt {vt} split {split} cap {cap}",
           softcap=cap)


def test_attention_repeat_runs_bit_stable():
    cache, d_pt, mp, ks, vs, q = _direct_case([2000], [300], seed=14)
    o1, l1 = _run(cache, d_pt, mp, [2000], [300], q, 40, 1)
    o2, l2 = _run(cache, d_pt, mp, [2000], [300], q, 40, 1)
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(l1, l2)


# ------------------------------------------------------- end to end
def _e2e_session(case, si, R, layers, Hq=40, split_kv=1, sample_rows=None, seed=0):
    """Splice already done; attention of the last R positions over the spliced
    cache on `layers`, checked against oracle splice + oracle attention."""
    w = case.w
    s = w.sessions[si]
    T = w.spliced_len(s)
    q = randn_bf16((len(layers), R, Hq, 128), 5000 + seed, DEV)
    o = torch.empty_like(q)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
    nbytes, _ = nexus.attention_workspace_size([T], [R], Hq, w.n_kv_heads, 1, split_kv)
    ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=DEV)
    for li, layer in enumerate(layers):
        nexus.suffix_attention(case.cache, case.d_pt, case.n_rows, case.max_pages, [T], [R],
                               q[li:li + 1], o[li:li + 1], lse[li:li + 1], Hq, layer, layer + 1,
                               rows=[2 * si + 1], split_kv=split_kv, workspace=ws,
                               workspace_bytes=nbytes)
    assert nexus.device_status() == nexus.OK
    live_k, live_v = case.live(si)
    for li, layer in enumerate(layers):
        want_k, want_v = oracle.splice_sequence(f64(live_k[[layer]]), f64(live_v[[layer]]),
                                                case.inserts_f64(si, [layer]), w.rope_theta)
        rows = np.arange(R) if sample_rows is None else sample_rows
        pos = oracle.suffix_positions(T, R)[rows]
        kmax = int(pos.max()) + 1
        want_o, want_l = oracle.attention(f64(q[li, rows]), want_k[0, :kmax], want_v[0, :kmax],
                                          pos, Hq // w.n_kv_heads)
        assert_attn_close(f64(o[li, rows]), want_o, f64(lse[li, rows]), want_l,
                          f"e2e layer {layer}")


@pytest.mark.parametrize("name", ["c1", "c2"])
def test_end_to_end_single_layer(name):
    w = workload(name)
    case = SplicedCase(w, DEV)
    case.splice()
    s = w.sessions[0]
    R = nexus.suffix_len(s.suffix_span, s.suffix_pct)
    assert R == oracle.redecode_len(s.suffix_span, 0, 256, s.suffix_pct, 4)
    _e2e_session(case, 0, R, [0])


@pytest.mark.parametrize("pct", [25, 50, 100])
def test_end_to_end_c3_transposed_v(pct):
    w = workload("c3")
    case = SplicedCase(w, DEV)
    case.splice()
    R = nexus.suffix_len(2192, pct)
    rows = np.random.default_rng(pct).choice(R, size=min(R, 96), replace=False)
    _e2e_session(case, 0, R, [0, 47], sample_rows=np.sort(rows), seed=pct)


def test_end_to_end_c5_split_kv_full_size():
    w = workload("c5")
    case = SplicedCase(w, DEV)
    case.splice()
    _e2e_session(case, 0, 64, [5, 40], split_kv=0, seed=7)


def test_c5_reprefill_full_size_sampled_rows():
    """Path B: causal self-attention of the 32768-token pre-splice context."""
    w = workload("c5")
    case = SplicedCase(w, DEV)
    T = w.sessions[0].n_past
    layer = 17
    q = randn_bf16((1, T, 40, 128), 777, DEV)
    o = torch.empty_like(q)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
    nexus.reprefill(case.cache, case.d_pt, case.n_rows, case.max_pages, [T], q, o, lse, 40,
                    layer, layer + 1, rows=[0])
    assert nexus.device_status() == nexus.OK
    rng = np.random.default_rng(3)
    rows = np.sort(np.concatenate([[0, 1, 24, 25, 127, 128, T - 1],
                                   rng.choice(T, size=57, replace=False)]))
    kmax = int(rows.max()) + 1
    live_k, live_v = case.live(0)
    want_o, want_l = oracle.attention(f64(q[0, rows]), f64(live_k[layer, :kmax]),
                                      f64(live_v[layer, :kmax]), rows, 5)
    assert_attn_close(f64(o[0, rows]), want_o, f64(lse[0, rows]), want_l, "c5 reprefill")


def test_end_to_end_c4_varlen_full_size():
    """c4: 32 sessions x 48 layers spliced in one launch, then one varlen suffix
    attention call per sampled layer over all 32 sessions (50 % of each session's
    spliced span re-decoded), checked on sampled rows of sampled sessions."""
    w = workload("c4")
    case = SplicedCase(w, DEV, keep_live=False)
    case.splice()
    assert nexus.device_status() == nexus.OK
    kv = [w.spliced_len(s) for s in w.sessions]
    ql = [nexus.suffix_len(s.suffix_span, s.suffix_pct) for s in w.sessions]
    assert ql == [oracle.redecode_len(s.suffix_span, 0, 256, s.suffix_pct, 4) for s in w.sessions]
    rows = [2 * i + 1 for i in range(len(w.sessions))]
    offs = np.concatenate([[0], np.cumsum(ql)])
    rng = np.random.default_rng(44)
    for layer in (0, 47):
        q = randn_bf16((1, int(offs[-1]), 40, 128), 4400 + layer, DEV)
        o = torch.empty_like(q)
        lse = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
        nexus.suffix_attention(case.cache, case.d_pt, case.n_rows, case.max_pages, kv, ql, q, o,
                               lse, 40, layer, layer + 1, rows=rows, split_kv=0)
        assert nexus.device_status() == nexus.OK
        for si in (0, 5, 19, 31):
            live_k, live_v = case.live(si)
            want_k, want_v = oracle.splice_sequence(f64(live_k[[layer]]), f64(live_v[[layer]]),
                                                    case.inserts_f64(si, [layer]), w.rope_theta)
            del live_k, live_v
            sel = np.sort(rng.choice(ql[si], size=min(12, ql[si]), replace=False))
            pos = oracle.suffix_positions(kv[si], ql[si])[sel]
            kmax = int(pos.max()) + 1
            want_o, want_l = oracle.attention(f64(q[0, offs[si] + sel]), want_k[0, :kmax],
                                              want_v[0, :kmax], pos, 5)
            assert_attn_close(f64(o[0, offs[si] + sel]), want_o, f64(lse[0, offs[si] + sel]),
                              want_l, f"c4 session {si} layer {layer}")


# ------------------------------------------------ soft-capped attention (Sec. V-B)
# The last two cases push the scores far into tanh's curved range with a large
# cap; V is scaled so that the concentrated outputs stay below 2, where half a
# bf16 ulp of the stored output is under 4e-3.
@pytest.mark.parametrize("cap,vt,split,qscale,vscale", [
    (50.0, True, 1, 1.0, 1.0), (50.0, False, 1, 1.0, 1.0), (5.0, True, 1, 8.0, 1.0),
    (1.5, False, 1, 20.0, 1.0), (30.0, True, 7, 1.0, 1.0), (50.0, False, 1, 16.0, 0.25),
    (15.0, True, 3, 8.0, 0.25)])
def test_softcap_attention(cap, vt, split, qscale, vscale):
    kv, ql = [1500, 333], [300, 17]
    cache, d_pt, mp, ks, vs, q = _direct_case(kv, ql, vt=vt, seed=int(cap) + split,
                                              vscale=vscale)
    q = (q.float() * qscale).to(torch.bfloat16)       # larger scores: more of them saturate
    o = torch.full_like(q, float("nan"))
    lse = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=DEV)
    nbytes, _ = nexus.attention_workspace_size(kv, ql, 40, 8, 1, split)
    ws = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=DEV)
    nexus.suffix_attention_softcap(cache, d_pt, 2, mp, kv, ql, q, o, lse, 40, 0, 1,
                                   split_kv=split, workspace=ws, workspace_bytes=nbytes,
                                   softcap=cap)
    assert nexus.device_status() == nexus.OK
    _check(ks, vs, q, o, lse, kv, ql, 5, what=f"softcap {cap}", softcap=cap)


def test_end_to_end_c3_softcap():
    """c3 (token-innermost V, 48 layers) with a Gemma-2-style cap of 50 over the
    whole 2192-row suffix, sampled rows of two layers."""
    w = workload("c3")
    case = SplicedCase(w, DEV)
    case.splice()
    s0 = w.sessions[0]
    T, R = w.spliced_len(s0), 2192
    q = randn_bf16((1, R, 40, 128), 3300, DEV)
    rows = np.sort(np.random.default_rng(33).choice(R, size=64, replace=False))
    for layer in (0, 47):
        o = torch.empty_like(q)
        lse = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
        nexus.suffix_attention_softcap(case.cache, case.d_pt, case.n_rows, case.max_pages, [T],
                                       [R], q, o, lse, 40, layer, layer + 1, rows=[1],
                                       split_kv=1, softcap=50.0)
        assert nexus.device_status() == nexus.OK
        live_k, live_v = case.live(0)
        want_k, want_v = oracle.splice_sequence(f64(live_k[[layer]]), f64(live_v[[layer]]),
                                                case.inserts_f64(0, [layer]), w.rope_theta)
        pos = oracle.suffix_positions(T, R)[rows]
        want_o, want_l = oracle.attention(f64(q[0, rows]), want_k[0], want_v[0], pos, 5,
                                          softcap=50.0)
        assert_attn_close(f64(o[0, rows]), want_o, f64(lse[0, rows]), want_l,
                          f"c3 softcap layer {layer}")
