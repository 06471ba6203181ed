"""Host logic of the C-ABI library on the CPU: exports, Eq. 2 policy, page
pool, splice planner and argument validation (no device compute is called)."""
import ctypes
import os
import re
from fractions import Fraction

import numpy as np
import torch
import pytest

import oracle
import oracle_pins as P
from paper_2608_20397_gb300 import nexus

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built_library():
    if not os.path.exists(nexus.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    nexus.lib()


def header_functions():
    src = open(os.path.join(ROOT, "include", "nexus.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(nexus_[a-z0-9_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    names = header_functions()
    assert len(names) >= 20
    L = ctypes.CDLL(nexus.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(nexus.EXPORTED)
    assert nexus.lib().nexus_version() == 1


def test_status_strings():
    for code in range(10):
        assert nexus.status_string(code)


# ----------------------------------------------------------------- policy
def test_policy_matches_table1_through_the_library():
    P.pin_table1(lambda n, M=256, R_base=5, K=4: nexus.recompute_pct(n, (M, R_base, K)))


def test_policy_matches_oracle_exactly():
    for K in (2, 4, 16):
        for Rb in (0, 5, 37, 100):
            for n in list(range(0, 3000, 37)) + [255, 256, 257, K * 256, K * 256 + 1]:
                pol = (256, Rb, K)
                assert nexus.recompute_pct(n, pol) == oracle.recompute_pct(n, 256, Rb, K)
                for S in (0, 1, 7, 64, 128, 2192, 32768):
                    assert nexus.redecode_len(S, n, pol) == oracle.redecode_len(S, n, 256, Rb, K)


def test_suffix_len_is_integer_ceil():
    for S in range(0, 300, 7):
        for pct in (0, 1, 25, 33, 50, 99, 100):
            assert nexus.suffix_len(S, pct) == -(-S * pct // 100)


def test_check_splice_declines_bare_deep_splice():
    pol = (256, 5, 4)
    assert nexus.check_splice(256, 128, 0, pol) == nexus.OK           # at P: bare splice allowed
    assert nexus.check_splice(257, 128, 0, pol) == nexus.EDECLINED    # past P: must redecode
    need = nexus.redecode_len(128, 600, pol)
    assert nexus.check_splice(600, 128, need, pol) == nexus.OK
    assert nexus.check_splice(600, 128, need - 1, pol) == nexus.EDECLINED


def test_policy_rejects_bad_parameters():
    with pytest.raises(nexus.NexusError):
        nexus.recompute_pct(10, (256, 5, 1))
    with pytest.raises(nexus.NexusError):
        nexus.recompute_pct(10, (0, 5, 4))
    with pytest.raises(nexus.NexusError):
        nexus.redecode_len(-1, 10)


# -------------------------------------------------------------- page pool
def test_page_pool_order_alloc_free():
    order = np.random.default_rng(0).permutation(40).astype(np.int32)
    pool = nexus.PagePool(40, order)
    a = pool.alloc(10)
    assert np.array_equal(a, order[:10])
    assert pool.available() == 30
    pool.free(a[:3])
    assert pool.available() == 33
    with pytest.raises(nexus.NexusError) as e:
        pool.free(a[:1])                       # double free
    assert e.value.code == nexus.EINVAL
    with pytest.raises(nexus.NexusError) as e:
        pool.free([99])
    assert e.value.code == nexus.ERANGE
    with pytest.raises(nexus.NexusError) as e:
        pool.alloc(34)
    assert e.value.code == nexus.ENOMEM
    assert pool.available() == 33
    b = pool.alloc(30)
    assert np.array_equal(b, order[10:40])     # pool order first, freed pages last
    assert np.array_equal(pool.alloc(3), a[:3])


def test_page_pool_rejects_bad_order():
    with pytest.raises(nexus.NexusError):
        nexus.PagePool(4, [0, 1, 1, 2])


# ---------------------------------------------------------------- planner
def _apply_segments(pool_k, pool_v, pts, segs, blocks_k, blocks_v, theta=1.0e6):
    """Executes planner segments with NumPy on logical arrays (test-side interpreter)."""
    out_k = pool_k.copy()
    out_v = pool_v.copy()
    for s in segs:
        for r in range(s.n_tokens):
            dpos = s.dst_start + r
            dpg, dsl = pts[s.dst_row][dpos // 16], dpos % 16
            if s.src_kind == nexus.SRC_BLOCK:
                k = blocks_k[s.src_index][:, s.src_start + r]
                v = blocks_v[s.src_index][:, s.src_start + r]
            else:
                spos = s.src_start + r
                spg, ssl = pts[s.src_index][spos // 16], spos % 16
                k = pool_k[:, spg, :, ssl]
                v = pool_v[:, spg, :, ssl]
            out_k[:, dpg, :, dsl] = oracle.rerotate(k, s.delta, theta)
            if not (s.flags & nexus.SEG_K_ONLY):
                out_v[:, dpg, :, dsl] = v
    return out_k, out_v


@pytest.mark.parametrize("case", range(8))
def test_planner_segments_reproduce_oracle_splice(case):
    rng = np.random.default_rng(100 + case)
    nL, H, d = 2, 2, 8
    n_past = int(rng.integers(0, 120))
    n_ins = int(rng.integers(1, 5))
    if case == 0:
        depths = [n_past] * n_ins               # append at the cursor
    elif case == 1:
        depths = [0] * n_ins                    # prepend
    else:
        depths = sorted(int(x) for x in rng.integers(0, n_past + 1, size=n_ins))
    lens = [int(x) for x in rng.integers(0 if case == 2 else 1, 40, size=n_ins)]
    anchors = [int(x) for x in rng.integers(0, 60, size=n_ins)]
    n_pages, max_pages = 64, 24
    order = rng.permutation(n_pages).astype(np.int32)
    pool = nexus.PagePool(n_pages, order)
    old_pt = np.full(max_pages, -1, np.int32)
    np_old = -(-n_past // 16)
    old_pt[:np_old] = pool.alloc(np_old)
    pool_k = rng.standard_normal((nL, n_pages, H, 16, d))
    pool_v = rng.standard_normal((nL, n_pages, H, 16, d))
    live_k = oracle.paged_gather(pool_k, old_pt, n_past)
    live_v = oracle.paged_gather(pool_v, old_pt, n_past)
    bks = [rng.standard_normal((nL, L, H, d)) for L in lens]
    bvs = [rng.standard_normal((nL, L, H, d)) for L in lens]
    blocks = [nexus.block(0x1000, 0x1000, L, m0, nL, H) for L, m0 in zip(lens, anchors)]
    new_pt, segs, freed = nexus.plan_splice(pool, old_pt, n_past, max_pages, blocks,
                                            list(zip(depths, range(n_ins))), 0, 1)
    T = n_past + sum(lens)
    assert np.all(new_pt[: -(-T // 16)] >= 0) and np.all(new_pt[-(-T // 16):] == -1)
    if depths[0] == n_past:
        assert np.array_equal(new_pt[:np_old], old_pt[:np_old]) and len(freed) == 0
    else:
        keep = depths[0] // 16
        assert np.array_equal(new_pt[:keep], old_pt[:keep])
        assert set(new_pt[keep: -(-T // 16)]).isdisjoint(set(old_pt[:np_old]))
        assert sorted(freed) == sorted(old_pt[keep:np_old])
    out_k, out_v = _apply_segments(pool_k, pool_v, [old_pt, new_pt], segs, bks, bvs)
    got_k = oracle.paged_gather(out_k, new_pt, T)
    got_v = oracle.paged_gather(out_v, new_pt, T)
    want_k, want_v = oracle.splice_sequence(live_k, live_v,
                                            [(p, bk, bv, m0) for p, bk, bv, m0 in
                                             zip(depths, bks, bvs, anchors)])
    assert np.array_equal(got_v, want_v)
    assert np.max(np.abs(got_k - want_k), initial=0) < 1e-12


def test_planner_errors():
    pool = nexus.PagePool(8)
    blk = [nexus.block(0x1000, 0x1000, 100, 0, 1)]
    with pytest.raises(nexus.NexusError) as e:          # does not fit max_pages
        nexus.plan_splice(pool, np.zeros(4, np.int32), 0, 4, blk, [(0, 0)], 0, 1)
    assert e.value.code == nexus.ERANGE
    with pytest.raises(nexus.NexusError) as e:          # pool too small (13 pages for 200 rows)
        nexus.plan_splice(pool, np.zeros(16, np.int32), 0, 16,
                          [nexus.block(0x1000, 0x1000, 200, 0, 1)], [(0, 0)], 0, 1)
    assert e.value.code == nexus.ENOMEM
    assert pool.available() == 8
    with pytest.raises(nexus.NexusError) as e:          # depths must not decrease
        nexus.plan_splice(pool, np.array([0, 1, -1, -1], np.int32), 20, 16,
                          [nexus.block(0x1000, 0x1000, 4, 0, 1)] * 2, [(10, 0), (5, 1)], 0, 1)
    assert e.value.code == nexus.EINVAL
    with pytest.raises(nexus.NexusError) as e:          # insertion inside needs a second row
        nexus.plan_splice(pool, np.array([0, 1, -1, -1], np.int32), 20, 16,
                          [nexus.block(0x1000, 0x1000, 4, 0, 1)], [(5, 0)], 0, 0)
    assert e.value.code == nexus.EINVAL


# --------------------------------------------------- validation before launch
FAKE = 0x7F0000000000   # never dereferenced: every call below fails validation first


def _cache(**kw):
    args = dict(k_pool=FAKE, v_pool=FAKE, n_pages=64, n_layers=2)
    args.update(kw)
    return nexus.kv_cache(**args)


def test_splice_rejects_rope_mismatch_and_layout():
    cache = _cache()
    pts = np.zeros((2, 8), np.int32)
    seg = [(nexus.SRC_BLOCK, 0, 0, 0, 0, 4, 0, 0)]
    for bad, code in ((dict(rope_theta=1.0e4), nexus.EROPE_MISMATCH),
                      (dict(rope_freq_scale=0.5), nexus.EROPE_MISMATCH),
                      (dict(rope_type=nexus.ROPE_GPTJ), nexus.EROPE_MISMATCH),
                      (dict(n_layers=3), nexus.ELAYOUT),
                      (dict(n_kv_heads=4), nexus.ELAYOUT)):
        args = dict(k=FAKE, v=FAKE, n_tokens=8, base_pos=0, n_layers=2)
        args.update(bad)
        with pytest.raises(nexus.NexusError) as e:
            nexus.splice_kv(cache, FAKE, pts, 2, 8, [nexus.block(**args)], seg, 0, 2, stream=0)
        assert e.value.code == code, bad


def test_splice_rejects_ranges_and_overlaps():
    cache = _cache()
    blk = [nexus.block(FAKE, FAKE, 8, 0, 2)]
    pts = np.array([[0, 1, 2, 3], [4, 5, 6, 7]], np.int32)
    cases = [
        ([(nexus.SRC_BLOCK, 0, 0, 0, 60, 8, 0, 0)], nexus.ERANGE),        # past max_pages
        ([(nexus.SRC_BLOCK, 0, 4, 0, 0, 8, 0, 0)], nexus.ERANGE),         # past block end
        ([(nexus.SRC_BLOCK, 3, 0, 0, 0, 8, 0, 0)], nexus.ERANGE),         # no such block
        ([(nexus.SRC_CACHE, 0, 0, 2, 0, 8, 0, 0)], nexus.ERANGE),         # no such row
        ([(nexus.SRC_BLOCK, 0, 0, 0, 0, 8, 0, 0),
          (nexus.SRC_BLOCK, 0, 0, 0, 4, 4, 0, 0)], nexus.EOVERLAP),       # written twice
    ]
    for segs, code in cases:
        with pytest.raises(nexus.NexusError) as e:
            nexus.splice_kv(cache, FAKE, pts, 2, 4, blk, segs, 0, 2, stream=0)
        assert e.value.code == code, segs
    # a tail moved within the same pages: rows 0..7 are read while rows 4..11 are written
    with pytest.raises(nexus.NexusError) as e:
        nexus.splice_kv(cache, FAKE, pts, 2, 4, blk, [(nexus.SRC_CACHE, 0, 0, 0, 4, 8, 4, 0)],
                        0, 2, stream=0)
    assert e.value.code == nexus.EOVERLAP
    # page id out of the pool
    bad = pts.copy()
    bad[1, 0] = 64
    with pytest.raises(nexus.NexusError) as e:
        nexus.splice_kv(cache, FAKE, bad, 2, 4, blk, [(nexus.SRC_BLOCK, 0, 0, 1, 0, 8, 0, 0)],
                        0, 2, stream=0)
    assert e.value.code == nexus.ERANGE
    with pytest.raises(nexus.NexusError) as e:          # layer range
        nexus.splice_kv(cache, FAKE, pts, 2, 4, blk, [], 1, 3, stream=0)
    assert e.value.code == nexus.ERANGE


def test_cache_shape_checks():
    with pytest.raises(nexus.NexusError) as e:
        nexus.copy_pages(_cache(v_pool=FAKE + 8), [0], [1], 0, 1, stream=0)
    assert e.value.code == nexus.ELAYOUT
    c = _cache()
    c.head_dim = 64
    with pytest.raises(nexus.NexusError) as e:
        nexus.copy_pages(c, [0], [1], 0, 1, stream=0)
    assert e.value.code == nexus.ELAYOUT
    with pytest.raises(nexus.NexusError) as e:
        nexus.copy_pages(_cache(), [0, 1], [1, 2], 0, 1, stream=0)   # 1 is source and destination
    assert e.value.code == nexus.EOVERLAP
    with pytest.raises(nexus.NexusError) as e:
        nexus.copy_pages(_cache(), [0], [64], 0, 1, stream=0)
    assert e.value.code == nexus.ERANGE


def test_attention_argument_checks():
    c = _cache()
    with pytest.raises(nexus.NexusError) as e:          # q_len > kv_len
        nexus.suffix_attention(c, FAKE, 1, 8, [10], [11], FAKE, FAKE, stream=0)
    assert e.value.code == nexus.EINVAL
    with pytest.raises(nexus.NexusError) as e:          # kv_len beyond the page table
        nexus.suffix_attention(c, FAKE, 1, 8, [200], [10], FAKE, FAKE, stream=0)
    assert e.value.code == nexus.ERANGE
    with pytest.raises(nexus.NexusError) as e:          # 40 heads over 16 KV heads
        nexus.suffix_attention(_cache(n_kv_heads=16), FAKE, 1, 8, [10], [5], FAKE, FAKE,
                               n_q_heads=40, stream=0)
    assert e.value.code == nexus.EINVAL
    with pytest.raises(nexus.NexusError) as e:          # split partials need a workspace
        nexus.suffix_attention(c, FAKE, 1, 4096, [60000], [64], FAKE, FAKE, split_kv=4, stream=0)
    assert e.value.code == nexus.ENOMEM
    with pytest.raises(nexus.NexusError) as e:          # misaligned q
        nexus.suffix_attention(c, FAKE, 1, 8, [10], [5], FAKE + 2, FAKE, stream=0)
    assert e.value.code == nexus.ELAYOUT


def test_workspace_size_and_split_choice():
    n, s = nexus.attention_workspace_size([34816], [64], 40, 8, 1, 0)
    assert s > 1 and n == s * 64 * 40 * (128 * 4 + 4)
    n, s = nexus.attention_workspace_size([32768], [32768], 40, 8, 1, 0)
    assert s == 1 and n == 0
    n, s = nexus.attention_workspace_size([34816], [64], 40, 8, 1, 7)
    assert s == 7 and n == 7 * 64 * 40 * 516
    n, s = nexus.attention_workspace_size([34816], [64], 40, 8, 1, 100)   # taken as 32
    assert s == 32 and n == 32 * 64 * 40 * 516
    n, s = nexus.attention_workspace_size([10] * 512, [1] * 512, 40, 8, 1, 1)
    assert s == 1 and n == 0
    assert nexus.attention_workspace_size([10] * 513, [1] * 513, 40, 8, 1, 1) == (0, 0)
    assert nexus.attention_workspace_size([10], [11], 40, 8, 1, 1) == (0, 0)


def test_split_choice_matches_the_measured_optima():
    """On 152 SMs (a GB300, and the count taken without a device) the planner
    picks the split counts that timing sweeps on the GB300 found fastest, one
    layer each: the c5 suffix (64 queries over 34816 keys) 10 for two-tile pairs
    (9 for one-tile pairs, which the size query does not show), c2 (1138
    queries over 8648 keys) 3, c3 at 25 / 50 % (548 / 1096 over 9216) 3, and
    c3 at 100 % (2192 queries, rows that see few keys) no split."""
    assert nexus.attention_workspace_size([34816], [64], 40, 8, 1, 0)[1] == 10
    assert nexus.attention_workspace_size([8648], [1138], 40, 8, 1, 0)[1] == 3
    assert nexus.attention_workspace_size([9216], [548], 40, 8, 1, 0)[1] == 3
    assert nexus.attention_workspace_size([9216], [1096], 40, 8, 1, 0)[1] == 3
    assert nexus.attention_workspace_size([9216], [2192], 40, 8, 1, 0)[1] == 1


def test_zero_work_calls_succeed_before_any_launch():
    """Calls with nothing to compute return OK after validation and before any
    launch or memory access (the FAKE pointers are never dereferenced)."""
    c = _cache()
    nexus.suffix_attention(c, FAKE, 2, 8, [10, 50], [0, 0], FAKE, FAKE, stream=0)
    nexus.suffix_attention(c, FAKE, 2, 8, [10, 50], [0, 0], FAKE, FAKE, split_kv=0, stream=0)
    nexus.reprefill(c, FAKE, 1, 8, [0], FAKE, FAKE, stream=0)
    nexus.suffix_attention(c, FAKE, 1, 8, [10], [5], FAKE, FAKE, layer_begin=1, layer_end=1,
                           stream=0)
    nexus.suffix_qkv(c, FAKE, 2, 8, [10, 3], [0, 0], FAKE, FAKE, None, FAKE, hidden=64, stream=0)
    tools = torch.zeros((16, 64), dtype=torch.int8)
    nexus.slb_route(tools, torch.zeros(16), torch.zeros((0, 64), dtype=torch.int8),
                    torch.zeros(0), torch.zeros((0, 2), dtype=torch.int32), torch.zeros((0, 2)),
                    torch.zeros(0, dtype=torch.int32), torch.zeros(16, dtype=torch.uint8),
                    stream=0)
    blk = [nexus.block(FAKE, FAKE, 8, 0, 2)]
    pts = np.array([[0, 1, 2, 3], [4, 5, 6, 7]], np.int32)
    nexus.splice_kv(c, FAKE, pts, 2, 4, blk, [], 0, 2, stream=0)
    nexus.splice_kv(c, FAKE, pts, 2, 4, blk, [(nexus.SRC_BLOCK, 0, 0, 0, 0, 8, 0, 0)], 1, 1,
                    stream=0)


def test_attention_rejects_more_than_512_sequences():
    with pytest.raises(nexus.NexusError) as e:
        nexus.suffix_attention(_cache(), FAKE, 513, 8, [10] * 513, [1] * 513, FAKE, FAKE,
                               stream=0)
    assert e.value.code == nexus.EINVAL


def test_softcap_must_be_positive():
    for cap in (0.0, -1.0, float("nan"), float("inf")):
        with pytest.raises(nexus.NexusError) as e:
            nexus.suffix_attention_softcap(_cache(), FAKE, 1, 8, [10], [5], FAKE, FAKE,
                                           softcap=cap, stream=0)
        assert e.value.code == nexus.EINVAL


def test_qkv_argument_checks():
    c = _cache()
    def call(kv=(40,), ql=(8,), hidden=64, x=FAKE, layer=0, hpt=None, rows=None, max_pages=8,
             n_rows=1, bias=None):
        nexus.suffix_qkv(c, FAKE, n_rows, max_pages, list(kv), list(ql), x, FAKE, bias, FAKE,
                         layer=layer, rows=rows, h_page_tables=hpt, hidden=hidden, stream=0)

    def code(**kw):
        with pytest.raises(nexus.NexusError) as e:
            call(**kw)
        return e.value.code

    assert code(ql=(41,)) == nexus.EINVAL                 # q_len > kv_len
    assert code(kv=(200,)) == nexus.ERANGE                # beyond the page table
    assert code(layer=2) == nexus.ERANGE                  # the cache has two layers
    assert code(hidden=60) == nexus.ELAYOUT               # rows of x not 16-byte multiples
    assert code(x=FAKE + 8) == nexus.ELAYOUT              # misaligned x
    assert code(bias=FAKE + 4) == nexus.ELAYOUT           # misaligned bias
    assert code(hidden=0) == nexus.EINVAL
    assert code(rows=[1]) == nexus.ERANGE                 # page-table row outside the table
    assert code(kv=((1 << 24) + 1,), max_pages=(1 << 20) + 1) == nexus.ERANGE   # float positions
    pt = np.arange(16, dtype=np.int32).reshape(2, 8)
    bad = pt.copy()
    bad[0, 2] = 64                                        # pool has 64 pages
    assert code(hpt=bad, n_rows=2) == nexus.ERANGE
    shared = pt.copy()
    shared[1, 2] = shared[0, 2]                           # both rows write page 2's slots
    assert code(kv=(40, 40), ql=(8, 8), rows=[0, 1], hpt=shared, n_rows=2) == nexus.EOVERLAP
    call(kv=(40, 40), ql=(0, 0), rows=[0, 1], hpt=pt, n_rows=2)   # nothing to do: no launch


def test_slb_quantize_matches_oracle():
    r = np.random.default_rng(41)
    x = r.standard_normal((40, 768)).astype(np.float32) * r.uniform(1e-3, 1e3, (40, 1)).astype(np.float32)
    x[3] = 0.0
    x[4, :4] = [127.0, 2.5, -3.5, 0.5]        # scale exactly 1: halves go to even
    x[4, 4:] = 0.0
    x[5] = r.integers(-127, 128, 768).astype(np.float32) * np.float32(0.125)
    c, s = nexus.slb_quantize(x)
    c2, s2 = oracle.slb_quantize(x)
    assert np.array_equal(c, c2) and np.array_equal(s, s2)
    assert list(c[4, :4]) == [127, 2, -4, 0]
    bad = np.zeros((1, 8), np.float32)
    bad[0, 1] = np.inf
    with pytest.raises(nexus.NexusError) as e:
        nexus.slb_quantize(bad)
    assert e.value.code == nexus.EINVAL


def test_slb_route_argument_checks():
    L = nexus.lib()
    ws = nexus.slb_workspace_size(250)
    assert ws >= 256 + 32 * 2 * 8 and nexus.slb_workspace_size(0) == 0
    def call(n_tools=250, dim=768, nq=1, tau=0.0136, tools=FAKE, queries=FAKE, ws_bytes=ws,
             wsp=FAKE):
        return L.nexus_slb_route(tools, FAKE, n_tools, dim, queries, FAKE, nq, tau, FAKE, FAKE,
                                 FAKE, wsp, ws_bytes, None)
    assert call(n_tools=0) == nexus.EINVAL
    assert call(dim=2) == nexus.EINVAL
    assert call(dim=8192) == nexus.EINVAL
    assert call(dim=770) == nexus.ELAYOUT
    assert call(tools=FAKE + 4) == nexus.ELAYOUT
    assert call(tau=float("nan")) == nexus.EINVAL
    assert call(ws_bytes=ws - 1) == nexus.ENOMEM
    assert call(wsp=None) == nexus.ENOMEM
    assert call(nq=0) == nexus.OK                # nothing to scan: no launch


def test_host_staging_argument_checks():
    L = nexus.lib()
    out = ctypes.c_void_p(1234)
    assert L.nexus_host_alloc(0, ctypes.byref(out)) == nexus.EINVAL and not out.value
    assert L.nexus_host_alloc(4096, None) == nexus.EINVAL
    assert L.nexus_host_alloc(1 << 60, ctypes.byref(out)) == nexus.EINVAL
    assert L.nexus_host_free(None, 4096) == nexus.OK
    # memory the library did not map is refused before anything is unmapped
    buf = ctypes.create_string_buffer(1 << 16)
    assert L.nexus_host_free(ctypes.c_void_p(ctypes.addressof(buf)), 1 << 16) == nexus.EINVAL
    assert L.nexus_host_free(ctypes.c_void_p(ctypes.addressof(buf)), 0) == nexus.EINVAL
    buf[0] = b"x"                                   # still mapped and writable
    import torch
    if not torch.cuda.is_available():
        # no driver to register with: nothing is left mapped and NULL comes back
        assert L.nexus_host_alloc(1 << 20, ctypes.byref(out)) == nexus.ECUDA and not out.value
        with pytest.raises(nexus.NexusError):
            nexus.host_empty((4, 4), torch.bfloat16)


def test_selftest_wait_argument_checks():
    L = nexus.lib()
    assert L.nexus_selftest_wait(0, None) == nexus.EINVAL
    assert L.nexus_selftest_wait(1000001, None) == nexus.EINVAL
