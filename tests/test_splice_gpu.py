"""Splice scatter + RoPE delta re-rotation + page copies on the GPU against
the fp64 oracle (Sec. III-B, Sec. V-A, Sec. V-B, Sec. V-D)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import SplicedCase, assert_k_close, f64, gather_rows, new_pools, write_rows
from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import randn_bf16, workload

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0") if torch.cuda.is_available() else None


def _check_session(case, si, layers):
    """Spliced session si against the oracle on the given layers: V and delta-0 K
    rows bit-exact, re-rotated K within tolerance."""
    w = case.w
    s = w.sessions[si]
    T = w.spliced_len(s)
    got_k, got_v = gather_rows(case.kp, case.vp, case.h_pt[2 * si + 1], T, case.vt, layers)
    live_k, live_v = case.live(si)
    want_k, want_v = oracle.splice_sequence(f64(live_k[layers]), f64(live_v[layers]),
                                            case.inserts_f64(si, layers), w.rope_theta)
    del live_k, live_v
    gk, gv = f64(got_k), f64(got_v)
    assert np.array_equal(gv, want_v), f"session {si}: V not bit-exact"
    # rows whose delta is 0 (the prefix before the first insert) keep their bits
    d1 = s.inserts[0].depth
    assert np.array_equal(gk[:, :d1], want_k[:, :d1]), f"session {si}: unshifted K changed"
    assert_k_close(gk, want_k, f"session {si}")
    return gk, want_k


@pytest.mark.parametrize("name", ["c1", "c2"])
def test_splice_single_layer_configs(name):
    case = SplicedCase(workload(name), DEV)
    case.splice()
    assert nexus.device_status() == nexus.OK
    _check_session(case, 0, [0])


def test_splice_c3_transposed_v_all_layers():
    case = SplicedCase(workload("c3"), DEV)
    case.splice()
    assert nexus.device_status() == nexus.OK
    # every layer's V is a bit copy: check all 48 against a torch gather
    s = case.w.sessions[0]
    T = case.w.spliced_len(s)
    got_k, got_v = gather_rows(case.kp, case.vp, case.h_pt[1], T, True)
    ins = s.inserts[0]
    live_k, live_v = case.live(0)
    want_v = torch.cat([live_v[:, :ins.depth], case.blk_v[0][0], live_v[:, ins.depth:]], dim=1)
    assert torch.equal(got_v.view(torch.int16), want_v.view(torch.int16))
    assert torch.equal(got_k[:, :ins.depth].view(torch.int16),
                       live_k[:, :ins.depth].view(torch.int16))
    for layers in ([0], [23], [47]):
        _check_session(case, 0, layers)


def test_splice_c4_sessions_shuffled_pages():
    w = workload("c4", n_layers=2)
    case = SplicedCase(w, DEV)
    case.splice()
    assert nexus.device_status() == nexus.OK
    for si in range(len(w.sessions)):
        _check_session(case, si, [0, 1])


def test_splice_c4_full_size_sampled():
    """32 sessions x 48 layers, four inserts each at random depths, shuffled pool
    pages, one launch; V of every layer of the sampled sessions bit-exact, K of
    sampled layers against the oracle."""
    w = workload("c4")
    case = SplicedCase(w, DEV, keep_live=False)
    case.splice()
    assert nexus.device_status() == nexus.OK
    for si in (0, 13, 31):
        s = w.sessions[si]
        T = w.spliced_len(s)
        _, got_v = gather_rows(case.kp, case.vp, case.h_pt[2 * si + 1], T, False)
        _, live_v = case.live(si)
        parts, cur = [], 0
        for j, ins in enumerate(s.inserts):
            parts += [live_v[:, cur:ins.depth], case.blk_v[si][j]]
            cur = ins.depth
        parts.append(live_v[:, cur:])
        assert torch.equal(got_v.view(torch.int16), torch.cat(parts, dim=1).view(torch.int16))
        del got_v, live_v, parts
        _check_session(case, si, [0, 47])


def test_splice_c5_full_size_sampled_layers():
    case = SplicedCase(workload("c5"), DEV)
    case.splice()
    assert nexus.device_status() == nexus.OK
    s = case.w.sessions[0]
    T = case.w.spliced_len(s)
    ins = s.inserts[0]
    got_k, got_v = gather_rows(case.kp, case.vp, case.h_pt[1], T, False)
    _, live_v = case.live(0)
    want_v = torch.cat([live_v[:, :ins.depth], case.blk_v[0][0], live_v[:, ins.depth:]], dim=1)
    assert torch.equal(got_v.view(torch.int16), want_v.view(torch.int16))
    del got_k, got_v, want_v, live_v
    for layers in ([0], [31]):
        _check_session(case, 0, layers)


def test_anchored_splice_is_bit_exact_for_special_values():
    """delta = 0 moves bits: -0.0, NaN payloads and infinities survive (Sec. IV-A)."""
    L, H, n_pages, maxp = 2, 8, 16, 8
    kp, vp = new_pools(L, n_pages, H, False, DEV)
    raw = torch.randint(0, 1 << 16, (L, 40, H, 128), dtype=torch.int32, device=DEV)
    bk = raw.to(torch.int16).view(torch.bfloat16)
    bk.view(torch.int16)[0, 0, 0, :8] = torch.tensor(
        [-32768, 0x7FC1, 0x7F80, -128, 0x7F81, 0x0001, -1, 0x7FFF], dtype=torch.int16, device=DEV)
    bv = bk.flip(1).contiguous()
    cache = nexus.kv_cache(kp, vp, n_pages, L, H)
    blk = nexus.block(bk, bv, 40, 5, L, H)
    h_pt = np.array([[3, 9, 1, 7, -1, -1, -1, -1]], np.int32)
    d_pt = torch.as_tensor(h_pt, device=DEV)
    seg = [(nexus.SRC_BLOCK, 0, 0, 0, 5, 40, 0, 0)]    # written at its anchor: delta 0
    nexus.splice_kv(cache, d_pt, h_pt, 1, maxp, [blk], seg, 0, L)
    assert nexus.device_status() == nexus.OK
    gk, gv = gather_rows(kp, vp, h_pt[0], 45, False)
    assert torch.equal(gk[:, 5:].view(torch.int16), bk.view(torch.int16))
    assert torch.equal(gv[:, 5:].view(torch.int16), bv.view(torch.int16))
    assert torch.equal(gk[:, :5].view(torch.int16), torch.zeros_like(gk[:, :5]).view(torch.int16))


@pytest.mark.parametrize("rope_type", [nexus.ROPE_NEOX, nexus.ROPE_GPTJ])
@pytest.mark.parametrize("delta", [1, -7, 300, 6000, 30000, -30000, 131071])
def test_rerotate_in_place_and_f32(rope_type, delta):
    L, H, n_pages, maxp, n = 3, 8, 40, 16, 200
    kp, vp = new_pools(L, n_pages, H, False, DEV)
    pt = np.random.default_rng(5).permutation(n_pages)[:maxp].astype(np.int32)
    k = randn_bf16((L, n, H, 128), 21, DEV)
    v = randn_bf16((L, n, H, 128), 22, DEV)
    write_rows(kp, vp, pt, k, v, False)
    h_pt = pt[None].copy()
    d_pt = torch.as_tensor(h_pt, device=DEV)
    cache = nexus.kv_cache(kp, vp, n_pages, L, H, rope_type=rope_type)
    rt = "neox" if rope_type == nexus.ROPE_NEOX else "gptj"
    p0, nt = 13, 150
    out32 = torch.empty((L - 1, nt, H, 128), dtype=torch.float32, device=DEV)
    nexus.rope_rerotate_f32(cache, d_pt, h_pt, 1, maxp, 0, p0, nt, delta, 1, L, out32)
    nexus.rope_rerotate(cache, d_pt, h_pt, 1, maxp, 0, p0, nt, delta, 1, L)
    assert nexus.device_status() == nexus.OK
    want = oracle.rerotate(f64(k[1:, p0:p0 + nt]), delta, 1.0e6, 1.0, rt)
    assert np.abs(f64(out32) - want).max() <= 2e-3
    gk, gv = gather_rows(kp, vp, pt, n, False)
    assert_k_close(f64(gk[1:, p0:p0 + nt]), want, "rerotate")
    assert torch.equal(gk[0].view(torch.int16), k[0].view(torch.int16))           # layer 0 untouched
    assert torch.equal(gk[:, :p0].view(torch.int16), k[:, :p0].view(torch.int16))  # rows outside
    assert torch.equal(gk[:, p0 + nt:].view(torch.int16), k[:, p0 + nt:].view(torch.int16))
    assert torch.equal(gv.view(torch.int16), v.view(torch.int16))                  # V untouched


def test_rerotate_composition_matches_single_rotation():
    """R(a) then R(b) on the GPU against R(a + b) in the oracle (bf16 storage in between)."""
    L, H, n_pages, maxp, n = 1, 8, 8, 8, 64
    kp, vp = new_pools(L, n_pages, H, False, DEV)
    pt = np.arange(maxp, dtype=np.int32)
    k = randn_bf16((L, n, H, 128), 31, DEV)
    write_rows(kp, vp, pt, k, k, False)
    h_pt = pt[None].copy()
    d_pt = torch.as_tensor(h_pt, device=DEV)
    cache = nexus.kv_cache(kp, vp, n_pages, L, H)
    nexus.rope_rerotate(cache, d_pt, h_pt, 1, maxp, 0, 0, n, 1234, 0, 1)
    nexus.rope_rerotate(cache, d_pt, h_pt, 1, maxp, 0, 0, n, -1234, 0, 1)
    assert nexus.device_status() == nexus.OK
    gk, _ = gather_rows(kp, vp, pt, n, False)
    # Each bf16 store errs by at most half an ulp of a value no larger than the
    # pair's norm, and the second rotation keeps the first error's length: every
    # element ends within 2 * sqrt(2) half-ulps of its pair norm (+ float32 noise).
    k64 = f64(k)
    norm = np.sqrt(k64[..., :64] ** 2 + k64[..., 64:] ** 2)
    bound = 2.0 * np.sqrt(2.0) * np.exp2(np.floor(np.log2(np.maximum(1.01 * norm, 1e-30))) - 8) + 1e-5
    err = np.abs(f64(gk) - k64)
    assert np.all(err[..., :64] <= bound) and np.all(err[..., 64:] <= bound)


def test_page_copy_bit_exact():
    L, H, n_pages = 3, 8, 32
    for vt in (False, True):
        kp, vp = new_pools(L, n_pages, H, vt, DEV)
        kp.view(torch.int16).copy_(torch.randint(-32768, 32767, kp.shape, device=DEV, dtype=torch.int16))
        vp.view(torch.int16).copy_(torch.randint(-32768, 32767, vp.shape, device=DEV, dtype=torch.int16))
        k0, v0 = kp.clone(), vp.clone()
        cache = nexus.kv_cache(kp, vp, n_pages, L, H, vt)
        src, dst = [1, 5, 6, 30], [2, 0, 31, 7]
        nexus.copy_pages(cache, src, dst, 1, 3)
        assert nexus.device_status() == nexus.OK
        for s, d in zip(src, dst):
            assert torch.equal(kp[1:, d].view(torch.int16), k0[1:, s].view(torch.int16))
            assert torch.equal(vp[1:, d].view(torch.int16), v0[1:, s].view(torch.int16))
            assert torch.equal(kp[0, d].view(torch.int16), k0[0, d].view(torch.int16))
        untouched = [i for i in range(n_pages) if i not in dst]
        assert torch.equal(kp[:, untouched].view(torch.int16), k0[:, untouched].view(torch.int16))


def test_splice_repeat_runs_bit_stable():
    outs = []
    for _ in range(2):
        case = SplicedCase(workload("c1"), DEV)
        case.splice()
        assert nexus.device_status() == nexus.OK
        outs.append((case.kp.clone(), case.vp.clone()))
    assert torch.equal(outs[0][0].view(torch.int16), outs[1][0].view(torch.int16))
    assert torch.equal(outs[0][1].view(torch.int16), outs[1][1].view(torch.int16))


def test_splice_edge_shapes():
    """Empty blocks, inserts at depth 0 and at the cursor, unaligned depths and
    more than one page piece per segment, in one launch over three sessions."""
    from paper_2608_20397_gb300.workloads import Insert, Session, Workload
    w = Workload("edge", 2, [
        Session(37, [Insert(0, 5, 3), Insert(0, 0, 0), Insert(17, 33, 100), Insert(37, 16, 0)], 1, 100),
        Session(16, [Insert(16, 1, 16)], 1, 100),
        Session(250, [Insert(31, 47, 2), Insert(200, 19, 9)], 1, 100),
    ], v_transposed=False, seed=9)
    for vt in (False, True):
        w.v_transposed = vt
        case = SplicedCase(w, DEV)
        case.splice()
        assert nexus.device_status() == nexus.OK
        for si in range(3):
            _check_session(case, si, [0, 1])


def test_splice_bad_device_page_is_skipped_and_reported():
    # Without the host tables the kernel checks the page ids itself: a piece
    # whose destination or source page lies outside the pool is skipped whole
    # (nothing read or written through the bad id) and the call reports it.
    w = workload("c1")                     # 128-row block at depth 300 of 512 (tail 212)
    clean = SplicedCase(w, DEV)
    clean.splice()
    assert nexus.device_status() == nexus.OK
    want_k, want_v = clean.kp.clone(), clean.vp.clone()

    # destination: page index 20 of the new table (block rows 20..35, positions 320..335)
    case = SplicedCase(w, DEV)
    k0, v0 = case.kp.clone(), case.vp.clone()
    bad = case.h_pt.copy()
    real = int(bad[1, 20])
    bad[1, 20] = case.n_pages + 5
    case.d_pt = torch.as_tensor(bad, device=DEV)
    case.splice(validate=False)
    assert nexus.device_status() == nexus.ERANGE
    assert nexus.device_status() == nexus.OK                 # the record is cleared
    others = torch.ones(case.n_pages, dtype=torch.bool, device=DEV)
    others[real] = False
    for got, want, before in ((case.kp, want_k, k0), (case.vp, want_v, v0)):
        assert torch.equal(got[:, others].view(torch.int16), want[:, others].view(torch.int16))
        assert torch.equal(got[:, real].view(torch.int16), before[:, real].view(torch.int16))

    # source: page index 25 of the old table (displaced rows at positions 400..415)
    case = SplicedCase(w, DEV)
    k0, v0 = case.kp.clone(), case.vp.clone()
    bad = case.h_pt.copy()
    bad[0, 25] = -1
    case.d_pt = torch.as_tensor(bad, device=DEV)
    case.splice(validate=False)
    assert nexus.device_status() == nexus.ERANGE
    for got, want, before in ((case.kp, want_k, k0), (case.vp, want_v, v0)):
        g, a, b = (x.view(torch.int16) for x in (got, want, before))
        # every 16-byte-wide row slice is either the clean result or untouched
        same = (g == a).all(-1) | (g == b).all(-1)
        assert bool(same.all())
        assert not torch.equal(g, a)                       # and something was skipped
