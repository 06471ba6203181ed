"""The L0 warm arena (Sec. V-D) on the GPU: requests forked from warm slots get
their prefix rows through shared pages plus one copied boundary page
(nexus_copy_pages), bit for bit; slots keep their rows while requests write
their own; attention over a warm-started sequence equals attention over the
same sequence written cold, bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_20397_gb300 import nexus
from test_warm_arena import agent_stream, prefix_rows

pytestmark = pytest.mark.gpu
PAGE = 16
L, H, D = 3, 8, 128


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return torch.device("cuda:0")


def kv_rows(hashes, dev):
    """[L][n][H][D] bf16 K and V rows, a fixed function of each position's hash."""
    h = torch.as_tensor(np.asarray(hashes) % 100003, dtype=torch.float32, device=dev)
    idx = torch.arange(L * H * D, dtype=torch.float32, device=dev)
    base = torch.remainder(h[:, None] * 0.0137 + idx[None, :] * 0.371, 8.0) - 4.0
    k = base.reshape(-1, L, H, D).permute(1, 0, 2, 3).to(torch.bfloat16)
    v = (-0.5 * base).reshape(-1, L, H, D).permute(1, 0, 2, 3).to(torch.bfloat16)
    return k.contiguous(), v.contiguous()


def write(kp, vp, pt, pos0, k, v):
    n = k.shape[1]
    if n == 0:
        return
    dev = kp.device
    pos = torch.arange(pos0, pos0 + n, device=dev)
    pg = torch.as_tensor(pt, device=dev).long()[pos // PAGE]
    kp[:, pg, :, pos % PAGE, :] = k.permute(1, 0, 2, 3)
    vp[:, pg, :, pos % PAGE, :] = v.permute(1, 0, 2, 3)


def read(kp, vp, pt, n):
    dev = kp.device
    pos = torch.arange(n, device=dev)
    pg = torch.as_tensor(pt, device=dev).long()[pos // PAGE]
    return (kp[:, pg, :, pos % PAGE, :].permute(1, 0, 2, 3),
            vp[:, pg, :, pos % PAGE, :].permute(1, 0, 2, 3))


def same_bits(a, b):
    return torch.equal(a.contiguous().view(torch.int16), b.contiguous().view(torch.int16))


def test_warm_forks_on_device(dev):
    n_pages = 1024
    kp = torch.full((L, n_pages, H, PAGE, D), float("nan"), dtype=torch.bfloat16, device=dev)
    vp = torch.full_like(kp, float("nan"))
    cache = nexus.kv_cache(kp, vp, n_pages, L, H)
    pool = nexus.PagePool(n_pages)
    arena = nexus.WarmArena(4, 2048)
    model = oracle.WarmArenaModel(4, 2048)
    copies = 0
    for q in agent_stream(7, 60):
        n = len(q)
        slot, m = arena.match(q)
        assert (slot, m) == model.match(q)
        max_pages = -(-n // PAGE)
        pt_pre = np.zeros(0, np.int32)
        if slot >= 0:
            pt_pre, src, dst = arena.fork(pool, slot, m, max_pages)
            model.fork(slot, m)
            if len(src):
                nexus.copy_pages(cache, src, dst, 0, L)
                copies += 1
        pt = np.concatenate([pt_pre, pool.alloc(max_pages - len(pt_pre))]).astype(np.int32)
        k, v = kv_rows(prefix_rows(q), dev)
        if m:
            gk, gv = read(kp, vp, pt, m)     # the warm rows, before the request writes its own
            assert same_bits(gk, k[:, :m]) and same_bits(gv, v[:, :m])
        write(kp, vp, pt, m, k[:, m:], v[:, m:])
        arena.store(pool, q, pt)
        model.store(q, np.zeros((1, n, 1, 1)), np.zeros((1, n, 1, 1)))
        pool.free(pt)
    torch.cuda.synchronize()
    assert copies > 0
    for s in range(4):
        ln, pages = arena.slot(s)
        if ln:
            k, v = kv_rows(prefix_rows(model.tokens[s]), dev)
            gk, gv = read(kp, vp, pages, ln)
            assert same_bits(gk, k) and same_bits(gv, v)
    arena.close(pool)
    assert pool.available() == n_pages


def test_warm_start_attention_equals_cold(dev):
    """A request of 700 tokens whose first 457 are warm: suffix attention of its
    last 64 queries over the warm-started cache is bit-identical to the same
    attention over the sequence written from scratch."""
    n_pages = 256
    kp = torch.zeros((L, n_pages, H, PAGE, D), dtype=torch.bfloat16, device=dev)
    vp = torch.zeros_like(kp)
    cache = nexus.kv_cache(kp, vp, n_pages, L, H)
    pool = nexus.PagePool(n_pages, np.random.default_rng(5).permutation(n_pages))
    arena = nexus.WarmArena(32, 4096)
    r = np.random.default_rng(9)
    warm = [int(t) for t in r.integers(0, 100, 500)]
    q_toks = warm[:457] + [int(t) for t in r.integers(100, 200, 243)]
    pt_w = pool.alloc(-(-500 // PAGE))
    k, v = kv_rows(prefix_rows(warm), dev)
    write(kp, vp, pt_w, 0, k, v)
    arena.store(pool, warm, pt_w)
    slot, m = arena.match(q_toks)
    assert (slot, m) == (0, 457)
    n = len(q_toks)
    pre, src, dst = arena.fork(pool, slot, m, -(-n // PAGE))
    nexus.copy_pages(cache, src, dst, 0, L)
    pt_warm = np.concatenate([pre, pool.alloc(-(-n // PAGE) - len(pre))]).astype(np.int32)
    kq, vq = kv_rows(prefix_rows(q_toks), dev)
    write(kp, vp, pt_warm, m, kq[:, m:], vq[:, m:])
    pt_cold = pool.alloc(-(-n // PAGE))
    write(kp, vp, pt_cold, 0, kq, vq)
    mp = -(-n // PAGE)
    d_pt = torch.as_tensor(np.stack([pt_warm, pt_cold]), device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(3)
    qx = torch.randn((L, 64, 40, D), generator=g, device=dev).to(torch.bfloat16)
    outs = []
    for row in (0, 1):
        o = torch.empty_like(qx)
        lse = torch.empty(qx.shape[:3], dtype=torch.float32, device=dev)
        nexus.suffix_attention(cache, d_pt, 2, mp, [n], [64], qx, o, lse, 40, 0, L, rows=[row],
                               split_kv=1)
        outs.append((o, lse))
    assert nexus.device_status() == nexus.OK
    assert same_bits(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1])
    assert torch.isfinite(outs[0][0].float()).all()


def test_warm_forks_at_bench_shape(dev):
    """The bench's arena shape: 48 layers x 8 KV heads, 32 slots holding a shared
    8192-token prompt and a 1024-token tail each; forks of 8192 + k tokens get
    rows bit-identical to the slot's, through one copied boundary page."""
    Lb, H = 48, 8
    n_pages = 512 + 32 * 64 + 64
    kp = torch.zeros((Lb, n_pages, H, PAGE, D), dtype=torch.bfloat16, device=dev)
    vp = torch.zeros_like(kp)
    cache = nexus.kv_cache(kp, vp, n_pages, Lb, H)
    pool = nexus.PagePool(n_pages)
    arena = nexus.WarmArena(32, 8192 + 1024)
    r = np.random.default_rng(77)
    system = [int(t) for t in r.integers(0, 32000, 8192)]
    sys_pt = pool.alloc(512)
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    kp[:, torch.as_tensor(sys_pt, device=dev).long()] = torch.randn(
        (Lb, 512, H, PAGE, D), generator=g, device=dev).to(torch.bfloat16)
    tails = []
    for s in range(32):
        tail = [int(t) for t in r.integers(0, 32000, 1024)]
        tails.append(tail)
        own = pool.alloc(64)
        kp[:, torch.as_tensor(own, device=dev).long()] = torch.randn(
            (Lb, 64, H, PAGE, D), generator=g, device=dev).to(torch.bfloat16)
        vp[:, torch.as_tensor(own, device=dev).long()] = -kp[:, torch.as_tensor(own, device=dev).long()]
        pt = np.concatenate([sys_pt, own]).astype(np.int32)
        pool.retain(sys_pt)
        arena.store(pool, system + tail, pt)
        pool.free(pt)
    pool.free(sys_pt)
    for j, k in ((0, 1), (7, 500), (31, 1023), (12, 16)):
        q = system + tails[j][:k] + [40000 + i for i in range(64)]
        slot, m = arena.match(q)
        assert m == 8192 + k
        pre, src, dst = arena.fork(pool, slot, m, -(-len(q) // PAGE))
        nexus.copy_pages(cache, src, dst, 0, Lb)
        torch.cuda.synchronize()
        _, spages = arena.slot(slot)
        gk, gv = read(kp, vp, pre, m)
        wk, wv = read(kp, vp, spages, m)
        assert same_bits(gk, wk) and same_bits(gv, wv)
        pool.free(pre)
    arena.close(pool)
    assert pool.available() == n_pages
