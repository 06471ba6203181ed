"""The L0 exact-token radix arena (Sec. V-D) on the CPU: the library's decisions
against the oracle model on random agent-like request streams, with a host
page store standing in for the cache (the page copies the library asks for are
applied to it), reference counts, copy-on-write, and argument checks.

A row's content is a hash of the token prefix that ends at it, as a model's KV
row depends on the tokens up to its position; equal tokens give equal rows.
"""
import os

import numpy as np
import pytest

import oracle
from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import agent_requests

PAGE = 16


@pytest.fixture(scope="module", autouse=True)
def built_library():
    if not os.path.exists(nexus.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    nexus.lib()


def prefix_rows(tokens):
    """One float per position: a hash of tokens[0 .. pos]."""
    h, out = 1469598103, []
    for t in tokens:
        h = (h * 1099511 + int(t) + 7) % 2147483629
        out.append(float(h))
    return np.asarray(out, dtype=np.float64)


class PageStore:
    """Host stand-in for the paged cache: page id -> 16 rows."""

    def __init__(self, n_pages):
        self.rows = np.full((n_pages, PAGE), np.nan)

    def copy(self, src, dst):
        for s, d in zip(src, dst):
            self.rows[d] = self.rows[s]

    def write(self, pt, pos0, values):
        for i, v in enumerate(values):
            p = pos0 + i
            self.rows[pt[p // PAGE], p % PAGE] = v

    def read(self, pt, n):
        return np.asarray([self.rows[pt[p // PAGE], p % PAGE] for p in range(n)])


def agent_stream(seed, n_requests):
    return agent_requests(seed, n_requests)


def run_stream(n_slots, max_tokens, seed, n_requests, n_pages=4096):
    pool = nexus.PagePool(n_pages)
    arena = nexus.WarmArena(n_slots, max_tokens)
    model = oracle.WarmArenaModel(n_slots, max_tokens)
    store = PageStore(n_pages)
    hits = 0
    for q in agent_stream(seed, n_requests):
        n = len(q)
        want = model.match(q)
        got = arena.match(q)
        assert got == want, (got, want)
        slot, m = got
        max_pages = -(-n // PAGE)
        if slot >= 0:
            hits += 1
            pt_pre, src, dst = arena.fork(pool, slot, m, max_pages)
            store.copy(src, dst)
            k_want, _ = model.fork(slot, m)
            assert len(src) == (1 if m % PAGE else 0)
            assert np.array_equal(store.read(pt_pre, m), k_want[0, :, 0, 0])
        else:
            pt_pre = np.zeros(0, np.int32)
        rest = pool.alloc(max_pages - len(pt_pre))
        pt = np.concatenate([pt_pre, rest]).astype(np.int32)
        rows = prefix_rows(q)
        store.write(pt, m, rows[m:])                      # the request's own prefill
        assert np.array_equal(store.read(pt, n), rows)
        s_got = arena.store(pool, q, pt)
        kv = rows.reshape(1, -1, 1, 1)
        assert s_got == model.store(q, kv, kv)
        pool.free(pt)                                     # the request ends
        # every slot still reads its own rows through its pages
        held = {}
        for s in range(n_slots):
            ln, pages = arena.slot(s)
            toks = model.tokens[s]
            assert ln == (0 if toks is None else len(toks))
            if ln:
                assert np.array_equal(store.read(pages, ln), prefix_rows(toks))
                for pg in pages:
                    held[int(pg)] = held.get(int(pg), 0) + 1
        for pg in range(n_pages):
            assert pool.refs(pg) == held.get(pg, 0)
        assert pool.available() == n_pages - len(held)
    arena.close(pool)
    assert pool.available() == n_pages
    return hits


@pytest.mark.parametrize("n_slots,max_tokens,seed", [(32, 4096, 1), (3, 4096, 2), (5, 200, 3),
                                                     (1, 1000, 4)])
def test_arena_matches_oracle_on_agent_streams(n_slots, max_tokens, seed):
    hits = run_stream(n_slots, max_tokens, seed, 120)
    assert hits > 0


def test_fork_shares_full_pages_and_copies_the_boundary():
    pool = nexus.PagePool(64)
    arena = nexus.WarmArena(4, 512)
    toks = list(range(100))
    pt = pool.alloc(7)
    arena.store(pool, toks, pt)
    for m, n_copy in ((0, 0), (16, 0), (48, 0), (35, 1), (100, 1), (1, 1)):
        new_pt, src, dst = arena.fork(pool, 0, m, 8)
        assert len(new_pt) == -(-m // 16) and len(src) == n_copy
        full = m // 16
        assert np.array_equal(new_pt[:full], pt[:full])
        if n_copy:
            assert src[0] == pt[full] and dst[0] == new_pt[full] and dst[0] not in pt
        pool.free(new_pt)
    assert all(pool.refs(int(p)) == 2 for p in pt)   # the table and the slot
    pool.free(pt)
    assert all(pool.refs(int(p)) == 1 for p in pt)   # the slot alone
    arena.close(pool)
    assert pool.available() == 64


def test_make_private_before_in_place_writes():
    pool = nexus.PagePool(32)
    store = PageStore(32)
    arena = nexus.WarmArena(2, 256)
    toks = list(range(64))
    pt = pool.alloc(4)
    store.write(pt, 0, prefix_rows(toks))
    arena.store(pool, toks, pt)
    new_pt, _, _ = arena.fork(pool, 0, 64, 4)      # all four pages shared
    new_pt = new_pt.astype(np.int32)
    src, dst = pool.make_private(new_pt, 1, 2)    # rows 16..47 are about to change
    assert len(src) == 2 and np.array_equal(src, pt[1:3]) and np.array_equal(dst, new_pt[1:3])
    store.copy(src, dst)
    store.write(new_pt, 20, [-1.0] * 10)
    assert np.array_equal(store.read(pt, 64), prefix_rows(toks))   # the slot is untouched
    src2, _ = pool.make_private(new_pt, 1, 2)     # already private: nothing to copy
    assert len(src2) == 0
    assert pool.refs(int(pt[1])) == 2 and pool.refs(int(new_pt[1])) == 1


def test_pool_reference_counts():
    pool = nexus.PagePool(8)
    a = pool.alloc(3)
    pool.retain(a[:2])
    assert [pool.refs(int(p)) for p in a] == [2, 2, 1]
    pool.free(a)
    assert [pool.refs(int(p)) for p in a] == [1, 1, 0] and pool.available() == 6
    with pytest.raises(nexus.NexusError) as e:
        pool.free([a[0], a[0]])                     # listed twice
    assert e.value.code == nexus.EINVAL
    with pytest.raises(nexus.NexusError) as e:
        pool.retain([a[2]])                         # free page
    assert e.value.code == nexus.EINVAL
    with pytest.raises(nexus.NexusError) as e:
        pool.retain([99])
    assert e.value.code == nexus.ERANGE
    assert pool.refs(99) == -1
    pool.free(a[:2])
    assert pool.available() == 8
    # freed pages return to the back of the order
    assert list(pool.alloc(8)) == [3, 4, 5, 6, 7, 2, 0, 1]


def test_arena_argument_checks():
    pool = nexus.PagePool(16)
    arena = nexus.WarmArena(2, 64)
    with pytest.raises(nexus.NexusError):
        nexus.WarmArena(33, 64)
    with pytest.raises(nexus.NexusError) as e:
        arena.fork(pool, 0, 1, 4)                   # empty slot
    assert e.value.code == nexus.ERANGE
    pt = pool.alloc(2)
    arena.store(pool, list(range(20)), pt)
    with pytest.raises(nexus.NexusError) as e:
        arena.fork(pool, 0, 21, 4)                  # past the slot's length
    assert e.value.code == nexus.ERANGE
    with pytest.raises(nexus.NexusError) as e:
        arena.fork(pool, 0, 20, 1)                  # page table too short
    assert e.value.code == nexus.ERANGE
    with pytest.raises(nexus.NexusError) as e:
        arena.store(pool, list(range(50, 70)), [14, 15])   # pages not in use
    assert e.value.code == nexus.EINVAL
    assert arena.match([50]) == (-1, 0)
    rest = pool.alloc(pool.available())
    with pytest.raises(nexus.NexusError) as e:
        arena.fork(pool, 0, 17, 4)                  # no page for the boundary copy
    assert e.value.code == nexus.ENOMEM
    assert pool.refs(int(pt[0])) == 2               # nothing changed
    pool.free(rest)
    assert arena.match(list(range(20)) + [1]) == (0, 20)
    assert arena.match([]) == (-1, 0)
