"""Parity of the INT8 tool scan and top-2 margin gate (Sec. IV-A) with the
oracle: top-2 indices, their float32 scores and the routing decision, all
exact (the integer dots are exact and both sides form the scores with the same
float32 operations).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import tool_queries, tool_registry

pytestmark = pytest.mark.gpu
TAU = 0.0136


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return torch.device("cuda:0")


def run(dev, tc, ts, qc, qs, tau=TAU, ws=None):
    nq = qc.shape[0]
    d = lambda a: torch.as_tensor(np.ascontiguousarray(a), device=dev)
    top_idx = torch.full((nq, 2), -7, dtype=torch.int32, device=dev)
    top_score = torch.full((nq, 2), float("nan"), dtype=torch.float32, device=dev)
    route = torch.full((nq,), -7, dtype=torch.int32, device=dev)
    if ws is None:
        ws = torch.zeros(nexus.slb_workspace_size(tc.shape[0]), dtype=torch.uint8, device=dev)
    nexus.slb_route(d(tc), d(ts), d(qc), d(qs), top_idx, top_score, route, ws, tau)
    torch.cuda.synchronize()
    return top_idx.cpu().numpy(), top_score.cpu().numpy(), route.cpu().numpy()


def check(got, tc, ts, qc, qs, tau=TAU):
    top_idx, top_score, route = got
    want = oracle.slb_route(qc, qs, tc, ts, np.float32(tau))
    for a, (i1, i2, s1, s2, r) in enumerate(want):
        assert (top_idx[a, 0], top_idx[a, 1]) == (i1, i2), a
        assert top_score[a, 0] == s1 and top_score[a, 1] == s2, a
        assert route[a] == r, a


def test_slb_paper_size(dev):
    # 250 tools x 768 dims; 33 queries: a full launch of 32 and one more
    x = tool_registry(250)
    q, _ = tool_queries(x, 33)
    tc, ts = oracle.slb_quantize(x)
    qc, qs = oracle.slb_quantize(q)
    got = run(dev, tc, ts, qc, qs)
    check(got, tc, ts, qc, qs)
    assert 0 < np.mean(got[2] == -1) < 1          # some queries escalate, some route


@pytest.mark.parametrize("nq", [1, 3, 8, 16, 32])
def test_slb_query_batches(dev, nq):
    x = tool_registry(1000, seed=4)
    q, _ = tool_queries(x, nq, seed=5)
    tc, ts = oracle.slb_quantize(x)
    qc, qs = oracle.slb_quantize(q)
    check(run(dev, tc, ts, qc, qs), tc, ts, qc, qs)


def test_slb_edge_cases(dev):
    r = np.random.default_rng(6)
    # a single tool: no runner-up, always routed
    tc = r.integers(-127, 128, (1, 64)).astype(np.int8)
    ts = np.array([0.01], np.float32)
    qc = r.integers(-127, 128, (3, 64)).astype(np.int8)
    qs = np.full(3, 0.02, np.float32)
    got = run(dev, tc, ts, qc, qs)
    check(got, tc, ts, qc, qs)
    assert list(got[0][:, 1]) == [-1] * 3 and list(got[2]) == [0] * 3
    # identical tools tie: the lower index ranks first and the zero margin escalates
    tc2 = np.repeat(tc, 5, axis=0)
    got = run(dev, tc2, np.full(5, 0.01, np.float32), qc, qs)
    check(got, tc2, np.full(5, 0.01, np.float32), qc, qs)
    assert list(got[0][:, 0]) == [0] * 3 and list(got[0][:, 1]) == [1] * 3
    assert list(got[2]) == [-1] * 3
    # dim 4, and a zero query (every score 0)
    tc3 = r.integers(-127, 128, (37, 4)).astype(np.int8)
    ts3 = r.random(37).astype(np.float32)
    qc3 = np.zeros((2, 4), np.int8)
    qc3[1] = [1, -2, 3, -4]
    qs3 = np.array([0.0, 0.5], np.float32)
    check(run(dev, tc3, ts3, qc3, qs3), tc3, ts3, qc3, qs3)


def test_slb_wide_rows(dev):
    # dim 4096 with 32 queries: 128 KiB of queries in shared memory
    x = tool_registry(300, dim=4096, seed=8)
    q, _ = tool_queries(x, 32, seed=9)
    tc, ts = oracle.slb_quantize(x)
    qc, qs = oracle.slb_quantize(q)
    check(run(dev, tc, ts, qc, qs), tc, ts, qc, qs)


def test_slb_large_registry_and_workspace_reuse(dev):
    # 100000 tools (77 MB of codes, several waves of CTAs); two calls on one workspace
    x = tool_registry(100_000, seed=10)
    q, _ = tool_queries(x, 40, seed=11)
    tc, ts = oracle.slb_quantize(x)
    qc, qs = oracle.slb_quantize(q)
    ws = torch.zeros(nexus.slb_workspace_size(tc.shape[0]), dtype=torch.uint8, device=dev)
    first = run(dev, tc, ts, qc, qs, ws=ws)
    check(first, tc, ts, qc, qs)
    second = run(dev, tc, ts, qc, qs, ws=ws)
    for a, b in zip(first, second):
        assert np.array_equal(a, b)
    assert not ws[:16].any()                        # the ticket is back at zero


def test_slb_bench_size_one_million_tools(dev):
    # The bench's large scan: 2^20 tools x 768 codes, one query and a batch of 32;
    # the oracle scores in chunks (exact integers times float32 scales) and the
    # top two are taken over all of them by the same ordering.
    r = np.random.default_rng(30)
    n = 1 << 20
    tc = r.integers(-127, 128, (n, 768), dtype=np.int8)
    ts = (r.random(n, dtype=np.float32) * np.float32(0.01)).astype(np.float32)
    qc = r.integers(-127, 128, (32, 768), dtype=np.int8)
    qs = (r.random(32, dtype=np.float32) * np.float32(0.01)).astype(np.float32)
    # plant near-ties: tool 5 copies tool 7 (equal scores when scales match)
    tc[5] = tc[7]
    ts[5] = ts[7]
    for nq in (1, 32):
        top_idx, top_score, route = run(dev, tc, ts, qc[:nq], qs[:nq])
        scores = np.concatenate([oracle.slb_scores(qc[:nq], qs[:nq], tc[i:i + 65536], ts[i:i + 65536])
                                 for i in range(0, n, 65536)], axis=1)
        for a in range(nq):
            order = np.lexsort((np.arange(n), -scores[a].astype(np.float64)))[:2]   # score, then index
            (i1, s1), (i2, s2) = [(int(j), scores[a, j]) for j in order]
            assert (top_idx[a, 0], top_idx[a, 1]) == (i1, i2), (nq, a)
            assert top_score[a, 0] == s1 and top_score[a, 1] == s2
            assert route[a] == (i1 if np.float32(s1 - s2) > np.float32(TAU) else -1)


@pytest.mark.parametrize("dim,n_tools", [(768, 16384 + 37), (4096, 16384 + 5), (64, 20000 + 3),
                                         (4, 16384), (72, 40001), (768, 100_003)])
@pytest.mark.parametrize("nq", [1, 2, 4])
def test_slb_streamed_registry(dev, dim, n_tools, nq):
    # Registries of 16384 tools and more with up to four queries stream through
    # shared memory by bulk copies; each CTA's last stage may be partial and is
    # read from global memory. Exact parity with the oracle.
    r = np.random.default_rng(dim * 7 + n_tools + nq)
    tc = r.integers(-127, 128, (n_tools, dim), dtype=np.int8)
    ts = (r.random(n_tools, dtype=np.float32) * np.float32(0.01)).astype(np.float32)
    qc = r.integers(-127, 128, (nq, dim), dtype=np.int8)
    qs = (r.random(nq, dtype=np.float32) * np.float32(0.01)).astype(np.float32)
    tc[n_tools - 1] = tc[3]            # a tie between the first and the last stage
    ts[n_tools - 1] = ts[3]
    got = run(dev, tc, ts, qc, qs)
    assert nexus.device_status() == nexus.OK
    check(got, tc, ts, qc, qs)


def test_slb_streamed_workspace_reuse(dev):
    x = tool_registry(50_000, seed=12)
    q, _ = tool_queries(x, 3, seed=13)
    tc, ts = oracle.slb_quantize(x)
    qc, qs = oracle.slb_quantize(q)
    ws = torch.zeros(nexus.slb_workspace_size(tc.shape[0]), dtype=torch.uint8, device=dev)
    first = run(dev, tc, ts, qc, qs, ws=ws)
    check(first, tc, ts, qc, qs)
    second = run(dev, tc, ts, qc, qs, ws=ws)
    for a, b in zip(first, second):
        assert np.array_equal(a, b)
    assert not ws[:16].any()


@pytest.mark.parametrize("dim,n_tools,nq", [(768, 16384 + 37, 5), (64, 20000 + 3, 32),
                                            (1024, 16384, 17), (512, 100_003, 8),
                                            (1088, 16384, 8)])
def test_slb_tensor_core_batches(dev, dim, n_tools, nq):
    # Batches of 5..32 queries over 16384 tools and more, dim a multiple of 64 up
    # to 1024, are scanned by bf16 products on the tensor cores: exact integer dots
    # (|partial sums| <= 1024 * 128^2 = 2^24), so exact parity. Rows of 127 and
    # -128 reach that bound (tool 12 with query 1: 2^24 at dim 1024); a three-way
    # tie, a zero scale and a partial last tile of 128 tools are planted. dim
    # 1088 is past the bound and keeps the dp4a scan.
    r = np.random.default_rng(dim + n_tools + nq)
    tc = r.integers(-127, 128, (n_tools, dim), dtype=np.int8)
    ts = (r.random(n_tools, dtype=np.float32) * np.float32(0.01)).astype(np.float32)
    qc = r.integers(-127, 128, (nq, dim), dtype=np.int8)
    qs = (r.random(nq, dtype=np.float32) * np.float32(0.01)).astype(np.float32)
    tc[11], tc[12] = 127, -128
    qc[0], qc[1] = 127, -128
    ts[13] = 0.0
    tc[2] = tc[3]
    tc[n_tools - 1] = tc[3]
    ts[2] = ts[n_tools - 1] = ts[3]
    got = run(dev, tc, ts, qc, qs)
    assert nexus.device_status() == nexus.OK
    check(got, tc, ts, qc, qs)
