"""The no-allocation attention entry point against the regular one and the oracle.

nexus_suffix_attention_noalloc serves callers that cannot allocate device
memory (code running while a stream is captured, plug-ins handed only their
buffers, processes with a fixed memory pool): its split-KV partials live in the
library's own array. With the same split count it runs the same kernels in the
same order as nexus_suffix_attention with a workspace, so the two must agree bit
for bit, also after another call has left different data in the shared array.
This file is collected last so that a run stopping at the first failure has
already run every other test; it passes on its own in a fresh process as well.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_attn_close, f64, new_pools, write_rows
from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import randn_bf16

pytestmark = pytest.mark.gpu
DEV = torch.device("cuda:0") if torch.cuda.is_available() else None


def _case(kv, ql, L=2, seed=41):
    H, Hq = 8, 40
    max_pages = max(-(-k // 16) for k in kv) + 1
    n_pages = sum(-(-k // 16) for k in kv) + 4
    kp, vp = new_pools(L, n_pages, H, False, DEV)
    order = np.random.default_rng(seed).permutation(n_pages)
    h_pt = np.full((len(kv), max_pages), -1, np.int32)
    rows = []
    cur = 0
    for i, T in enumerate(kv):
        npg = -(-T // 16)
        h_pt[i, :npg] = order[cur:cur + npg]
        cur += npg
        k = randn_bf16((L, T, H, 128), seed + 2 * i, DEV)
        v = randn_bf16((L, T, H, 128), seed + 2 * i + 1, DEV)
        write_rows(kp, vp, h_pt[i], k, v, False)
        rows.append((k, v))
    cache = nexus.kv_cache(kp, vp, n_pages, L, H)
    q = randn_bf16((L, sum(ql), Hq, 128), seed + 99, DEV)
    return cache, torch.as_tensor(h_pt, device=DEV), max_pages, q, rows


def _noalloc(cache, d_pt, kv, ql, q, mp, L):
    o = torch.full_like(q, float("nan"))
    l = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=DEV)
    nexus.suffix_attention_noalloc(cache, d_pt, len(kv), mp, kv, ql, q, o, l, 40, 0, L, split_kv=0)
    assert nexus.device_status() == nexus.OK
    return o, l


def test_noalloc_matches_workspace_entry_point_twice():
    kv, ql, L = [5000, 2100], [64, 17], 2
    cache, d_pt, mp, q, rows = _case(kv, ql, L)
    need, splits = nexus.attention_workspace_size(kv, ql, 40, 8, L, 0)
    assert splits > 1 and 0 < need <= 32 << 20
    ws = torch.empty(need, dtype=torch.uint8, device=DEV)
    ref_o = torch.empty_like(q)
    ref_l = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
    nexus.suffix_attention(cache, d_pt, 2, mp, kv, ql, q, ref_o, ref_l, 40, 0, L, split_kv=0,
                           workspace=ws, workspace_bytes=need)
    assert nexus.device_status() == nexus.OK

    o, l = _noalloc(cache, d_pt, kv, ql, q, mp, L)
    assert torch.equal(o, ref_o) and torch.equal(l, ref_l)

    # another shape in between leaves different partials in the shared array
    kv2, ql2 = [3000], [40]
    c2, d2, mp2, q2, _ = _case(kv2, ql2, 1, seed=77)
    _noalloc(c2, d2, kv2, ql2, q2, mp2, 1)

    o, l = _noalloc(cache, d_pt, kv, ql, q, mp, L)
    assert torch.equal(o, ref_o) and torch.equal(l, ref_l)

    # and against the oracle: every row of both sequences of layer 1
    off = 0
    for si, (T, R) in enumerate(zip(kv, ql)):
        k, v = rows[si]
        want, want_l = oracle.attention(f64(q[1, off:off + R]), f64(k[1]), f64(v[1]),
                                        oracle.suffix_positions(T, R), 5)
        assert_attn_close(f64(o[1, off:off + R]), want, f64(l[1, off:off + R]), want_l,
                          f"no-alloc sequence {si}")
        off += R


def test_noalloc_rejects_requests_beyond_its_array():
    kv, ql = [40000], [2000]
    cache, d_pt, mp, q, _ = _case(kv, ql, 1)
    o = torch.empty_like(q)
    with pytest.raises(nexus.NexusError) as e:
        nexus.suffix_attention_noalloc(cache, d_pt, 1, mp, kv, ql, q, o, None, 40, 0, 1, split_kv=32)
    assert e.value.code == nexus.ENOMEM
    # argument errors are reported as the workspace entry point reports them
    with pytest.raises(nexus.NexusError) as e:
        nexus.suffix_attention_noalloc(cache, d_pt, 1, mp, kv, ql, q, o, None, 40, 1, 0, split_kv=32)
    assert e.value.code == nexus.ERANGE
