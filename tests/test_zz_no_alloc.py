"""The no-allocation attention entry point against the regular one.

nexus_suffix_attention_noalloc serves callers that cannot allocate device
memory (stream capture, plug-ins given only their buffers, fixed pools): its
split-KV partials live in the library's own array. This file is collected last
so that a run stopping at the first failure has already run every other test;
it passes on its own in a fresh process as well.
"""
import numpy as np
import pytest
import torch

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
    cur = 0
    for i, T in enumerate(kv):
        npg = -(-T // 16)
        h_pt[i, :npg] = order[cur:cur + npg]
        cur += npg
        write_rows(kp, vp, h_pt[i], randn_bf16((L, T, H, 128), seed + 2 * i, DEV),
                   randn_bf16((L, T, H, 128), seed + 2 * i + 1, DEV), False)
    cache = nexus.kv_cache(kp, vp, n_pages, L, H)
    q = randn_bf16((L, sum(ql), Hq, 128), seed + 99, DEV)
    return cache, torch.as_tensor(h_pt, device=DEV), max_pages, q


def test_noalloc_matches_workspace_entry_point_twice():
    kv, ql, L = [5000, 2100], [64, 17], 2
    cache, d_pt, mp, q = _case(kv, ql, L)
    need, splits = nexus.attention_workspace_size(kv, ql, 40, 8, L, 0)
    assert splits > 1 and 0 < need <= 32 << 20
    ws = torch.empty(need, dtype=torch.uint8, device=DEV)
    ref_o = torch.empty_like(q)
    ref_l = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
    nexus.suffix_attention(cache, d_pt, 2, mp, kv, ql, q, ref_o, ref_l, 40, 0, L, split_kv=0,
                           workspace=ws, workspace_bytes=need)
    assert nexus.device_status() == nexus.OK
    for _ in range(2):   # two calls in a row share the library's scratch array
        o = torch.full_like(q, float("nan"))
        l = torch.full(q.shape[:3], float("nan"), dtype=torch.float32, device=DEV)
        nexus.suffix_attention_noalloc(cache, d_pt, 2, mp, kv, ql, q, o, l, 40, 0, L, split_kv=0)
        assert nexus.device_status() == nexus.OK
        for layer in range(L):
            assert_attn_close(f64(o[layer]), f64(ref_o[layer]), f64(l[layer]), f64(ref_l[layer]),
                              f"no-alloc layer {layer}")


def test_noalloc_rejects_requests_beyond_its_array():
    kv, ql = [40000], [2000]
    cache, d_pt, mp, q = _case(kv, ql, 1)
    o = torch.empty_like(q)
    with pytest.raises(nexus.NexusError) as e:
        nexus.suffix_attention_noalloc(cache, d_pt, 1, mp, kv, ql, q, o, None, 40, 0, 1, split_kv=32)
    assert e.value.code == nexus.ENOMEM
