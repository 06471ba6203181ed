"""The failure path of the bounded device waits on the GPU: a wait that runs out
(on a barrier nothing arrives on) is recorded, reported once by
nexus_device_status as NEXUS_ETIMEOUT, and leaves the context usable: the next
attention call matches the oracle."""
import numpy as np
import pytest
import torch

import oracle
from gpu_cases import assert_attn_close, f64, new_pools, write_rows
from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import randn_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return torch.device("cuda:0")


def test_bounded_wait_reports_timeout_once(dev):
    assert nexus.device_status() == nexus.OK
    nexus.selftest_wait(2000)                     # gives up after 2 ms
    assert nexus.device_status() == nexus.ETIMEOUT
    assert nexus.device_status() == nexus.OK      # the record is cleared
    nexus.selftest_wait(1)
    nexus.selftest_wait(500)
    assert nexus.device_status() == nexus.ETIMEOUT
    assert nexus.device_status() == nexus.OK


def test_context_usable_after_timeout(dev):
    nexus.selftest_wait(1000)
    assert nexus.device_status() == nexus.ETIMEOUT
    # a 300-key cache, the last 40 positions re-decoded, 10 / 2 heads
    T, R, H, Hq = 300, 40, 2, 10
    n_pages = T // 16 + 2
    kp, vp = new_pools(1, n_pages, H, False, dev)
    pt = np.random.default_rng(3).permutation(n_pages).astype(np.int32)[: -(-T // 16)]
    k = randn_bf16((1, T, H, 128), 11, dev)
    v = randn_bf16((1, T, H, 128), 12, dev)
    write_rows(kp, vp, pt, k, v, False)
    q = randn_bf16((1, R, Hq, 128), 13, dev)
    o = torch.empty_like(q)
    lse = torch.empty((1, R, Hq), dtype=torch.float32, device=dev)
    cache = nexus.kv_cache(kp, vp, n_pages, 1, H)
    d_pt = torch.as_tensor(pt.reshape(1, -1), device=dev)
    nexus.suffix_attention(cache, d_pt, 1, len(pt), [T], [R], q, o, lse, Hq, 0, 1, split_kv=1)
    assert nexus.device_status() == nexus.OK
    want_o, want_lse = oracle.attention(f64(q[0]), f64(k[0]), f64(v[0]),
                                        oracle.suffix_positions(T, R), Hq // H)
    assert_attn_close(f64(o[0]), want_o, lse[0].double().cpu().numpy(), want_lse, "after timeout")
