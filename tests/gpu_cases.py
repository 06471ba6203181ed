"""Test-side plumbing for the GPU parity tests: paged pools filled by torch
indexing, oracle-side conversions and the tolerance checks of the path.

Tolerances (written here once, used by every GPU test):
* splice V and every delta = 0 K row: bit-exact;
* re-rotated K (bf16 store): |K - K_oracle| <= 2e-3 + half a bf16 ulp of
  |K_oracle| (the bf16 store alone errs by up to half an ulp, 3.9e-3 at
  |k| in [1, 2)); the float32 output of the same arithmetic: <= 2e-3;
* attention output: |O - O_oracle| <= 1e-2 wherever the bf16 output can hold a
  value that close (|O_oracle| < 4, where half a bf16 ulp is at most 7.8e-3);
  from |O_oracle| >= 4 on, half an ulp alone is 1.6e-2 or more, so there the
  bound is 1e-2 plus half a bf16 ulp of |O_oracle|; relative L2 <= 5e-3; LSE
  max abs <= 1e-2.
"""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_20397_gb300 import nexus
from paper_2608_20397_gb300.workloads import randn_bf16

ATTN_ABS = 1e-2
ATTN_REL = 5e-3
K_ABS = 2e-3


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().double().numpy()


def half_ulp_bf16(x: np.ndarray) -> np.ndarray:
    ax = np.maximum(np.abs(x), 2.0 ** -126)
    return np.exp2(np.floor(np.log2(ax)) - 8)


def assert_k_close(got: np.ndarray, want: np.ndarray, what=""):
    err = np.abs(got - want)
    bound = K_ABS + half_ulp_bf16(want)
    bad = err > bound
    assert not bad.any(), f"{what}: {bad.sum()} K elements out of tolerance, worst {err.max():.3e}"


def attn_abs_bound(want: np.ndarray) -> np.ndarray:
    """1e-2, widened by half a bf16 ulp only where that half ulp is itself 1.6e-2 or more."""
    return np.where(np.abs(want) < 4.0, ATTN_ABS, ATTN_ABS + half_ulp_bf16(want))


def assert_attn_close(got: np.ndarray, want: np.ndarray, got_lse=None, want_lse=None, what=""):
    err = np.abs(got - want)
    rel = np.linalg.norm(got - want) / max(np.linalg.norm(want), 1e-30)
    bad = err > attn_abs_bound(want)
    assert not bad.any(), f"{what}: {bad.sum()} outputs out of tolerance, max abs {err.max():.3e}"
    assert rel <= ATTN_REL, f"{what}: rel L2 {rel:.3e}"
    if got_lse is not None:
        e = np.abs(got_lse - want_lse)
        assert e.max() <= 1e-2, f"{what}: lse max abs {e.max():.3e}"


def new_pools(n_layers, n_pages, H, vt, dev, fill=0.0):
    k = torch.full((n_layers, n_pages, H, 16, 128), fill, dtype=torch.bfloat16, device=dev)
    if vt:
        v = torch.full((n_layers, n_pages, H, 128, 16), fill, dtype=torch.bfloat16, device=dev)
    else:
        v = torch.full((n_layers, n_pages, H, 16, 128), fill, dtype=torch.bfloat16, device=dev)
    return k, v


def write_rows(kp, vp, pt, k_rows, v_rows, vt, pos0=0):
    """Logical rows [L][n][H][d] -> pool positions pos0 .. pos0 + n - 1 of a page table."""
    n = k_rows.shape[1]
    if n == 0:
        return
    dev = kp.device
    pos = torch.arange(pos0, pos0 + n, device=dev)
    pg = torch.as_tensor(np.asarray(pt), device=dev)[pos // 16].long()
    sl = pos % 16
    kp[:, pg, :, sl, :] = k_rows.permute(1, 0, 2, 3)
    if vt:
        vp[:, pg, :, :, sl] = v_rows.permute(1, 0, 2, 3)
    else:
        vp[:, pg, :, sl, :] = v_rows.permute(1, 0, 2, 3)


def gather_rows(kp, vp, pt, n, vt, layers=None):
    dev = kp.device
    pos = torch.arange(n, device=dev)
    pg = torch.as_tensor(np.asarray(pt), device=dev)[pos // 16].long()
    sl = pos % 16
    ks = kp if layers is None else kp[layers]
    vs = vp if layers is None else vp[layers]
    k = ks[:, pg, :, sl, :].permute(1, 0, 2, 3)
    v = (vs[:, pg, :, :, sl] if vt else vs[:, pg, :, sl, :]).permute(1, 0, 2, 3)
    return k, v


class SplicedCase:
    """A workload's sessions written into a paged pool, planned and spliced
    through the C ABI. Rows 2s / 2s+1 of the page-table array are session s's
    pre- and post-splice tables."""

    def __init__(self, w, dev, layers=None, spare_pages=64, garbage_fill=None, keep_live=True):
        from paper_2608_20397_gb300.workloads import page_order
        self.w = w
        self.dev = dev
        L = w.n_layers if layers is None else layers
        self.L = L
        H = w.n_kv_heads
        self.vt = w.v_transposed
        pages_needed = 0
        for s in w.sessions:
            pages_needed += -(-s.n_past // 16) + -(-w.spliced_len(s) // 16) + 1
        self.n_pages = pages_needed + spare_pages
        self.max_pages = max(-(-w.spliced_len(s) // 16) for s in w.sessions) + 1
        fill = 0.0 if garbage_fill is None else garbage_fill
        self.kp, self.vp = new_pools(L, self.n_pages, H, self.vt, dev, fill)
        self.pool = nexus.PagePool(self.n_pages, page_order(self.n_pages, w.seed, w.shuffle_pages))
        self.cache = nexus.kv_cache(self.kp, self.vp, self.n_pages, L, H, self.vt,
                                    rope_theta=w.rope_theta)
        n_rows = 2 * len(w.sessions)
        self.h_pt = np.full((n_rows, self.max_pages), -1, np.int32)
        self.live_k, self.live_v, self.blk_k, self.blk_v, self.blocks = [], [], [], [], []
        seed = w.seed * 100
        for si, s in enumerate(w.sessions):
            npg = -(-s.n_past // 16)
            self.h_pt[2 * si, :npg] = self.pool.alloc(npg)
            lk = randn_bf16((L, s.n_past, H, 128), seed + 1, dev)
            lv = randn_bf16((L, s.n_past, H, 128), seed + 2, dev)
            write_rows(self.kp, self.vp, self.h_pt[2 * si], lk, lv, self.vt)
            # large cases regenerate the live rows from their seeds when checked
            self.live_k.append(lk if keep_live else (L, s.n_past, H, seed + 1))
            self.live_v.append(lv if keep_live else (L, s.n_past, H, seed + 2))
            del lk, lv
            bks, bvs = [], []
            for j, ins in enumerate(s.inserts):
                bk = randn_bf16((L, ins.length, H, 128), seed + 10 + 2 * j, dev)
                bv = randn_bf16((L, ins.length, H, 128), seed + 11 + 2 * j, dev)
                bks.append(bk)
                bvs.append(bv)
            self.blk_k.append(bks)
            self.blk_v.append(bvs)
            seed += 1000
        self.segments = []
        for si, s in enumerate(w.sessions):
            base = len(self.blocks)
            for j, ins in enumerate(s.inserts):
                self.blocks.append(nexus.block(self.blk_k[si][j], self.blk_v[si][j], ins.length,
                                               ins.base_pos, L, H, rope_theta=w.rope_theta))
            new_pt, segs, _ = nexus.plan_splice(
                self.pool, self.h_pt[2 * si], s.n_past, self.max_pages, self.blocks,
                [(ins.depth, base + j) for j, ins in enumerate(s.inserts)], 2 * si, 2 * si + 1,
                seg_capacity=4 * len(s.inserts) + 4)
            self.h_pt[2 * si + 1] = new_pt
            self.segments += segs
        self.d_pt = torch.as_tensor(self.h_pt, device=dev)
        self.n_rows = n_rows

    def splice(self, stream=None, validate=True):
        nexus.splice_kv(self.cache, self.d_pt, self.h_pt if validate else None, self.n_rows,
                        self.max_pages, self.blocks, self.segments, 0, self.L, stream)

    def live(self, si):
        """Session si's pre-splice K and V (regenerated from the seeds if not kept)."""
        def get(x):
            if isinstance(x, tuple):
                L, n, H, sd = x
                return randn_bf16((L, n, H, 128), sd, self.dev)
            return x
        return get(self.live_k[si]), get(self.live_v[si])

    def inserts_f64(self, si, layers):
        s = self.w.sessions[si]
        return [(ins.depth, f64(self.blk_k[si][j][layers]), f64(self.blk_v[si][j][layers]),
                 ins.base_pos) for j, ins in enumerate(s.inserts)]
