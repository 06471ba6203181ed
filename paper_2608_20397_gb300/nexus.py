"""Thin ctypes binding of ``libnexus.so`` (see ``include/nexus.h``).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels or its C++ host runtime. Device buffers may be given as torch tensors
(their ``data_ptr()`` is passed) or as raw integer addresses; torch supplies
device memory and streams, nothing else. Importing this module does not load
the library; the first call does, and it raises ``NexusLibraryMissing`` if the
library has not been built (there is no fallback of any kind).
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_int32, c_int64, c_size_t, c_void_p
from fractions import Fraction
from typing import Optional, Sequence

import numpy as np

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libnexus.so")

OK, EINVAL, ERANGE, EROPE_MISMATCH, ELAYOUT, ENOMEM, EDECLINED, ECUDA, ETIMEOUT, EOVERLAP = range(10)
ROPE_NEOX, ROPE_GPTJ = 0, 1
SRC_BLOCK, SRC_CACHE = 0, 1
SEG_K_ONLY = 1


class NexusLibraryMissing(RuntimeError):
    pass


class NexusError(RuntimeError):
    def __init__(self, fn: str, code: int):
        self.code = int(code)
        super().__init__(f"{fn}: {status_string(code)} (status {code})")


class KvCache(ctypes.Structure):
    _fields_ = [
        ("k_pool", c_void_p), ("v_pool", c_void_p), ("n_pages", c_int64),
        ("n_layers", c_int32), ("n_kv_heads", c_int32), ("head_dim", c_int32),
        ("page_size", c_int32), ("v_transposed", c_int32), ("rope_type", c_int32),
        ("rope_theta", c_double), ("rope_freq_scale", c_double),
    ]


class Block(ctypes.Structure):
    _fields_ = [
        ("k", c_void_p), ("v", c_void_p), ("n_tokens", c_int32), ("base_pos", c_int32),
        ("n_layers", c_int32), ("n_kv_heads", c_int32), ("head_dim", c_int32),
        ("rope_type", c_int32), ("rope_theta", c_double), ("rope_freq_scale", c_double),
    ]


class Segment(ctypes.Structure):
    _fields_ = [
        ("src_kind", c_int32), ("src_index", c_int32), ("src_start", c_int32),
        ("dst_row", c_int32), ("dst_start", c_int32), ("n_tokens", c_int32),
        ("delta", c_int32), ("flags", c_int32),
    ]


class Policy(ctypes.Structure):
    _fields_ = [("splice_threshold", c_int32), ("r_base_pct", c_int32), ("full_mult", c_int32)]


class Insert(ctypes.Structure):
    _fields_ = [("depth", c_int32), ("block_index", c_int32)]


DEFAULT_POLICY = (256, 5, 4)   # P = M = 256, R_base = 5 %, K = 4 (Sec. III-B / III-C)

_i32p = POINTER(c_int32)
_SIGS = {
    "nexus_status_string": (ctypes.c_char_p, [c_int32]),
    "nexus_version": (c_int32, []),
    "nexus_device_status": (c_int32, [c_void_p]),
    "nexus_recompute_pct": (c_int32, [c_int32, POINTER(Policy), POINTER(c_int64), POINTER(c_int64)]),
    "nexus_redecode_len": (c_int32, [c_int32, c_int32, POINTER(Policy)]),
    "nexus_suffix_len": (c_int32, [c_int32, c_int32]),
    "nexus_check_splice": (c_int32, [c_int32, c_int32, c_int32, POINTER(Policy)]),
    "nexus_page_pool_create": (c_int32, [c_int64, _i32p, POINTER(c_void_p)]),
    "nexus_page_pool_destroy": (None, [c_void_p]),
    "nexus_page_pool_alloc": (c_int32, [c_void_p, c_int32, _i32p]),
    "nexus_page_pool_free": (c_int32, [c_void_p, c_int32, _i32p]),
    "nexus_page_pool_available": (c_int64, [c_void_p]),
    "nexus_page_pool_retain": (c_int32, [c_void_p, c_int32, _i32p]),
    "nexus_page_pool_refs": (c_int64, [c_void_p, c_int32]),
    "nexus_page_pool_make_private": (c_int32, [c_void_p, _i32p, c_int32, c_int32, _i32p, _i32p,
                                               c_int32, _i32p]),
    "nexus_warm_arena_create": (c_int32, [c_int32, c_int32, POINTER(c_void_p)]),
    "nexus_warm_arena_destroy": (None, [c_void_p, c_void_p]),
    "nexus_warm_arena_match": (c_int32, [c_void_p, _i32p, c_int32, _i32p, _i32p]),
    "nexus_warm_arena_fork": (c_int32, [c_void_p, c_void_p, c_int32, c_int32, _i32p, c_int32,
                                        _i32p, _i32p, _i32p]),
    "nexus_warm_arena_store": (c_int32, [c_void_p, c_void_p, _i32p, c_int32, _i32p, _i32p]),
    "nexus_warm_arena_slot": (c_int32, [c_void_p, c_int32, _i32p, _i32p, c_int32]),
    "nexus_slb_quantize": (c_int32, [c_void_p, c_int32, c_int32, c_void_p, c_void_p]),
    "nexus_slb_workspace_size": (c_size_t, [c_int32]),
    "nexus_slb_route": (c_int32, [c_void_p, c_void_p, c_int32, c_int32, c_void_p, c_void_p,
                                  c_int32, ctypes.c_float, c_void_p, c_void_p, c_void_p,
                                  c_void_p, c_size_t, c_void_p]),
    "nexus_plan_splice": (c_int32, [c_void_p, _i32p, c_int32, c_int32, POINTER(Block), c_int32,
                                    POINTER(Insert), c_int32, c_int32, c_int32, _i32p,
                                    POINTER(Segment), c_int32, _i32p, _i32p, _i32p]),
    "nexus_splice_kv": (c_int32, [POINTER(KvCache), c_void_p, _i32p, c_int32, c_int32,
                                  POINTER(Block), c_int32, POINTER(Segment), c_int32,
                                  c_int32, c_int32, c_void_p]),
    "nexus_rope_rerotate": (c_int32, [POINTER(KvCache), c_void_p, _i32p, c_int32, c_int32, c_int32,
                                      c_int32, c_int32, c_int32, c_int32, c_int32, c_void_p]),
    "nexus_rope_rerotate_f32": (c_int32, [POINTER(KvCache), c_void_p, _i32p, c_int32, c_int32,
                                          c_int32, c_int32, c_int32, c_int32, c_int32, c_int32,
                                          c_void_p, c_void_p]),
    "nexus_copy_pages": (c_int32, [POINTER(KvCache), _i32p, _i32p, c_int32, c_int32, c_int32,
                                   c_void_p]),
    "nexus_suffix_attention": (c_int32, [POINTER(KvCache), c_void_p, c_int32, c_int32, c_int32,
                                         _i32p, _i32p, _i32p, c_void_p, c_void_p, c_void_p,
                                         c_int32, c_int32, c_int32, c_int32, c_void_p, c_size_t,
                                         c_void_p]),
    "nexus_suffix_attention_softcap": (c_int32, [POINTER(KvCache), c_void_p, c_int32, c_int32,
                                                 c_int32, _i32p, _i32p, _i32p, c_void_p,
                                                 c_void_p, c_void_p, c_int32, c_int32, c_int32,
                                                 c_int32, c_void_p, c_size_t, ctypes.c_float,
                                                 c_void_p]),
    "nexus_reprefill": (c_int32, [POINTER(KvCache), c_void_p, c_int32, c_int32, c_int32, _i32p,
                                  _i32p, c_void_p, c_void_p, c_void_p, c_int32, c_int32, c_int32,
                                  c_int32, c_void_p, c_size_t, c_void_p]),
    "nexus_attention_workspace_size": (c_size_t, [c_int32, _i32p, _i32p, c_int32, c_int32,
                                                  c_int32, c_int32, _i32p]),
    "nexus_suffix_attention_noalloc": (c_int32, [POINTER(KvCache), c_void_p, c_int32, c_int32,
                                                 c_int32, _i32p, _i32p, _i32p, c_void_p,
                                                 c_void_p, c_void_p, c_int32, c_int32, c_int32,
                                                 c_int32, c_void_p]),
    "nexus_suffix_qkv": (c_int32, [POINTER(KvCache), c_void_p, _i32p, c_int32, c_int32, c_int32,
                                   _i32p, _i32p, _i32p, c_void_p, c_int32, c_void_p, c_void_p,
                                   c_int32, c_int32, c_void_p, c_void_p]),
    "nexus_selftest_wait": (c_int32, [ctypes.c_uint32, c_void_p]),
    "nexus_host_alloc": (c_int32, [c_size_t, POINTER(c_void_p)]),
    "nexus_host_free": (c_int32, [c_void_p, c_size_t]),
}
EXPORTED = tuple(_SIGS)

_lib = None


def lib():
    """The loaded library; raises NexusLibraryMissing if it was never built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise NexusLibraryMissing(
                f"{LIB_PATH} is missing: build it with __graft_entry__.build() (no fallback exists)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def status_string(code: int) -> str:
    return lib().nexus_status_string(int(code)).decode()


def _check(fn: str, code: int):
    if code != OK:
        raise NexusError(fn, code)


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _i32(a) -> Optional[ctypes.Array]:
    """A host int32 array as a ctypes buffer (kept alive by the caller's scope)."""
    if a is None:
        return None
    arr = np.ascontiguousarray(np.asarray(a, dtype=np.int32))
    return arr.ctypes.data_as(_i32p), arr


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def _policy(policy) -> Policy:
    p = policy if policy is not None else DEFAULT_POLICY
    return Policy(int(p[0]), int(p[1]), int(p[2]))


# ---------------------------------------------------------------- policy
def recompute_pct(n_past: int, policy=None) -> Fraction:
    num, den = c_int64(), c_int64()
    pol = _policy(policy)
    _check("nexus_recompute_pct", lib().nexus_recompute_pct(int(n_past), ctypes.byref(pol),
                                                            ctypes.byref(num), ctypes.byref(den)))
    return Fraction(num.value, den.value)


def redecode_len(S: int, n_past: int, policy=None) -> int:
    pol = _policy(policy)
    r = lib().nexus_redecode_len(int(S), int(n_past), ctypes.byref(pol))
    if r < 0:
        raise NexusError("nexus_redecode_len", EINVAL)
    return int(r)


def suffix_len(S: int, pct: int) -> int:
    r = lib().nexus_suffix_len(int(S), int(pct))
    if r < 0:
        raise NexusError("nexus_suffix_len", EINVAL)
    return int(r)


def check_splice(n_past: int, S: int, n_redecode: int, policy=None) -> int:
    pol = _policy(policy)
    return int(lib().nexus_check_splice(int(n_past), int(S), int(n_redecode), ctypes.byref(pol)))


# ------------------------------------------------------------- page pool
class PagePool:
    def __init__(self, n_pages: int, order: Optional[Sequence[int]] = None):
        h = c_void_p()
        buf = _i32(order)
        _check("nexus_page_pool_create",
               lib().nexus_page_pool_create(int(n_pages), buf[0] if buf else None, ctypes.byref(h)))
        self._h = h
        self.n_pages = int(n_pages)

    @property
    def handle(self):
        return self._h

    def alloc(self, n: int) -> np.ndarray:
        out = np.zeros(int(n), dtype=np.int32)
        _check("nexus_page_pool_alloc",
               lib().nexus_page_pool_alloc(self._h, int(n), out.ctypes.data_as(_i32p)))
        return out

    def free(self, pages) -> None:
        buf = _i32(pages)
        _check("nexus_page_pool_free", lib().nexus_page_pool_free(self._h, len(buf[1]), buf[0]))

    def available(self) -> int:
        return int(lib().nexus_page_pool_available(self._h))

    def retain(self, pages) -> None:
        buf = _i32(pages)
        _check("nexus_page_pool_retain", lib().nexus_page_pool_retain(self._h, len(buf[1]), buf[0]))

    def refs(self, page: int) -> int:
        return int(lib().nexus_page_pool_refs(self._h, int(page)))

    def make_private(self, pt: np.ndarray, first_page: int, n: int):
        """Copy-on-write of pt[first_page, first_page + n) in place (pt: int32
        array); returns the (old, fresh) page pairs to copy before writing."""
        assert pt.dtype == np.int32 and pt.flags.c_contiguous
        cap = max(int(n), 1)
        src = np.zeros(cap, np.int32)
        dst = np.zeros(cap, np.int32)
        k = c_int32()
        _check("nexus_page_pool_make_private", lib().nexus_page_pool_make_private(
            self._h, pt.ctypes.data_as(_i32p), int(first_page), int(n),
            src.ctypes.data_as(_i32p), dst.ctypes.data_as(_i32p), cap, ctypes.byref(k)))
        return src[:k.value].copy(), dst[:k.value].copy()

    def close(self):
        if self._h:
            lib().nexus_page_pool_destroy(self._h)
            self._h = c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# -------------------------------------------------------------- structs
def kv_cache(k_pool, v_pool, n_pages: int, n_layers: int, n_kv_heads: int = 8,
             v_transposed: bool = False, rope_type: int = ROPE_NEOX, rope_theta: float = 1.0e6,
             rope_freq_scale: float = 1.0) -> KvCache:
    c = KvCache(_ptr(k_pool), _ptr(v_pool), int(n_pages), int(n_layers), int(n_kv_heads), 128,
                16, int(bool(v_transposed)), int(rope_type), float(rope_theta),
                float(rope_freq_scale))
    c._keep = (k_pool, v_pool)   # the descriptor holds raw pointers: keep the buffers alive
    return c


def block(k, v, n_tokens: int, base_pos: int, n_layers: int, n_kv_heads: int = 8,
          rope_type: int = ROPE_NEOX, rope_theta: float = 1.0e6,
          rope_freq_scale: float = 1.0) -> Block:
    b = Block(_ptr(k), _ptr(v), int(n_tokens), int(base_pos), int(n_layers), int(n_kv_heads),
              128, int(rope_type), float(rope_theta), float(rope_freq_scale))
    b._keep = (k, v)
    return b


def segments_array(segs) -> ctypes.Array:
    arr = (Segment * max(1, len(segs)))()
    for i, s in enumerate(segs):
        arr[i] = s if isinstance(s, Segment) else Segment(*[int(x) for x in s])
    return arr


# --------------------------------------------------------------- planner
def plan_splice(pool: PagePool, old_pt, n_past: int, max_pages: int, blocks: Sequence[Block],
                inserts: Sequence[tuple], old_row: int, new_row: int, seg_capacity: int = 64):
    """Returns (new_pt [max_pages] int32, list of Segment, freed pages)."""
    barr = (Block * max(1, len(blocks)))(*blocks)
    iarr = (Insert * max(1, len(inserts)))(*[Insert(int(d), int(b)) for d, b in inserts])
    old = _i32(old_pt if old_pt is not None else np.zeros(max_pages, np.int32))
    new_pt = np.zeros(int(max_pages), dtype=np.int32)
    segs = (Segment * seg_capacity)()
    nseg = c_int32()
    freed = np.zeros(int(max_pages), dtype=np.int32)
    nfreed = c_int32()
    _check("nexus_plan_splice", lib().nexus_plan_splice(
        pool.handle, old[0], int(n_past), int(max_pages), barr, len(blocks), iarr, len(inserts),
        int(old_row), int(new_row), new_pt.ctypes.data_as(_i32p), segs, int(seg_capacity),
        ctypes.byref(nseg), freed.ctypes.data_as(_i32p), ctypes.byref(nfreed)))
    return new_pt, [segs[i] for i in range(nseg.value)], freed[: nfreed.value].copy()


# ---------------------------------------------------------------- device
def splice_kv(cache: KvCache, d_page_tables, h_page_tables, n_rows: int, max_pages: int,
              blocks: Sequence[Block], segments, layer_begin: int, layer_end: int, stream=None):
    barr = (Block * max(1, len(blocks)))(*blocks)
    sarr = segments_array(segments)
    hpt = _i32(h_page_tables)
    _check("nexus_splice_kv", lib().nexus_splice_kv(
        ctypes.byref(cache), _ptr(d_page_tables), hpt[0] if hpt else None, int(n_rows),
        int(max_pages), barr, len(blocks), sarr, len(segments), int(layer_begin), int(layer_end),
        _stream(stream)))


def rope_rerotate(cache: KvCache, d_page_tables, h_page_tables, n_rows: int, max_pages: int,
                  row: int, pos_begin: int, n_tokens: int, delta: int, layer_begin: int,
                  layer_end: int, stream=None):
    hpt = _i32(h_page_tables)
    _check("nexus_rope_rerotate", lib().nexus_rope_rerotate(
        ctypes.byref(cache), _ptr(d_page_tables), hpt[0] if hpt else None, int(n_rows),
        int(max_pages), int(row), int(pos_begin), int(n_tokens), int(delta), int(layer_begin),
        int(layer_end), _stream(stream)))


def rope_rerotate_f32(cache: KvCache, d_page_tables, h_page_tables, n_rows: int, max_pages: int,
                      row: int, pos_begin: int, n_tokens: int, delta: int, layer_begin: int,
                      layer_end: int, out_f32, stream=None):
    hpt = _i32(h_page_tables)
    _check("nexus_rope_rerotate_f32", lib().nexus_rope_rerotate_f32(
        ctypes.byref(cache), _ptr(d_page_tables), hpt[0] if hpt else None, int(n_rows),
        int(max_pages), int(row), int(pos_begin), int(n_tokens), int(delta), int(layer_begin),
        int(layer_end), _ptr(out_f32), _stream(stream)))


def copy_pages(cache: KvCache, src_pages, dst_pages, layer_begin: int, layer_end: int, stream=None):
    s = _i32(src_pages)
    d = _i32(dst_pages)
    _check("nexus_copy_pages", lib().nexus_copy_pages(
        ctypes.byref(cache), s[0], d[0], len(s[1]), int(layer_begin), int(layer_end),
        _stream(stream)))


def attention_workspace_size(kv_len, q_len, n_q_heads: int, n_kv_heads: int, n_layers_call: int,
                             split_kv: int = 0):
    kv = _i32(kv_len)
    ql = _i32(q_len)
    splits = c_int32()
    n = lib().nexus_attention_workspace_size(len(kv[1]), kv[0], ql[0], int(n_q_heads),
                                             int(n_kv_heads), int(n_layers_call), int(split_kv),
                                             ctypes.byref(splits))
    return int(n), int(splits.value)


def suffix_attention(cache: KvCache, d_page_tables, n_rows: int, max_pages: int, kv_len, q_len,
                     q, out, lse=None, n_q_heads: int = 40, layer_begin: int = 0,
                     layer_end: int = 1, rows=None, split_kv: int = 0, workspace=None,
                     workspace_bytes: int = 0, stream=None):
    kv = _i32(kv_len)
    ql = _i32(q_len)
    rw = _i32(rows)
    _check("nexus_suffix_attention", lib().nexus_suffix_attention(
        ctypes.byref(cache), _ptr(d_page_tables), int(n_rows), int(max_pages), len(kv[1]),
        rw[0] if rw else None, kv[0], ql[0], _ptr(q), _ptr(out), _ptr(lse), int(n_q_heads),
        int(layer_begin), int(layer_end), int(split_kv), _ptr(workspace), int(workspace_bytes),
        _stream(stream)))


def suffix_attention_softcap(cache: KvCache, d_page_tables, n_rows: int, max_pages: int, kv_len,
                             q_len, q, out, lse=None, n_q_heads: int = 40, layer_begin: int = 0,
                             layer_end: int = 1, rows=None, split_kv: int = 0, workspace=None,
                             workspace_bytes: int = 0, softcap: float = 50.0, stream=None):
    kv = _i32(kv_len)
    ql = _i32(q_len)
    rw = _i32(rows)
    _check("nexus_suffix_attention_softcap", lib().nexus_suffix_attention_softcap(
        ctypes.byref(cache), _ptr(d_page_tables), int(n_rows), int(max_pages), len(kv[1]),
        rw[0] if rw else None, kv[0], ql[0], _ptr(q), _ptr(out), _ptr(lse), int(n_q_heads),
        int(layer_begin), int(layer_end), int(split_kv), _ptr(workspace), int(workspace_bytes),
        float(softcap), _stream(stream)))


def reprefill(cache: KvCache, d_page_tables, n_rows: int, max_pages: int, kv_len, q, out,
              lse=None, n_q_heads: int = 40, layer_begin: int = 0, layer_end: int = 1, rows=None,
              split_kv: int = 1, workspace=None, workspace_bytes: int = 0, stream=None):
    kv = _i32(kv_len)
    rw = _i32(rows)
    _check("nexus_reprefill", lib().nexus_reprefill(
        ctypes.byref(cache), _ptr(d_page_tables), int(n_rows), int(max_pages), len(kv[1]),
        rw[0] if rw else None, kv[0], _ptr(q), _ptr(out), _ptr(lse), int(n_q_heads),
        int(layer_begin), int(layer_end), int(split_kv), _ptr(workspace), int(workspace_bytes),
        _stream(stream)))


def device_status(stream=None) -> int:
    """Synchronises the stream; OK, ETIMEOUT (a bounded device wait gave up) or ECUDA."""
    return int(lib().nexus_device_status(_stream(stream)))


def selftest_wait(budget_us: int = 2000, stream=None) -> None:
    """Launches the bounded-wait self-test (see nexus_selftest_wait): the next
    device_status() reports ETIMEOUT."""
    _check("nexus_selftest_wait", lib().nexus_selftest_wait(int(budget_us), _stream(stream)))


def suffix_attention_noalloc(cache: KvCache, d_page_tables, n_rows: int, max_pages: int, kv_len,
                             q_len, q, out, lse=None, n_q_heads: int = 40, layer_begin: int = 0,
                             layer_end: int = 1, rows=None, split_kv: int = 0, stream=None):
    """nexus_suffix_attention for callers that cannot allocate device memory:
    the split partials use the library's own 32 MiB array (see nexus.h)."""
    kv = _i32(kv_len)
    ql = _i32(q_len)
    rw = _i32(rows)
    _check("nexus_suffix_attention_noalloc", lib().nexus_suffix_attention_noalloc(
        ctypes.byref(cache), _ptr(d_page_tables), int(n_rows), int(max_pages), len(kv[1]),
        rw[0] if rw else None, kv[0], ql[0], _ptr(q), _ptr(out), _ptr(lse), int(n_q_heads),
        int(layer_begin), int(layer_end), int(split_kv), _stream(stream)))


def suffix_qkv(cache: KvCache, d_page_tables, n_rows: int, max_pages: int, kv_len, q_len, x,
               w_qkv, b_qkv, q_out, layer: int = 0, n_q_heads: int = 40, rows=None,
               h_page_tables=None, hidden: Optional[int] = None, stream=None):
    """Fresh Q, K, V of the re-decoded suffix tokens of one layer (see nexus.h):
    x [sum q_len][hidden] bf16, w_qkv [(Hq + 2 Hkv) 128][hidden] bf16, b_qkv float
    or None; Q goes to q_out [sum q_len][Hq][128], K and V into the cache."""
    kv = _i32(kv_len)
    ql = _i32(q_len)
    rw = _i32(rows)
    hpt = _i32(h_page_tables)
    _check("nexus_suffix_qkv", lib().nexus_suffix_qkv(
        ctypes.byref(cache), _ptr(d_page_tables), hpt[0] if hpt else None, int(n_rows),
        int(max_pages), len(kv[1]), rw[0] if rw else None, kv[0], ql[0], _ptr(x),
        int(hidden if hidden is not None else x.shape[-1]), _ptr(w_qkv), _ptr(b_qkv), int(n_q_heads),
        int(layer), _ptr(q_out), _stream(stream)))


# ------------------------------------------------------------ warm arena
class WarmArena:
    """The L0 exact-token radix arena of warm prefixes (see nexus.h)."""

    def __init__(self, n_slots: int = 32, max_tokens: int = 1 << 16):
        h = c_void_p()
        _check("nexus_warm_arena_create",
               lib().nexus_warm_arena_create(int(n_slots), int(max_tokens), ctypes.byref(h)))
        self._h = h
        self.n_slots = int(n_slots)
        self.max_tokens = int(max_tokens)

    def match(self, tokens):
        buf = _i32(tokens)
        slot, pre = c_int32(), c_int32()
        _check("nexus_warm_arena_match", lib().nexus_warm_arena_match(
            self._h, buf[0], len(buf[1]), ctypes.byref(slot), ctypes.byref(pre)))
        return slot.value, pre.value

    def fork(self, pool: PagePool, slot: int, m: int, max_pages: int):
        """Page table prefix (int32 [ceil(m / 16)]) of a sequence started from
        the first m tokens of `slot`, and the page copies to run first."""
        pt = np.full(max(int(max_pages), 1), -1, np.int32)
        src = np.zeros(1, np.int32)
        dst = np.zeros(1, np.int32)
        k = c_int32()
        _check("nexus_warm_arena_fork", lib().nexus_warm_arena_fork(
            self._h, pool.handle, int(slot), int(m), pt.ctypes.data_as(_i32p), int(max_pages),
            src.ctypes.data_as(_i32p), dst.ctypes.data_as(_i32p), ctypes.byref(k)))
        return pt[: -(-int(m) // 16)].copy(), src[:k.value].copy(), dst[:k.value].copy()

    def store(self, pool: PagePool, tokens, pt) -> int:
        tb = _i32(tokens)
        pb = _i32(pt)
        slot = c_int32()
        _check("nexus_warm_arena_store", lib().nexus_warm_arena_store(
            self._h, pool.handle, tb[0], len(tb[1]), pb[0], ctypes.byref(slot)))
        return slot.value

    def slot(self, slot: int):
        """(token count, pages) of a slot."""
        n = c_int32()
        pages = np.zeros(-(-self.max_tokens // 16), np.int32)
        _check("nexus_warm_arena_slot", lib().nexus_warm_arena_slot(
            self._h, int(slot), ctypes.byref(n), pages.ctypes.data_as(_i32p), len(pages)))
        return n.value, pages[: -(-n.value // 16)].copy()

    def close(self, pool: Optional[PagePool] = None):
        if self._h:
            lib().nexus_warm_arena_destroy(self._h, pool.handle if pool is not None else None)
            self._h = c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# ------------------------------------------------------ INT8 tool scan + gate
def slb_quantize(x: np.ndarray):
    """Host INT8 quantisation of embedding rows: (codes int8, scales float32)."""
    x = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    n, dim = x.shape
    codes = np.zeros((n, dim), np.int8)
    scales = np.zeros(n, np.float32)
    _check("nexus_slb_quantize", lib().nexus_slb_quantize(
        x.ctypes.data, int(n), int(dim), codes.ctypes.data, scales.ctypes.data))
    return codes, scales


def slb_workspace_size(n_tools: int) -> int:
    return int(lib().nexus_slb_workspace_size(int(n_tools)))


def slb_route(tools, tool_scales, queries, query_scales, top_idx, top_score, route, workspace,
              tau: float = 0.0136, stream=None):
    """Scan and gate on device tensors (see nexus.h): tools int8 [N][dim],
    queries int8 [Q][dim]; writes top_idx int32 [Q][2], top_score float [Q][2],
    route int32 [Q]. The workspace (nexus_slb_workspace_size bytes) starts zeroed."""
    _check("nexus_slb_route", lib().nexus_slb_route(
        _ptr(tools), _ptr(tool_scales), int(tools.shape[0]), int(tools.shape[1]), _ptr(queries),
        _ptr(query_scales), int(queries.shape[0]), float(tau), _ptr(top_idx), _ptr(top_score),
        _ptr(route), _ptr(workspace), int(workspace.numel()), _stream(stream)))


# ---------------------------------------------------- host staging memory
class _HostMapping:
    """Owns one nexus_host_alloc mapping; freed when the last tensor viewing it
    is gone."""

    def __init__(self, nbytes: int):
        self.ptr, self.nbytes = 0, int(nbytes)   # set before the call that can fail
        p = c_void_p()
        _check("nexus_host_alloc", lib().nexus_host_alloc(int(nbytes), ctypes.byref(p)))
        self.ptr, self.nbytes = int(p.value), int(nbytes)

    def __del__(self):
        if self.ptr and _lib is not None:
            _lib.nexus_host_free(c_void_p(self.ptr), c_size_t(self.nbytes))
            self.ptr = 0


def host_empty(shape, dtype):
    """A CPU torch tensor of ``shape`` / ``dtype`` (zero-filled) in page-locked
    staging memory from nexus_host_alloc: copies between it and the device with
    ``non_blocking=True`` are asynchronous (torch's ``is_pinned()`` reports only
    its own allocator's memory and says False here). The memory is returned when
    the tensor and every view of it are gone."""
    import torch
    shape = tuple(int(n) for n in shape)
    nbytes = int(np.prod(shape, dtype=np.int64)) * torch.empty((), dtype=dtype).element_size()
    m = _HostMapping(max(nbytes, 1))
    raw = (ctypes.c_char * max(nbytes, 1)).from_address(m.ptr)
    raw._mapping = m                        # the tensor's storage keeps `raw`, and so `m`, alive
    return torch.frombuffer(raw, dtype=torch.uint8)[:nbytes].view(dtype).view(shape)


_GROUP_ALIGN = 1 << 16


def host_empty_group(specs):
    """Several staging tensors, ``[(shape, dtype), ...]``, carved out of ONE
    nexus_host_alloc mapping at 64 KiB-aligned offsets, in order. Small buffers
    staged together this way share the huge pages a large mapping gets (a
    mapping of less than a quarter of the huge page size is made of base pages,
    from which copies can be many times slower). Returns the tensors as a list;
    the mapping lives while any of them does."""
    import torch
    layout, total = [], 0
    for shape, dtype in specs:
        shape = tuple(int(n) for n in shape)
        nbytes = int(np.prod(shape, dtype=np.int64)) * torch.empty((), dtype=dtype).element_size()
        layout.append((total, nbytes, shape, dtype))
        total += -(-nbytes // _GROUP_ALIGN) * _GROUP_ALIGN
    if not layout:
        return []
    base = host_empty((max(total, 1),), torch.uint8)
    return [base[off:off + n].view(dtype).view(shape) for off, n, shape, dtype in layout]
