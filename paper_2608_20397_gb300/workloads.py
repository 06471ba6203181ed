"""Seeded synthetic workloads shaped like Qwen2.5-14B attention.

This module only draws random numbers and fixes shapes. It holds none of the
splice, rotation, policy or attention arithmetic, and both the CUDA path and
the fp64 oracle take their inputs from it.

Recipe (all values bf16 from float32 N(0, 1), round-to-nearest-even):

* live K/V of each session: N(0, 1) rows, read as keys already rotated at
  their positions (a rotation maps N(0, I) to N(0, I));
* compiled schema blocks: N(0, 1) rows compiled at anchor ``base_pos``;
* queries: N(0, 1) rows, read as already rotated at their positions;
* integers (block lengths, depths, context lengths, page order) from a
  NumPy PCG64 generator seeded per workload.

Named workloads (Hq = 40, Hkv = 8, d = 128, 16-token pages):

* ``c1``  1 layer, n_past 512, one 128-token block (anchor 0) at depth 300,
  64 suffix queries over the 640-token cache;
* ``c2``  1 layer, n_past 4096, 16 blocks of U{64..512} tokens appended back to
  back at the cursor, suffix of 25 % of the spliced span;
* ``c3``  48 layers, n_past 8192, one 1024-token block at depth 6000,
  transposed-V cache, suffix of {25, 50, 100} % of the 2192 displaced rows;
* ``c4``  32 sessions x 48 layers, n_past log-uniform in [1024, 16384], four
  blocks of U{128..768} tokens at sorted U{0..n_past} depths, suffix 50 % of
  the spliced span, pool pages handed out in a shuffled order;
* ``c5``  48 layers, n_past 32768, one 2048-token block at depth 30000; a full
  causal re-prefill of the 32768-token context and a 64-query suffix over the
  34816-token spliced cache.

Re-decoded suffix tokens (fresh Q, K, V): hidden states x ~ N(0, 1) bf16 of
width 5120; the fused QKV weight [(40 + 2 * 8) * 128][5120] is N(0, 1) bf16
scaled by 2^-6 (exact in bf16), so each projected feature has a standard
deviation near 1.1, as in a trained layer after its input norm; the bias is
float32 N(0, 1) / 2.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import numpy as np
import torch

HIDDEN = 5120
N_Q_HEADS = 40
N_KV_HEADS = 8
HEAD_DIM = 128
PAGE_SIZE = 16
ROPE_THETA = 1.0e6


@dataclasses.dataclass
class Insert:
    depth: int        # position in the pre-splice sequence
    length: int       # block tokens
    base_pos: int     # compile anchor m0 of the block's first token


@dataclasses.dataclass
class Session:
    n_past: int
    inserts: List[Insert]
    suffix_span: int          # S, the span the redecode fraction applies to
    suffix_pct: int           # fixed redecode percentage of S for this workload


@dataclasses.dataclass
class Workload:
    name: str
    n_layers: int
    sessions: List[Session]
    v_transposed: bool = False
    shuffle_pages: bool = False
    seed: int = 0
    suffix_pcts: tuple = ()           # extra percentages swept (c3)
    reprefill: bool = False           # c5: causal self-attention of the pre-splice context
    n_q_heads: int = N_Q_HEADS
    n_kv_heads: int = N_KV_HEADS
    head_dim: int = HEAD_DIM
    page_size: int = PAGE_SIZE
    rope_theta: float = ROPE_THETA

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    def spliced_len(self, s: Session) -> int:
        return s.n_past + sum(i.length for i in s.inserts)


def _rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def workload(name: str, n_layers: Optional[int] = None) -> Workload:
    """One of the named workloads; ``n_layers`` overrides the layer count (tests)."""
    name = name.lower()
    if name == "c1":
        w = Workload("c1", 1, [Session(512, [Insert(300, 128, 0)], 64, 100)], seed=1)
    elif name == "c2":
        r = _rng(2)
        lens = r.integers(64, 512, size=16, endpoint=True)
        ins = [Insert(4096, int(L), 0) for L in lens]
        w = Workload("c2", 1, [Session(4096, ins, int(lens.sum()), 25)], seed=2)
    elif name == "c3":
        w = Workload("c3", 48, [Session(8192, [Insert(6000, 1024, 0)], 2192, 25)],
                     v_transposed=True, seed=3, suffix_pcts=(25, 50, 100))
    elif name == "c4":
        r = _rng(4)
        sessions = []
        for _ in range(32):
            n_past = int(math.floor(math.exp(r.uniform(math.log(1024), math.log(16384)))))
            lens = r.integers(128, 768, size=4, endpoint=True)
            depths = np.sort(r.integers(0, n_past, size=4, endpoint=True))
            ins = [Insert(int(p), int(L), 0) for p, L in zip(depths, lens)]
            sessions.append(Session(n_past, ins, int(lens.sum()), 50))
        w = Workload("c4", 48, sessions, shuffle_pages=True, seed=4)
    elif name == "c5":
        w = Workload("c5", 48, [Session(32768, [Insert(30000, 2048, 0)], 64, 100)],
                     seed=5, reprefill=True)
    else:
        raise KeyError(f"unknown workload {name!r}")
    if n_layers is not None:
        w.n_layers = int(n_layers)
    return w


def page_order(n_pages: int, seed: int, shuffle: bool) -> np.ndarray:
    """Order in which a pool hands out its pages: identity, or a seeded permutation."""
    if not shuffle:
        return np.arange(n_pages, dtype=np.int32)
    return _rng(seed + 1000).permutation(n_pages).astype(np.int32)


def randn_bf16(shape, seed: int, device="cpu") -> torch.Tensor:
    """float32 N(0, 1) from a seeded torch generator, rounded to bf16.

    Large tensors are drawn in slices along dim 0 so the float32 staging stays
    small; each slice has its own derived seed, so the result depends only on
    (shape, seed), not on the device memory available.
    """
    shape = tuple(int(s) for s in shape)
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    if out.numel() == 0:
        return out
    per = max(1, out[0].numel() if len(shape) > 0 else 1)
    chunk = max(1, (1 << 26) // per)
    for i0 in range(0, shape[0], chunk):
        i1 = min(shape[0], i0 + chunk)
        g = torch.Generator(device=device)
        g.manual_seed(int(seed) * 1_000_003 + i0)
        out[i0:i1] = torch.randn((i1 - i0,) + shape[1:], generator=g, device=device,
                                 dtype=torch.float32).to(torch.bfloat16)
    return out


def qkv_weights(n_heads: int, hidden: int, seed: int, device="cpu", bias: bool = True):
    """Fused QKV weight [n_heads * 128][hidden] (bf16) and bias (float32 or None)."""
    w = randn_bf16((n_heads * HEAD_DIM, hidden), seed, device) * (2.0 ** -6)
    b = None
    if bias:
        g = torch.Generator(device=device)
        g.manual_seed(int(seed) * 1_000_003 + 7)
        b = torch.randn((n_heads * HEAD_DIM,), generator=g, device=device, dtype=torch.float32) * 0.5
    return w, b


def agent_requests(seed: int, n_requests: int, n_agents: int = 6, sys_len: int = 300,
                   vocab: int = 50):
    """Token sequences of agent requests, seeded: agents share one system prompt;
    each request extends one agent's history by a reply and a new message; now
    and then an agent starts a new conversation or its history diverges inside
    its last turn (an edit). Yields lists of int token ids."""
    r = _rng(seed)
    system = [int(t) for t in r.integers(0, vocab, sys_len)]

    def fresh():
        return system + [int(t) for t in r.integers(0, vocab, int(r.integers(5, 40)))]

    hist = [fresh() for _ in range(n_agents)]
    for _ in range(n_requests):
        a = int(r.integers(0, n_agents))
        if r.random() < 0.1:
            hist[a] = fresh()
        elif r.random() < 0.15:
            cut = max(len(system), len(hist[a]) - int(r.integers(1, 30)))
            hist[a] = hist[a][:cut] + [int(t) for t in r.integers(vocab, vocab + 10, 4)]
        hist[a] = hist[a] + [int(t) for t in r.integers(0, vocab, int(r.integers(1, 60)))]
        yield list(hist[a])


def tool_registry(n_tools: int, dim: int = 768, seed: int = 0, family: int = 5,
                  spread: float = 0.2):
    """Unit-norm float32 tool embeddings [n_tools][dim] in families of `family`
    tools scattered around a shared direction (tools of one server that share
    words), so that neighbours are close and some top-2 margins are small. With
    the default spread and query noise, the gate threshold 0.0136 falls near the
    20th percentile of the top-2 margins of 250 tools, where the paper puts it."""
    r = _rng(seed)
    n_fam = -(-n_tools // family)
    centers = r.standard_normal((n_fam, dim))
    centers /= np.linalg.norm(centers, axis=1, keepdims=True)
    x = centers[np.arange(n_tools) // family] + spread * r.standard_normal((n_tools, dim)) / np.sqrt(dim)
    x /= np.linalg.norm(x, axis=1, keepdims=True)
    return x.astype(np.float32)


def tool_queries(registry: np.ndarray, n_queries: int, seed: int = 1, noise: float = 1.2):
    """Query embeddings: a tool's embedding plus noise, renormalised; returns
    (queries float32 [n][dim], the tool each was drawn from)."""
    r = _rng(seed)
    n_tools, dim = registry.shape
    src = r.integers(0, n_tools, n_queries)
    q = registry[src].astype(np.float64) + noise * r.standard_normal((n_queries, dim)) / np.sqrt(dim)
    q /= np.linalg.norm(q, axis=1, keepdims=True)
    return q.astype(np.float32), src
