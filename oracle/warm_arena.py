"""Plain model of the L0 exact-token radix arena (Sec. V-D).

TEST INFRASTRUCTURE, like the rest of ``oracle/``: only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU baseline may use it.

The paper describes the arena in one paragraph (Sec. V-D; its latency and
warm-hit rate are in Table III): a fixed pool of 32 sequence slots, a new
request reuses the warm prefix of the slot with the longest exact-token common
prefix, and the prefix's KV is copied within memory reserved up front instead
of being recomputed. This model keeps the slots' tokens and KV rows as plain
arrays and takes every decision by brute force.

Readings where the paper is silent (listed in the design notes):

* match: the slot with the longest common prefix wins; equal prefixes go to
  the most recently used slot; a query sharing no token with any slot is a
  miss (slot -1). Matching reads the arena only.
* fork: a new sequence starts from the first m rows of a slot, m at most the
  slot's length; it counts as a use of the slot.
* store: a finished sequence (its first ``max_tokens`` tokens) enters the
  arena. If a slot already holds a sequence that starts with these tokens, only
  that slot's use is refreshed. Otherwise a slot whose tokens are a prefix of
  the new ones is replaced (the longest such), else the lowest empty slot, else
  the least recently used slot.
* uses are ordered by one counter that each fork and store advances.
* equal tokens mean equal KV rows (the premise of exact-token reuse).
"""
from __future__ import annotations

from typing import List, Optional, Sequence, Tuple

import numpy as np

__all__ = ["common_prefix_len", "warm_match", "WarmArenaModel"]


def common_prefix_len(a: Sequence[int], b: Sequence[int]) -> int:
    """Number of leading positions where the two token sequences agree."""
    n = 0
    for x, y in zip(a, b):
        if int(x) != int(y):
            break
        n += 1
    return n


def warm_match(slot_tokens: List[Optional[Sequence[int]]], last_use: Sequence[int],
               query: Sequence[int]) -> Tuple[int, int]:
    """(slot, prefix length) of the best warm slot for ``query``; (-1, 0) on a miss.

    ``slot_tokens[s]`` is None for an empty slot. Longest prefix first, then the
    most recent use."""
    best, best_len, best_use = -1, 0, -1
    for s, toks in enumerate(slot_tokens):
        if toks is None:
            continue
        n = common_prefix_len(toks, query)
        if n == 0:
            continue
        if n > best_len or (n == best_len and last_use[s] > best_use):
            best, best_len, best_use = s, n, last_use[s]
    return best, best_len


class WarmArenaModel:
    """Slots of (tokens, K rows, V rows) with the decisions of the arena.

    K and V rows are arrays whose axis 1 is the position (e.g. [layer][n][head][d]);
    they are stored and handed out as copies, so the model's contents change only
    through ``store``."""

    def __init__(self, n_slots: int = 32, max_tokens: int = 1 << 20):
        self.n_slots = int(n_slots)
        self.max_tokens = int(max_tokens)
        self.tokens: List[Optional[List[int]]] = [None] * self.n_slots
        self.k: List[Optional[np.ndarray]] = [None] * self.n_slots
        self.v: List[Optional[np.ndarray]] = [None] * self.n_slots
        self.last_use = [0] * self.n_slots
        self.clock = 0

    def _touch(self, s: int):
        self.clock += 1
        self.last_use[s] = self.clock

    def match(self, query: Sequence[int]) -> Tuple[int, int]:
        return warm_match(self.tokens, self.last_use, query)

    def fork(self, s: int, m: int):
        """The first m K and V rows of slot s (copies)."""
        toks = self.tokens[s]
        if toks is None or not 0 <= m <= len(toks):
            raise ValueError("fork outside the slot")
        self._touch(s)
        return self.k[s][:, :m].copy(), self.v[s][:, :m].copy()

    def store(self, tokens: Sequence[int], k: np.ndarray, v: np.ndarray) -> int:
        """Enter a finished sequence; returns the slot that holds it."""
        toks = [int(t) for t in tokens[: self.max_tokens]]
        n = len(toks)
        if n == 0:
            raise ValueError("empty sequence")
        for s, st in enumerate(self.tokens):
            if st is not None and len(st) >= n and st[:n] == toks:
                self._touch(s)
                return s
        target, target_len = -1, -1
        for s, st in enumerate(self.tokens):
            if st is not None and len(st) < n and toks[: len(st)] == st and len(st) > target_len:
                target, target_len = s, len(st)
        if target < 0:
            empty = [s for s, st in enumerate(self.tokens) if st is None]
            if empty:
                target = empty[0]
            else:
                target = min(range(self.n_slots), key=lambda s: self.last_use[s])
        self.tokens[target] = toks
        self.k[target] = np.array(k[:, :n], copy=True)
        self.v[target] = np.array(v[:, :n], copy=True)
        self._touch(target)
        return target
