"""Valid-item prefix tree for constrained generation (Sec. 3.1: LLM recommenders
decode only valid item identifiers; Sec. 2: every identifier has length L)."""
from __future__ import annotations

from typing import Dict, Tuple

import numpy as np


class Trie:
    """children(prefix) = sorted codes c such that prefix + (c,) starts some item."""

    def __init__(self, items: np.ndarray):
        items = np.asarray(items)
        self.L = int(items.shape[1])
        kids: Dict[Tuple[int, ...], set] = {}
        for row in items.tolist():
            for l in range(self.L):
                kids.setdefault(tuple(row[:l]), set()).add(int(row[l]))
        self._kids = {p: np.array(sorted(s), dtype=np.int64) for p, s in kids.items()}
        self.items = {tuple(r) for r in items.tolist()}

    def children(self, prefix) -> np.ndarray:
        return self._kids.get(tuple(int(c) for c in prefix), np.zeros(0, dtype=np.int64))

    def is_item(self, seq) -> bool:
        return tuple(int(c) for c in seq) in self.items
