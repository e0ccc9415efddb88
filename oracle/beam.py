"""Constrained log-softmax, beam expansion and exact top-K (fp32, the kernels' precision).

Beam search over item identifiers (Sec. 2: the target "generates top-K ranked
items via beam search"), restricted to valid identifiers (Sec. 3.1,
constrained generation).  Readings where the paper is silent:

* MASKED normalisation (default): lp(c | b) = logit_c - logsumexp over the
  valid children of b; FULL: logsumexp over the whole vocabulary, then mask.
* a sequence score is the fp32 sum of its token log-probs, in token order;
* candidates of a level are indexed parent_rank * 256 + code and ranked by
  (score descending, index ascending): exact ties go to the lower index;
* when fewer than K candidates exist all are kept.
"""
from __future__ import annotations

from typing import List, Optional, Sequence, Tuple

import numpy as np

F32 = np.float32
CODES = 256


def logsumexp_f32(x: np.ndarray) -> np.float32:
    x = np.asarray(x, dtype=F32)
    m = np.max(x)
    s = np.sum(np.exp(x - m), dtype=F32)
    return F32(m + np.log(s))


def constrained_logprobs(logits_level: np.ndarray, children: np.ndarray,
                         full_row: Optional[np.ndarray] = None) -> np.ndarray:
    """fp32 log-probs of the valid children (MASKED), or of the children under the
    full-vocabulary normaliser when ``full_row`` (the whole logit row) is given."""
    x = np.asarray(logits_level, dtype=F32)[children]
    lse = logsumexp_f32(full_row) if full_row is not None else logsumexp_f32(x)
    return (x - lse).astype(F32)


class Cands:
    """Candidates of one level in index order: parent rank, code, fp32 score."""

    def __init__(self, parent: np.ndarray, code: np.ndarray, score: np.ndarray):
        self.parent = np.asarray(parent, dtype=np.int64)
        self.code = np.asarray(code, dtype=np.int64)
        self.score = np.asarray(score, dtype=F32)

    @property
    def index(self) -> np.ndarray:
        return self.parent * CODES + self.code

    def __len__(self) -> int:
        return int(self.parent.shape[0])


def expand(paths: Sequence[Tuple[int, ...]], scores: Sequence[float], rows: Sequence[np.ndarray], trie,
           full_rows: Optional[Sequence[np.ndarray]] = None) -> Cands:
    """Every valid one-token extension of every beam, scored S_b + lp(c | b) in fp32."""
    par, cod, sc = [], [], []
    for r, (p, s, row) in enumerate(zip(paths, scores, rows)):
        kids = trie.children(p)
        if kids.size == 0:
            continue
        lp = constrained_logprobs(row, kids, None if full_rows is None else full_rows[r])
        par.append(np.full(kids.size, r))
        cod.append(kids)
        sc.append((F32(s) + lp).astype(F32))
    if not par:
        return Cands(np.zeros(0), np.zeros(0), np.zeros(0))
    return Cands(np.concatenate(par), np.concatenate(cod), np.concatenate(sc))


def rank_order(score: np.ndarray, index: np.ndarray) -> np.ndarray:
    """Permutation sorting by (score descending, index ascending)."""
    return np.lexsort((np.asarray(index), -np.asarray(score, dtype=np.float64)))


def topk(c: Cands, k: int) -> np.ndarray:
    """Positions (into ``c``) of the exact top-k, ranked."""
    return rank_order(c.score, c.index)[:k]


def child_paths(paths: Sequence[Tuple[int, ...]], c: Cands, sel: np.ndarray) -> List[Tuple[int, ...]]:
    return [tuple(paths[int(c.parent[i])]) + (int(c.code[i]),) for i in sel]
