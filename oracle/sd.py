"""Speculative beam decoding for generative recommendation (Sec. 2, Sec. 3.2, Alg. 1, Alg. 2).

One SD step at depth d (0 <= d < L, L = 4 codes per item):

* drafting (Eq. 1): gamma' = min(gamma, L - d) beam-search steps of the draft
  model with width N.  Strict mode keeps the top-N candidates; relaxed mode
  samples N distinct candidates from q_j = softmax of the draft's sequence
  scores over the level's candidates (Alg. 2, "Sample ... from q_j").  Level 1
  extends the incoming beams, which carry the target's scores (reading: the
  draft continues the target's beam state).
* one target call over every drafted beam (tree attention, Sec. 3.3): logits
  for the incoming beams (d > 0; at d = 0 the prefill gives them) and for the
  drafted levels 1 .. min(gamma', L - d - 1) (level-L tokens complete an item).
* verification:
  - strict (Alg. 1): Y^p_j = top-K over the extensions of Y^p_{j-1} with target
    scores; step j is accepted iff Y^p_j is a subset of Y^q_j (the paper's
    "Y_p in Y_q"); stop at the first rejection and output Y^p there; if all
    gamma' steps pass, output Y^p_{gamma'+1} (or Y^p_{gamma'} when the item is
    complete).  Extending Y^p_{j-1} rather than all drafted beams is the reading
    under which the method is lossless, as the paper states and reports.
  - relaxed (Sec. 3.2, Alg. 2): C_j = extensions of the drafted Y^q_{j-1};
    p_j, q_j = softmax over C_j of the target / draft sequence scores; every
    drafted y is accepted iff u <= min(1, p_j(y)/q_j(y)); |A| >= K accepts the
    step; otherwise output A plus K - |A| draws from norm(max(0, p_j - q_j))
    (zero on A; p_j on C_j \\ A when that mass is zero) and stop.  All steps
    accepted: K draws from p_{gamma'+1}, or K uniform picks from A when the
    item is complete.
* advance = min(a + 1, L - d) with a the number of accepted steps.

Sampling without replacement is done with Gumbel keys (top-n of log-weight +
Gumbel noise), which has the same law as n sequential draws that renormalise
after each draw.  All scores and decisions are fp32.
"""
from __future__ import annotations

import dataclasses
from typing import Callable, Dict, List, Optional, Sequence, Tuple

import numpy as np

from .beam import Cands, child_paths, expand, logsumexp_f32, rank_order, topk
from .philox import (STREAM_ACCEPT, STREAM_DRAFT, STREAM_RESAMPLE, STREAM_SUBSET, draw_u32, gumbel,
                     u_accept)

F32 = np.float32
Path = Tuple[int, ...]
RowsFn = Callable[[Sequence[Path]], List[np.ndarray]]


@dataclasses.dataclass
class StepResult:
    a: int                      # accepted steps
    advance: int                # depth gained by this SD step
    paths: List[Path]           # output beams, ranked
    scores: np.ndarray          # fp32 target scores of the output beams
    n_accepted_last: int = 0    # |A| at the last verified level (relaxed)


@dataclasses.dataclass
class Tree:
    d: int
    incoming: List[Path]
    incoming_sp: np.ndarray           # fp32 target scores of the incoming beams
    levels: List[List[Path]]          # drafted Y^q_1 .. Y^q_gamma', draft order
    levels_sq: List[np.ndarray]       # fp32 draft scores of the drafted beams


@dataclasses.dataclass
class Philox:
    seed: int
    sd_step: int
    user: int

    def u32(self, stream: int, level: int, draw) -> np.ndarray:
        return draw_u32(self.seed, stream, level, self.sd_step, self.user, draw)

    def gumbel(self, stream: int, level: int, draw) -> np.ndarray:
        return gumbel(self.u32(stream, level, draw))


def tree_tokens(tree: Tree, L: int) -> int:
    """Tokens the target forwards in the verification call: incoming beams (d > 0)
    plus drafted levels 1 .. min(gamma', L - d - 1)."""
    R = 0 if tree.d == 0 else len(tree.incoming)
    upto = min(len(tree.levels), L - tree.d - 1)
    return R + sum(len(tree.levels[j]) for j in range(upto))


def forwarded_paths(tree: Tree, L: int) -> List[Path]:
    out = list(tree.incoming)
    upto = min(len(tree.levels), L - tree.d - 1)
    for j in range(upto):
        out += tree.levels[j]
    return out


def _guard(rows_fn: RowsFn, allowed: Sequence[Path]) -> RowsFn:
    ok = set(allowed)

    def f(paths):
        for p in paths:
            assert tuple(p) in ok, f"target logits requested for a node outside the drafted tree: {p}"
        return rows_fn(paths)
    return f


# ------------------------------------------------------------------------------------------------
# drafting (Eq. 1)
# ------------------------------------------------------------------------------------------------

def draft(d: int, L: int, gamma: int, N: int, incoming: Sequence[Path], incoming_sp: np.ndarray,
          draft_rows: RowsFn, trie, relaxed: bool, rng: Optional[Philox]) -> Tree:
    g = min(gamma, L - d)
    prev, prev_sq = list(incoming), np.asarray(incoming_sp, dtype=F32)
    levels, levels_sq = [], []
    for j in range(1, g + 1):
        C = expand(prev, prev_sq, draft_rows(prev), trie)
        if relaxed:
            keys = (C.score + rng.gumbel(STREAM_DRAFT, d + j, C.index)).astype(F32)
            sel = rank_order(keys, C.index)[:N]
        else:
            sel = topk(C, N)
        prev = child_paths(prev, C, sel)
        prev_sq = C.score[sel]
        levels.append(prev)
        levels_sq.append(prev_sq)
    return Tree(d, list(incoming), np.asarray(incoming_sp, dtype=F32), levels, levels_sq)


# ------------------------------------------------------------------------------------------------
# strict top-K verification (Alg. 1)
# ------------------------------------------------------------------------------------------------

def strict_verify(tree: Tree, L: int, K: int, target_rows: RowsFn, trie) -> StepResult:
    d, g = tree.d, len(tree.levels)
    rows = _guard(target_rows, forwarded_paths(tree, L))
    yp, yp_sp = list(tree.incoming), np.asarray(tree.incoming_sp, dtype=F32)
    for j in range(1, g + 1):
        C = expand(yp, yp_sp, rows(yp), trie)
        sel = topk(C, K)
        nxt, nxt_sp = child_paths(yp, C, sel), C.score[sel]
        if not set(nxt) <= set(tree.levels[j - 1]):
            return StepResult(j - 1, j, nxt, nxt_sp)
        yp, yp_sp = nxt, nxt_sp
    if d + g < L:
        C = expand(yp, yp_sp, rows(yp), trie)
        sel = topk(C, K)
        return StepResult(g, g + 1, child_paths(yp, C, sel), C.score[sel])
    return StepResult(g, g, yp, yp_sp)


# ------------------------------------------------------------------------------------------------
# relaxed sampling verification (Sec. 3.2, Alg. 2)
# ------------------------------------------------------------------------------------------------

def _softmax_log(score: np.ndarray) -> np.ndarray:
    return (np.asarray(score, dtype=F32) - logsumexp_f32(score)).astype(F32)


def _rank(paths: List[Path], sp: np.ndarray, idx: np.ndarray) -> Tuple[List[Path], np.ndarray]:
    o = rank_order(sp, idx)
    return [paths[i] for i in o], np.asarray(sp, dtype=F32)[o]


def relaxed_verify(tree: Tree, L: int, K: int, target_rows: RowsFn, draft_rows: RowsFn, trie,
                   rng: Philox) -> StepResult:
    d, g = tree.d, len(tree.levels)
    rows_p = _guard(target_rows, forwarded_paths(tree, L))
    prev = list(tree.incoming)
    prev_sp = np.asarray(tree.incoming_sp, dtype=F32)
    prev_sq = prev_sp.copy()                      # incoming beams carry the target's scores
    for j in range(1, g + 1):
        lvl = d + j
        Cp = expand(prev, prev_sp, rows_p(prev), trie)
        Cq = expand(prev, prev_sq, draft_rows(prev), trie)
        assert np.array_equal(Cp.index, Cq.index)
        logp, logq = _softmax_log(Cp.score), _softmax_log(Cq.score)
        pos_of = {int(x): i for i, x in enumerate(Cp.index)}
        drafted = tree.levels[j - 1]
        dpos = np.array([pos_of[prev.index(p[:-1]) * 256 + p[-1]] for p in drafted], dtype=np.int64)
        u = u_accept(rng.u32(STREAM_ACCEPT, lvl, np.arange(len(drafted))))
        ratio = np.minimum(F32(1.0), np.exp((logp[dpos] - logq[dpos]).astype(F32))).astype(F32)
        acc = np.nonzero(u <= ratio)[0]           # draft order
        if len(acc) >= K:
            if j < g:
                prev, prev_sp, prev_sq = list(drafted), Cp.score[dpos], Cq.score[dpos]
                continue
            if d + g < L:
                # every step passed, item not complete: K draws without replacement from p at the
                # next level (a draw at the wrong level or a top-K fails
                # test_oracle_relaxed_laws.py::test_all_accepted_draws_next_level_from_target)
                C2 = expand(drafted, Cp.score[dpos], rows_p(drafted), trie)
                keys = (C2.score + rng.gumbel(STREAM_RESAMPLE, lvl + 1, C2.index)).astype(F32)
                sel = rank_order(keys, C2.index)[:K]
                out, sp = _rank(child_paths(drafted, C2, sel), C2.score[sel], C2.index[sel])
                return StepResult(g, g + 1, out, sp, len(acc))
            # item complete: K picks uniform over the K-subsets of A (taking the first K of A fails
            # test_oracle_relaxed_laws.py::test_complete_item_picks_uniform_subset_of_accepted)
            keys = rng.u32(STREAM_SUBSET, lvl, acc).astype(np.int64)
            pick = acc[np.lexsort((acc, keys))[:K]]
            out, sp = _rank([drafted[i] for i in pick], Cp.score[dpos[pick]], Cp.index[dpos[pick]])
            return StepResult(g, g, out, sp, len(acc))
        # step rejected: keep A, resample K - |A| from norm(max(0, p - q)) with p' = 0 on A
        # (drawing from p or q instead, or letting A be drawn again, fails
        # test_oracle_relaxed_laws.py::test_rejected_step_resamples_from_residual)
        p = np.exp(logp).astype(F32)
        q = np.exp(logq).astype(F32)
        pr = np.maximum(F32(0.0), (p - q).astype(F32))
        inA = np.zeros(len(Cp), dtype=bool)
        inA[dpos[acc]] = True
        elig = np.nonzero(~inA)[0]
        G = rng.gumbel(STREAM_RESAMPLE, lvl, Cp.index[elig])
        has = pr[elig] > 0
        with np.errstate(divide="ignore"):
            key = np.where(has, np.log(np.where(has, pr[elig], F32(1.0))).astype(F32), logp[elig]).astype(F32)
        key = (key + G).astype(F32)
        o = np.lexsort((Cp.index[elig], -key.astype(np.float64), ~has))
        chosen = elig[o[:K - len(acc)]]
        allpos = np.concatenate([dpos[acc], chosen])
        paths = child_paths(prev, Cp, allpos)
        out, sp = _rank(paths, Cp.score[allpos], Cp.index[allpos])
        return StepResult(j - 1, j, out, sp, len(acc))
    raise AssertionError("unreachable: the loop always returns")


# ------------------------------------------------------------------------------------------------
# the decoding loops
# ------------------------------------------------------------------------------------------------

@dataclasses.dataclass
class DecodeStats:
    accepted_steps: int = 0
    verify_calls: int = 0
    tree_tokens: int = 0
    steps: List[Tuple[int, int, int, int]] = dataclasses.field(default_factory=list)  # (d, a, advance, T)


def sd_decode(target_rows: RowsFn, draft_rows: RowsFn, trie, K: int, N: int, gamma: int, mode: str,
              seed: int = 0, user: int = 0, L: int = 4):
    """Speculative beam decoding of one user's recommendation list.

    Returns (K item paths ranked, fp32 scores, DecodeStats)."""
    assert mode in ("strict", "relaxed")
    d, beams, sp, step = 0, [()], np.zeros(1, dtype=F32), 0
    st = DecodeStats()
    while d < L:
        rng = Philox(seed, step, user)
        tree = draft(d, L, gamma, N, beams, sp, draft_rows, trie, mode == "relaxed", rng)
        T = tree_tokens(tree, L)
        if mode == "strict":
            r = strict_verify(tree, L, K, target_rows, trie)
        else:
            r = relaxed_verify(tree, L, K, target_rows, draft_rows, trie, rng)
        st.accepted_steps += r.a
        st.verify_calls += 1
        st.tree_tokens += T
        st.steps.append((d, r.a, r.advance, T))
        beams, sp = r.paths, r.scores
        d += r.advance
        step += 1
    return beams, sp, st


def plain_beam_search(target_rows: RowsFn, trie, K: int, L: int = 4, sample: bool = False, seed: int = 0,
                      user: int = 0, full_rows: Optional[RowsFn] = None):
    """Target-only constrained beam search (top-K), or sampling beam search at temperature 1.

    Sampling draws level l's K beams without replacement (Gumbel keys) from the Philox stream 3
    counter with sd_step = l - 1, i.e. the number of steps taken before, as in the SD loop.
    ``full_rows`` (the whole-vocabulary logit rows of the beams) selects FULL normalisation (O4):
    each token's log-prob is normalised over the whole vocabulary, then masked to the trie."""
    beams, sp = [()], np.zeros(1, dtype=F32)
    for lvl in range(1, L + 1):
        C = expand(beams, sp, target_rows(beams), trie, None if full_rows is None else full_rows(beams))
        if sample:
            keys = (C.score + Philox(seed, lvl - 1, user).gumbel(STREAM_RESAMPLE, lvl, C.index)).astype(F32)
            sel = rank_order(keys, C.index)[:K]
            sel = sel[rank_order(C.score[sel], C.index[sel])]
        else:
            sel = topk(C, K)
        beams, sp = child_paths(beams, C, sel), C.score[sel]
    return beams, sp
