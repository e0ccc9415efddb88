"""Output laws of the oracle's relaxed verification with K > 1 (Sec. 3.2, App. A.1, Alg. 2),
pinned against exact enumeration on small candidate sets.

Each test fixes a tiny trie, the target / draft logit rows and a drafted level, runs
``oracle.sd.relaxed_verify`` over 12 000 Philox seeds, and compares the empirical law of the
output with the law computed here by enumerating every acceptance set and every ordered sequence
of draws without replacement (fp64):

* rejected step (|A| < K): the output is A plus K - |A| sequential draws without replacement from
  p' = norm(max(0, p - q)) over the candidates outside A (p on the rest once p' has no mass left);
* every step accepted and the item not complete (d + gamma' < L): K draws without replacement from
  p at the next level, over the extensions of the drafted beams;
* every step accepted and the item complete: K picks uniform over the K-subsets of A.

Each law gets a chi-square test over the output sets plus 4-sigma bounds on every candidate's
inclusion frequency.  A plausible slip in any branch (drawing from p or q instead of p', drawing
at the wrong level, taking the top-K instead of sampling, taking the first K of A) moves some
frequency by tens of sigma.
"""
import itertools
from collections import Counter

import numpy as np
import pytest
from scipy import stats

from oracle.sd import Philox, Tree, relaxed_verify
from oracle.trie import Trie

SEEDS = 12000


def _rows(table):
    """Logit rows from a {path: {code: logit}} table (unlisted codes are -30, never valid)."""
    def f(paths):
        out = []
        for p in paths:
            r = np.full(256, -30.0, np.float32)
            for c, v in table.get(tuple(p), {}).items():
                r[c] = v
            out.append(r)
        return out
    return f


def _softmax(v):
    v = np.asarray(v, np.float64)
    e = np.exp(v - v.max())
    return e / e.sum()


def _ordered_draws(weights, avail, m, fallback=None):
    """{tuple of drawn keys: probability} for m sequential draws without replacement from `avail`,
    each proportional to `weights` among the remaining candidates with positive weight, and, once
    none is left, proportional to `fallback`."""
    out = {}

    def rec(rem, seq, pr):
        if len(seq) == m:
            out[tuple(seq)] = out.get(tuple(seq), 0.0) + pr
            return
        pos = [c for c in rem if weights[c] > 0]
        use, w = (pos, weights) if pos else (list(rem), fallback)
        tot = sum(w[c] for c in use)
        for c in use:
            rec([x for x in rem if x != c], seq + [c], pr * w[c] / tot)
    rec(list(avail), [], 1.0)
    return out


def _check_law(emitted, exact, universe):
    """chi-square over output sets and 4-sigma inclusion bounds against the exact law."""
    n = len(emitted)
    assert n > 2000, n
    cnt = Counter(emitted)
    assert set(cnt) <= set(exact), set(cnt) - set(exact)
    keys = [k for k in exact if exact[k] * n >= 5]
    rest = 1.0 - sum(exact[k] for k in keys)
    obs = [cnt[k] for k in keys] + ([n - sum(cnt[k] for k in keys)] if rest * n >= 5 else [])
    exp_ = [exact[k] * n for k in keys] + ([rest * n] if rest * n >= 5 else [])
    scale = n / sum(exp_)
    chi = stats.chisquare(obs, [e * scale for e in exp_])
    assert chi.pvalue > 1e-4, (chi, obs, exp_)
    for c in universe:
        pe = sum(p for k, p in exact.items() if c in k)
        f = sum(v for k, v in cnt.items() if c in k) / n
        sig = np.sqrt(max(pe * (1 - pe), 1e-12) / n)
        assert abs(f - pe) <= 4 * sig + 1e-9, (c, f, pe, sig)


def test_rejected_step_resamples_from_residual():
    """|A| < K: A plus K - |A| draws without replacement from norm(max(0, p - q)) outside A."""
    # the drafted codes have q > p (each accepted with probability p / q < 1); the three undrafted
    # ones have p > q, with residual proportions (0.58, 0.29, 0.13) unlike p's (0.49, 0.40, 0.11)
    codes = [10, 20, 30, 40, 50, 60]
    items = np.array([[c, 0, 0, 0] for c in codes], np.int32)
    trie = Trie(items)
    lt = {10: 1.0, 20: 0.8, 30: 0.2, 40: 0.5, 50: 0.0, 60: -0.5}
    ld = {10: 0.0, 20: 0.5, 30: 1.0, 40: 1.3, 50: 1.2, 60: -1.5}
    tgt = _rows({(): lt, **{(c,): {0: 0.0} for c in codes}})
    drf = _rows({(): ld})
    drafted = [40, 30, 50]               # draft order
    K = 3
    tree = Tree(0, [()], np.zeros(1, np.float32), [[(c,) for c in drafted]], [np.zeros(3, np.float32)])
    p = dict(zip(codes, _softmax([lt[c] for c in codes])))
    q = dict(zip(codes, _softmax([ld[c] for c in codes])))
    r = {c: min(1.0, p[c] / q[c]) for c in drafted}
    pr = {c: max(0.0, p[c] - q[c]) for c in codes}
    exact = {}
    for mask in itertools.product([0, 1], repeat=len(drafted)):
        A = [c for c, m in zip(drafted, mask) if m]
        if len(A) >= K:
            continue
        pa = np.prod([r[c] if m else 1 - r[c] for c, m in zip(drafted, mask)])
        for seq, ps in _ordered_draws(pr, [c for c in codes if c not in A], K - len(A), p).items():
            key = frozenset(A) | frozenset(seq)
            exact[key] = exact.get(key, 0.0) + pa * ps
    p_rej = sum(exact.values())
    exact = {k: v / p_rej for k, v in exact.items()}
    emitted = []
    for s in range(SEEDS):
        res = relaxed_verify(tree, 4, K, tgt, drf, trie, Philox(s, 0, 0))
        if res.a == 0:
            out = [pth[0] for pth in res.paths]
            assert len(out) == K == len(set(out)) and res.advance == 1
            emitted.append(frozenset(out))
    assert abs(len(emitted) / SEEDS - p_rej) < 4 * np.sqrt(p_rej * (1 - p_rej) / SEEDS)
    _check_law(emitted, exact, codes)


def test_all_accepted_draws_next_level_from_target():
    """Every drafted beam accepted (p = q) and the item not complete: K draws without replacement
    from p over the extensions of the drafted beams (next level)."""
    kids = {10: [1, 2, 3], 20: [4, 5, 6], 30: [7]}
    items = np.array([[a, b, 0, 0] for a, bs in kids.items() for b in bs], np.int32)
    trie = Trie(items)
    l1 = {10: 0.3, 20: 0.0, 30: -0.2}
    l2 = {(10,): {1: 1.0, 2: 0.0, 3: -1.0}, (20,): {4: 0.5, 5: 0.4, 6: -0.8}, (30,): {7: 0.0}}
    rows = _rows({(): l1, **l2})
    drafted = [20, 10]
    K = 2
    tree = Tree(0, [()], np.zeros(1, np.float32), [[(c,) for c in drafted]], [np.zeros(2, np.float32)])
    # sequence scores of the next level: log p1(a) + log p2(b | a), p1 over the three first codes
    p1 = dict(zip(l1, _softmax(list(l1.values()))))
    score = {}
    for a in drafted:
        p2 = _softmax(list(l2[(a,)].values()))
        for b, pb in zip(l2[(a,)], p2):
            score[(a, b)] = np.log(p1[a]) + np.log(pb)
    w = dict(zip(score, _softmax(list(score.values()))))
    exact = {}
    for seq, ps in _ordered_draws(w, list(score), K).items():
        exact[frozenset(seq)] = exact.get(frozenset(seq), 0.0) + ps
    emitted = []
    for s in range(SEEDS):
        res = relaxed_verify(tree, 4, K, rows, rows, trie, Philox(s, 0, 0))
        assert res.a == 1 and res.advance == 2
        out = [tuple(pth) for pth in res.paths]
        assert len(out) == K == len(set(out)) and all(len(o) == 2 for o in out)
        sc = res.scores.astype(np.float64)
        assert np.all(np.diff(sc) <= 0)                              # ranked by target score
        emitted.append(frozenset(out))
    _check_law(emitted, exact, list(score))


def test_complete_item_picks_uniform_subset_of_accepted():
    """Every drafted beam accepted (p = q) at the last level: K picks uniform over the K-subsets
    of A."""
    items = np.array([[1, 1, 1, x] for x in (1, 2, 3)] + [[2, 2, 2, y] for y in (4, 5)], np.int32)
    trie = Trie(items)
    rows = _rows({(1, 1, 1): {1: 0.9, 2: 0.1, 3: -0.4}, (2, 2, 2): {4: 0.2, 5: -0.3}})
    incoming = [(1, 1, 1), (2, 2, 2)]
    drafted = [(2, 2, 2, 4), (1, 1, 1, 2), (1, 1, 1, 1), (2, 2, 2, 5)]
    K = 2
    tree = Tree(3, incoming, np.array([-0.5, -0.9], np.float32), [drafted], [np.zeros(4, np.float32)])
    exact = {frozenset(c): 1.0 / 6.0 for c in itertools.combinations(drafted, K)}
    emitted = []
    for s in range(SEEDS):
        res = relaxed_verify(tree, 4, K, rows, rows, trie, Philox(s, 1, 0))
        assert res.a == 1 and res.advance == 1
        out = [tuple(pth) for pth in res.paths]
        assert len(out) == K == len(set(out))
        emitted.append(frozenset(out))
    _check_law(emitted, exact, drafted)
