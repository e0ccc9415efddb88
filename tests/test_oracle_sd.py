"""Pins for oracle.sd: losslessness of strict verification (Alg. 1), the strict acceptance
definition (Sec. 3.1), and the statistical laws of relaxed sampling verification (Eq. 4,
speculative-sampling output law, Gumbel sampling without replacement)."""
import itertools

import numpy as np
import pytest

import synth
from oracle.beam import expand, topk
from oracle.model import Model, PathEvaluator
from oracle.philox import draw_u32, gumbel
from oracle.sd import (Philox, Tree, draft, plain_beam_search, relaxed_verify, sd_decode, strict_verify,
                       tree_tokens)
from oracle.trie import Trie


def hashed_rows(seed, std=3.0, sign=1.0):
    def f(paths):
        return [(sign * np.random.default_rng([seed, len(p), *p]).standard_normal(256) * std).astype(np.float32)
                for p in paths]
    return f


def _world(n_items=1000, dist="uniform", seed=1):
    return Trie(synth.make_items(n_items, dist, 1.1, seed))


@pytest.mark.parametrize("K,N,gamma", [(5, 10, 2), (10, 40, 4), (1, 1, 4), (3, 3, 1), (20, 80, 3)])
@pytest.mark.parametrize("draft_kind", ["random", "same", "adversarial"])
def test_strict_sd_is_lossless(K, N, gamma, draft_kind):
    """Strict top-K verification returns exactly plain target beam search (lossless)."""
    trie = _world(3000, "zipf", 7)
    for user in range(3):
        tgt = hashed_rows(1000 + user)
        drf = {"random": hashed_rows(2000 + user), "same": tgt,
               "adversarial": hashed_rows(1000 + user, sign=-1.0)}[draft_kind]
        ref, ref_sp = plain_beam_search(tgt, trie, K)
        out, sp, st = sd_decode(tgt, drf, trie, K, N, gamma, "strict", user=user)
        assert out == ref
        np.testing.assert_array_equal(sp, ref_sp)
        assert st.verify_calls >= 1 and sum(s[2] for s in st.steps) == 4


def test_strict_same_draft_accepts_first_step_and_full_width_accepts_all():
    trie = _world(500, "uniform", 3)
    tgt = hashed_rows(5)
    _, _, st = sd_decode(tgt, tgt, trie, 4, 8, 4, "strict")
    assert all(a >= 1 for (_, a, _, _) in st.steps)
    _, _, st = sd_decode(tgt, tgt, trie, 4, 10 ** 6, 4, "strict")
    assert st.verify_calls == 1 and st.accepted_steps == 4


def test_strict_adversarial_draft_rejects_first_step():
    trie = _world(3000, "uniform", 4)
    tgt = hashed_rows(11)
    adv = hashed_rows(11, sign=-1.0)
    K = 5
    _, _, st = sd_decode(tgt, adv, trie, K, K, 4, "strict")
    assert st.steps[0][1] == 0        # ~250 first codes: draft's worst K never meet target's best K


def test_strict_accept_matches_acceptance_rate_definition():
    """Sec. 3.1: step accepted iff some K-subset of the drafted sequences all have target
    probability >= p(y_K), y_K the target's K-th best (no exact ties here)."""
    trie = _world(2000, "zipf", 9)
    rng = np.random.default_rng(0)
    for trial in range(40):
        K, N = int(rng.integers(1, 6)), int(rng.integers(1, 12))
        tgt, drf = hashed_rows(trial), hashed_rows(500 + trial, std=float(rng.uniform(0.5, 4)))
        tree = draft(0, 4, 1, N, [()], np.zeros(1, np.float32), drf, trie, False, None)
        r = strict_verify(tree, 4, K, tgt, trie)
        C = expand([()], [0.0], tgt([()]), trie)
        sK = C.score[topk(C, K)][-1]
        drafted = set(tree.levels[0])
        n_ok = sum(1 for i in range(len(C)) if (int(C.code[i]),) in drafted and C.score[i] >= sK)
        assert (r.a >= 1) == (n_ok >= K)


def test_tree_token_count():
    trie = _world()
    tgt = hashed_rows(1)
    tree = draft(0, 4, 4, 10, [()], np.zeros(1, np.float32), tgt, trie, False, None)
    assert tree_tokens(tree, 4) == sum(len(l) for l in tree.levels[:3])
    inc = tree.levels[0][:5]
    t2 = draft(1, 4, 4, 10, inc, np.zeros(5, np.float32), tgt, trie, False, None)
    assert len(t2.levels) == 3 and tree_tokens(t2, 4) == 5 + sum(len(l) for l in t2.levels[:2])


def test_strict_sd_lossless_on_tiny_model():
    """Same as above with the real decoder (tiny workload): tree-node logits come from the
    causal forward of prompt + path; the guard asserts verification only reads tree nodes."""
    w = synth.workload("tiny")
    items = synth.make_items(w.n_items, w.code_dist, w.zipf_a, w.seed)
    trie = Trie(items)
    prompt = synth.make_prompts(1, w.prompt_len, w.target.vocab, w.seed)[0]
    tm = Model(w.target, synth.model_weights(w.target, w.seed, "target"), w.code_base)
    dm = Model(w.draft, synth.model_weights(w.draft, w.seed, "draft"), w.code_base)
    te, de = PathEvaluator(tm, prompt), PathEvaluator(dm, prompt)

    def rows(ev):
        def f(paths):
            return [ev.logits([p])[0][256 * len(p):256 * (len(p) + 1)].astype(np.float32) for p in paths]
        return f
    ref, ref_sp = plain_beam_search(rows(te), trie, w.K)
    out, sp, st = sd_decode(rows(te), rows(de), trie, w.K, w.N, w.gamma, "strict")
    assert out == ref and np.array_equal(sp, ref_sp)
    assert all(trie.is_item(p) for p in out)


# ----------------------------------------------------------------------------------------------
# relaxed sampling verification
# ----------------------------------------------------------------------------------------------

def _last_level_case(trie_items, seed_p, seed_q, temp_q=1.0):
    trie = Trie(trie_items)
    pre = tuple(int(c) for c in trie_items[0, :3])
    tgt = hashed_rows(seed_p, std=1.0)
    drf = hashed_rows(seed_q, std=temp_q)
    return trie, pre, tgt, drf


def test_relaxed_single_draw_acceptance_rate_is_one_minus_tvd():
    """K = N = 1 at the last level: acceptance frequency -> sum_y min(p, q) = 1 - TVD (Eq. 4),
    and the output follows p (speculative sampling)."""
    items = np.array([[1, 2, 3, c] for c in (0, 5, 9, 11, 40, 77)], dtype=np.int32)
    trie, pre, tgt, drf = _last_level_case(items, 3, 4, 1.5)
    C = expand([pre], [0.0], tgt([pre]), trie)
    p = np.exp(C.score.astype(np.float64)); p /= p.sum()
    Cq = expand([pre], [0.0], drf([pre]), trie)
    q = np.exp(Cq.score.astype(np.float64)); q /= q.sum()
    trials = 20000
    acc = 0
    counts = np.zeros(len(C))
    for t in range(trials):
        rng = Philox(0, 0, t)
        tree = draft(3, 4, 1, 1, [pre], np.zeros(1, np.float32), drf, trie, True, rng)
        r = relaxed_verify(tree, 4, 1, tgt, drf, trie, rng)
        acc += r.n_accepted_last
        counts[np.searchsorted(C.code, r.paths[0][-1])] += 1
    b = np.minimum(p, q).sum()
    assert abs(acc / trials - b) < 4 * np.sqrt(b * (1 - b) / trials)
    e = p * trials
    chi2 = np.sum((counts - e) ** 2 / e)
    assert chi2 < 5 + 6 * np.sqrt(10)
    assert abs(b - (1 - 0.5 * np.abs(p - q).sum())) < 1e-12


def test_relaxed_p_equals_q_accepts_every_draft():
    trie = _world(2000, "zipf", 5)
    tgt = hashed_rows(21)
    for user in range(3):
        out, sp, st = sd_decode(tgt, tgt, trie, 3, 8, 4, "relaxed", seed=9, user=user)
        assert st.verify_calls == 1 and st.accepted_steps == 4
        assert len(set(out)) == 3 and all(trie.is_item(p) for p in out)


def test_relaxed_outputs_are_valid_distinct_and_ranked():
    trie = _world(3000, "zipf", 6)
    for user in range(4):
        tgt, drf = hashed_rows(31 + user), hashed_rows(61 + user)
        out, sp, st = sd_decode(tgt, drf, trie, 10, 40, 4, "relaxed", seed=123, user=user)
        assert len(out) == 10 and len(set(out)) == 10
        assert all(trie.is_item(p) for p in out)
        assert np.all(np.diff(sp.astype(np.float64)) <= 0)
        assert sum(s[2] for s in st.steps) == 4


def test_gumbel_keys_sample_without_replacement_law():
    """Top-2 of log w + Gumbel has the law of two sequential draws without replacement:
    P(i then j) = w_i w_j / (1 - w_i)."""
    w = np.array([0.4, 0.3, 0.2, 0.1])
    trials = 40000
    g = gumbel(draw_u32(5, 0, 1, 0, 0, np.arange(trials * 4))).reshape(trials, 4).astype(np.float64)
    keys = np.log(w)[None, :] + g
    top2 = np.argsort(-keys, axis=1)[:, :2]
    counts = {}
    for a, b in top2:
        counts[(a, b)] = counts.get((a, b), 0) + 1
    chi2 = 0.0
    for i, j in itertools.permutations(range(4), 2):
        e = trials * w[i] * w[j] / (1 - w[i])
        chi2 += (counts.get((i, j), 0) - e) ** 2 / e
    assert chi2 < 11 + 6 * np.sqrt(22)


def test_relaxed_multi_draw_step_acceptance_loose():
    """Loose sanity of beta ~ prod_K b (with-replacement approximation, App. A.2.1) for a
    large candidate set and small K: the empirical step-acceptance rate is within 0.1."""
    items = np.array([[1, 2, 3, c] for c in range(0, 256, 2)], dtype=np.int32)
    trie, pre, tgt, drf = _last_level_case(items, 7, 8, 1.0)
    C = expand([pre], [0.0], tgt([pre]), trie)
    p = np.exp(C.score.astype(np.float64)); p /= p.sum()
    Cq = expand([pre], [0.0], drf([pre]), trie)
    q = np.exp(Cq.score.astype(np.float64)); q /= q.sum()
    b = np.minimum(p, q).sum()
    K, trials, ok = 2, 3000, 0
    for t in range(trials):
        rng = Philox(1, 0, t)
        tree = draft(3, 4, 1, K, [pre], np.zeros(1, np.float32), drf, trie, True, rng)
        r = relaxed_verify(tree, 4, K, tgt, drf, trie, rng)
        ok += r.a == 1
    assert abs(ok / trials - b ** K) < 0.1
