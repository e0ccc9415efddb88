"""Full-size checks at the 7B-shape workload the bench times (32 layers, d 4096, one user, P = 512,
K = 10, N = 40, gamma = 4, 50 000 Zipf items), in the bench's launch configuration.

The oracle cannot run a 32-layer 7B forward in test time, so these check properties that hold at
any size (the sampled 7B-shape node logits against the oracle are in test_gpu_engine.py, cut to
one layer):

* strict speculative decoding is lossless: its recommendation list equals the plain target beam
  search, bit for bit (same logits, same ranking);
* the persistent forward and the one-kernel-per-op forward give the same tree-node logits, bit for
  bit, on the verification call;
* relaxed speculative decoding returns K distinct valid items ranked by target score, also for the
  16-user workload (ragged 256-1 024-token histories, K = 20, N = 80), reproducibly per seed.
"""
import numpy as np
import pytest
import torch

import synth
from oracle.trie import Trie

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ats():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2410_05165_gb300 as m
    return m


@pytest.fixture(scope="module")
def world(ats):
    w = synth.workload("7b")

    def to_dev(spec, role):
        return {n: torch.from_numpy(a).to(device="cuda", dtype=torch.bfloat16)
                for n, a in synth.iter_model_tensors(spec, w.seed, role)}
    tw, dw = to_dev(w.target, "target"), to_dev(w.draft, "draft")
    items = synth.make_items(w.n_items, w.code_dist, w.zipf_a, w.seed)
    prompt = synth.make_prompts(1, w.prompt_len, w.target.vocab, w.seed)[0]
    toks = torch.from_numpy(prompt.astype(np.int32)).cuda()
    yield w, tw, dw, items, prompt, toks
    del tw, dw
    torch.cuda.empty_cache()


def _ctx(ats, world):
    w, tw, dw, items, prompt, _ = world
    return ats.Context(w.target, tw, w.draft, dw, items, w.code_base, max_users=1, max_prompt=len(prompt),
                       max_K=w.K, max_N=w.N, max_gamma=w.gamma)


def test_7b_strict_sd_is_lossless(ats, world):
    w, _, _, items, prompt, toks = world
    ctx = _ctx(ats, world)
    o = ats.opts(w.K, w.N, w.gamma, w.philox_seed)
    off = [0, len(prompt)]
    sd_items, sd_sc, stats = ctx.beam_search(toks, off, o, ats.SD_STRICT)
    pl_items, pl_sc, _ = ctx.beam_search(toks, off, o, ats.PLAIN_TOPK)
    np.testing.assert_array_equal(sd_items.cpu().numpy(), pl_items.cpu().numpy())
    np.testing.assert_array_equal(sd_sc.cpu().numpy(), pl_sc.cpu().numpy())
    assert stats[0, 1] >= 1 and stats[0, 0] >= 1
    ctx.close()


def test_7b_persistent_forward_equals_per_op(ats, world, monkeypatch):
    w, _, _, items, prompt, toks = world
    o = ats.opts(w.K, w.N, w.gamma, w.philox_seed)
    outs = []
    for mode in ("per_op", "persistent"):
        monkeypatch.setenv("ATSPEED_FORWARD", mode)
        ctx = _ctx(ats, world)
        ctx.prefill(toks, [0, len(prompt)])
        ctx.begin_step(o)
        for _ in range(w.gamma):
            ctx.draft_step(o, ats.STRICT)
        ctx.verify(o, ats.STRICT)
        _, _, slots_in, slots_lvl = ctx.tree_shape()
        # the root (prefill row) and a sample of the drafted nodes of levels 1-3 (the forwarded ones)
        rng = np.random.default_rng(3)
        slots = [0] + sorted(set((slots_in + rng.integers(0, 3 * slots_lvl, size=24)).tolist()))
        outs.append(np.stack([ctx.node_logits(0, 0, s) for s in slots]))
        ctx.close()
    np.testing.assert_array_equal(outs[0], outs[1])


def test_7b_relaxed_outputs_are_valid_distinct_ranked(ats, world):
    w, _, _, items, prompt, toks = world
    ctx = _ctx(ats, world)
    o = ats.opts(w.K, w.N, w.gamma, w.philox_seed)
    got, sc, stats = ctx.beam_search(toks, [0, len(prompt)], o, ats.SD_RELAXED)
    got = [tuple(int(c) for c in r) for r in got[0].cpu().numpy()]
    sc = sc[0].cpu().numpy()
    trie = Trie(items)
    valid = {tuple(int(c) for c in it) for it in items}
    assert len(got) == w.K and len(set(got)) == w.K
    assert all(g in valid for g in got)
    assert np.all(np.diff(sc) <= 0)
    assert stats[0, 1] >= 1
    del trie
    ctx.close()


@pytest.mark.parametrize("B,K,gamma,N,full", [(4, 5, 2, 10, False), (1, 20, 3, 80, False), (4, 1, 4, 4, False),
                                               (1, 10, 4, 40, True)])
def test_7b_sweep_points_strict_lossless(ats, world, B, K, gamma, N, full):
    """Points of the verification-call sweep (batch x K x gamma x N, 512-token histories), and the
    bench point under FULL normalisation: strict speculative decoding returns the plain target beam
    search's lists bit for bit, for every user."""
    w, _, _, items, _, _ = world
    prompts = synth.make_prompts(B, w.prompt_len, w.target.vocab, w.seed + 7)
    P = [len(p) for p in prompts]
    ctx = ats.Context(w.target, world[1], w.draft, world[2], items, w.code_base, max_users=B, max_prompt=max(P),
                      max_K=20, max_N=80, max_gamma=4)
    toks = torch.from_numpy(np.concatenate(prompts).astype(np.int32)).cuda()
    off = np.concatenate([[0], np.cumsum(P)]).astype(np.int32).tolist()
    o = ats.opts(K, N, gamma, w.philox_seed, norm=ats.NORM_FULL if full else ats.NORM_MASKED)
    sd_items, sd_sc, stats = ctx.beam_search(toks, off, o, ats.SD_STRICT)
    pl_items, pl_sc, _ = ctx.beam_search(toks, off, o, ats.PLAIN_TOPK)
    np.testing.assert_array_equal(sd_items.cpu().numpy(), pl_items.cpu().numpy())
    np.testing.assert_array_equal(sd_sc.cpu().numpy(), pl_sc.cpu().numpy())
    assert sd_items.shape == (B, K, 4)
    ctx.close()


def test_7b_b16_relaxed_config_valid_and_reproducible(ats, world):
    """The 16-user workload the bench's second line times (histories of 256 to 1 024 tokens, 200 000
    Zipf items, K = 20, N = 80, gamma = 4, relaxed verification with per-user Philox streams):
    every user gets K distinct valid items ranked by target score, and a second decode with the same
    seed reproduces every list bit for bit; with another seed some list changes."""
    w7 = synth.workload("7b_b16")
    items = synth.make_items(w7.n_items, w7.code_dist, w7.zipf_a, w7.seed)
    prompts = synth.make_prompts(w7.n_users, w7.prompt_len, w7.target.vocab, w7.seed)
    P = [len(p) for p in prompts]
    assert min(P) >= 256 and max(P) <= 1024 and len(set(P)) > 1   # ragged histories
    ctx = ats.Context(w7.target, world[1], w7.draft, world[2], items, w7.code_base, max_users=w7.n_users,
                      max_prompt=max(P), max_K=w7.K, max_N=w7.N, max_gamma=w7.gamma)
    toks = torch.from_numpy(np.concatenate(prompts).astype(np.int32)).cuda()
    off = np.concatenate([[0], np.cumsum(P)]).astype(np.int32).tolist()
    o = ats.opts(w7.K, w7.N, w7.gamma, w7.philox_seed)
    a_items, a_sc, stats = ctx.beam_search(toks, off, o, ats.SD_RELAXED)
    b_items, b_sc, _ = ctx.beam_search(toks, off, o, ats.SD_RELAXED)
    c_items, _, _ = ctx.beam_search(toks, off, ats.opts(w7.K, w7.N, w7.gamma, w7.philox_seed + 1), ats.SD_RELAXED)
    ctx.close()
    np.testing.assert_array_equal(a_items.cpu().numpy(), b_items.cpu().numpy())
    np.testing.assert_array_equal(a_sc.cpu().numpy(), b_sc.cpu().numpy())
    assert not np.array_equal(a_items.cpu().numpy(), c_items.cpu().numpy())
    valid = {tuple(int(c) for c in it) for it in items}
    for u in range(w7.n_users):
        got = [tuple(int(c) for c in r) for r in a_items[u].cpu().numpy()]
        assert len(set(got)) == w7.K and all(g in valid for g in got), u
        assert np.all(np.diff(a_sc[u].cpu().numpy()) <= 0), u
    assert np.all(stats[:, 1] >= 1)
