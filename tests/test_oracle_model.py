"""Pins for oracle.model: the paper's worked tree-mask example, the flattened-tree
formulation against per-beam causal forwards, closed forms and library attention."""
import os

import numpy as np
import torch

import synth
from oracle.model import (CODES, Model, PathEvaluator, _attend, causal_forward, forward_tree_flat,
                          path_tokens, tree_mask)

GOLD = os.path.join(os.path.dirname(__file__), "golden")

SPEC = synth.ModelSpec(2, 64, 4, 128, 1024)


def _model(seed=11, rnd=True, spec=SPEC):
    return Model(spec, synth.model_weights(spec, seed, "target"), 0, round_bf16=rnd)


def test_table6_mask_rows():
    # App. A.3.1 Table 6: flattened "a1 a2 b1 b2 c1 c2"; parents b1->a1, b2->a2, c1->b1, c2->b1
    parents = [-1, -1, 0, 1, 2, 2]
    names, rows = [], []
    with open(os.path.join(GOLD, "table6_tree_mask.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                t = line.split()
                names.append(t[0])
                rows.append([int(x) for x in t[1:]])
    assert names == ["a1", "a2", "b1", "b2", "c1", "c2"]
    np.testing.assert_array_equal(tree_mask(parents).astype(int), np.array(rows))


def test_attend_matches_torch_sdpa():
    rng = np.random.default_rng(3)
    q = rng.standard_normal((7, 3, 16))
    k = rng.standard_normal((7, 3, 16))
    v = rng.standard_normal((7, 3, 16))
    causal = np.tril(np.ones((7, 7), dtype=bool))
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(q).transpose(0, 1), torch.from_numpy(k).transpose(0, 1),
        torch.from_numpy(v).transpose(0, 1), is_causal=True).transpose(0, 1).numpy()
    np.testing.assert_allclose(_attend(q, k, v, causal), ref, rtol=1e-10, atol=1e-12)


def test_flattened_tree_equals_per_beam_forwards():
    """Tree attention (one pass over the flattened beams with the App. A.3.1 mask) must give
    every drafted beam exactly the logits of its own causal forward (Sec. 3.3)."""
    m = _model()
    prompt = [5, 900, 17, 333, 64, 2, 1000, 7]
    # Table 6 shape: two steps of beam size 2 then two children of b1
    codes = [3, 9, 200, 41, 7, 8]
    parents = [-1, -1, 0, 1, 2, 2]
    depths = [1, 1, 2, 2, 3, 3]
    flat = forward_tree_flat(m, prompt, codes, parents, depths)
    ev = PathEvaluator(m, prompt)
    paths = []
    for i in range(6):
        p, j = [], i
        while j >= 0:
            p.append(codes[j]); j = parents[j]
        paths.append(tuple(reversed(p)))
    per_path = ev.logits(paths)
    for i in range(6):
        np.testing.assert_allclose(flat[i], per_path[i], rtol=1e-9, atol=1e-9)
        whole = causal_forward(m, list(prompt) + path_tokens(paths[i], 0))[0][-1]
        np.testing.assert_allclose(per_path[i], whole, rtol=1e-9, atol=1e-9)


def test_causality():
    m = _model()
    a = causal_forward(m, [1, 2, 3, 4, 5, 6])[0]
    b = causal_forward(m, [1, 2, 3, 4, 99, 600])[0]
    np.testing.assert_array_equal(a[:4], b[:4])
    assert not np.allclose(a[4:], b[4:])


def test_zero_blocks_reduce_to_embedding_head():
    """With W_o = W_down = 0 every layer is the identity on the residual, so the logits are
    the LM head applied to RMSNorm(embedding) (closed form, no rounding)."""
    w = synth.model_weights(SPEC, 4, "target")
    for l in range(SPEC.n_layers):
        w[f"layers.{l}.wo"] = np.zeros_like(w[f"layers.{l}.wo"])
        w[f"layers.{l}.wdown"] = np.zeros_like(w[f"layers.{l}.wdown"])
    m = Model(SPEC, w, 0, round_bf16=False)
    toks = [10, 20, 30]
    lg = causal_forward(m, toks)[0]
    e = w["embed"][toks].astype(np.float64)
    x = e / np.sqrt(np.mean(e * e, axis=1, keepdims=True) + 1e-6) * w["final_norm"]
    np.testing.assert_allclose(lg, x @ w["lm_head"][:4 * CODES].astype(np.float64).T, rtol=1e-12)


def test_single_token_attention_returns_v():
    """One key: softmax is 1, so the attention output equals v (then W_o)."""
    m = _model(rnd=False)
    from oracle.model import _layer_pre_attn
    h = m.W("embed")[[42]].copy()
    q, k, v = _layer_pre_attn(m, 0, h, np.array([0]))
    np.testing.assert_allclose(_attend(q, k, v, None), v, rtol=1e-13)


def test_head_permutation_invariance():
    """Permuting heads consistently in W_q, W_k, W_v and the input columns of W_o leaves the
    output unchanged: catches head-indexing mistakes in the attention layout."""
    w = synth.model_weights(SPEC, 5, "target")
    d, H = SPEC.d_model, SPEC.n_heads
    hd = d // H
    perm = np.array([2, 0, 3, 1])
    rows = np.concatenate([np.arange(h * hd, (h + 1) * hd) for h in perm])
    w2 = dict(w)
    for l in range(SPEC.n_layers):
        qkv = w[f"layers.{l}.wqkv"]
        w2[f"layers.{l}.wqkv"] = np.concatenate([qkv[:d][rows], qkv[d:2 * d][rows], qkv[2 * d:][rows]])
        w2[f"layers.{l}.wo"] = w[f"layers.{l}.wo"][:, rows]
    toks = [3, 1000, 77, 5]
    a = causal_forward(Model(SPEC, w, 0, False), toks)[0]
    b = causal_forward(Model(SPEC, w2, 0, False), toks)[0]
    np.testing.assert_allclose(a, b, rtol=1e-11, atol=1e-11)


def test_unrounded_layer_is_the_textbook_prenorm_block():
    """With the rounding points off, the layer functions (norm scale applied after the projection)
    equal the textbook LLaMA block written with torch's own rms_norm and silu: RMSNorm, then the
    QKV projection and RoPE; residual + O projection, RMSNorm, gate/up, SiLU(gate) * up."""
    from oracle.model import _layer_mlp_act, _layer_pre_attn
    from oracle.numerics import rope
    m = _model(rnd=False)
    sp = SPEC
    d, H, hd, f = sp.d_model, sp.n_heads, sp.head_dim, sp.d_ffn
    rng = np.random.default_rng(5)
    h = rng.standard_normal((6, d)) * 3.0
    pos = np.arange(6) + 4
    th = torch.from_numpy
    for l in range(sp.n_layers):
        x = torch.nn.functional.rms_norm(th(h), (d,), th(m.W(f"layers.{l}.attn_norm")), eps=sp.rms_eps).numpy()
        qkv = x @ m.W(f"layers.{l}.wqkv").T
        q, k, v = _layer_pre_attn(m, l, h, pos)
        np.testing.assert_allclose(q, rope(qkv[:, :d].reshape(-1, H, hd), pos, sp.rope_theta), rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(k, rope(qkv[:, d:2 * d].reshape(-1, H, hd), pos, sp.rope_theta), rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(v, qkv[:, 2 * d:].reshape(-1, H, hd), rtol=1e-10, atol=1e-12)
        o = rng.standard_normal((6, d))
        h2 = h + o @ m.W(f"layers.{l}.wo").T
        x2 = torch.nn.functional.rms_norm(th(h2), (d,), th(m.W(f"layers.{l}.mlp_norm")), eps=sp.rms_eps)
        gu = x2 @ th(m.W(f"layers.{l}.wgate_up")).T
        act = (torch.nn.functional.silu(gu[:, :f]) * gu[:, f:]).numpy()
        h_out, a = _layer_mlp_act(m, l, h, o)
        np.testing.assert_allclose(h_out, h2, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(a, act, rtol=1e-10, atol=1e-12)


def test_rounding_points_are_bf16():
    m = _model()
    from oracle.model import _layer_pre_attn
    from oracle.numerics import bf16
    h = m.W("embed")[[1, 2, 3]].copy()
    q, k, v = _layer_pre_attn(m, 0, h, np.array([0, 1, 2]))
    for t in (q, k, v):
        np.testing.assert_array_equal(t, bf16(t))
