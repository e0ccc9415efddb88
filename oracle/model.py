"""LLaMA-style decoder forward (fp64 with bf16 rounding points), and tree-node logits.

The target model of the paper is LC-Rec on LLaMA-7B (Sec. 4.1); the draft is a
LLaMA-68M.  Both are pre-norm decoders: RMSNorm -> QKV -> RoPE -> causal
attention -> O projection -> residual; RMSNorm -> SiLU-gated MLP -> residual.

bf16 rounding points (both the oracle and the CUDA path round here, ties to
even; everything else is fp64 here and fp32 on the GPU):
  * the embedding row (weights are bf16 already) enters an fp32/fp64 residual;
  * the inputs of the QKV and gate/up projections: RMSNorm(h) = s(h) * (g * h)
    with the per-row scale s(h) = 1 / sqrt(mean(h^2) + eps), and since s(h)
    is one number per token it commutes with the projection:
    W RMSNorm(h) = s(h) * (W (g * h)).  The GEMM input is g * h, rounded to
    bf16; s(h) multiplies the GEMM's output;
  * the final RMSNorm's output (the LM head's input), rounded after the
    whole norm;
  * q and k after RoPE, and v (k and v are stored as bf16 in the KV cache);
  * the attention output o (input of the O projection);
  * the SwiGLU product silu(gate) * up (input of the down projection).
GEMM outputs are added to the residual without rounding; logits are not rounded.

Tree-node logits (Sec. 3.3 "Tree-based Attention", App. A.3.1): the logits of a
drafted node n are by definition the last-position logits of the plain causal
forward of ``prompt + path(n)``, path(n) being the item tokens from depth 1 to
n.  Position of the depth-t token is P + t - 1.  ``PathEvaluator`` evaluates
exactly that, reusing the prompt's rows (which causal attention makes
independent of the path).  ``forward_tree_flat`` is the paper's formulation
(flattened beams + L_f x L_f tree mask) and is pinned against it.
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

from .numerics import bf16, rms_scale, rmsnorm, rope, silu, softmax

L_ITEM = 4
CODES = 256


class Model:
    """Weights (float32 arrays holding bf16 values) plus dimensions.

    ``weights`` maps the names produced by ``synth.model_tensor_names``.
    ``round_bf16=False`` turns every rounding point off (pure fp64 forward).
    """

    def __init__(self, spec, weights: Dict[str, np.ndarray], code_base: int, round_bf16: bool = True):
        self.spec = spec
        self.w = weights
        self.code_base = int(code_base)
        self.rnd = bf16 if round_bf16 else (lambda x: np.asarray(x, dtype=np.float64))
        self._f64: Dict[str, np.ndarray] = {}

    def W(self, name: str) -> np.ndarray:
        a = self._f64.get(name)
        if a is None:
            a = np.asarray(self.w[name], dtype=np.float64)
            self._f64[name] = a
        return a

    def drop_cache(self) -> None:
        self._f64.clear()

    # ---- item-code LM-head rows: code c at level l is token code_base + 256*l + c
    def item_rows(self) -> np.ndarray:
        return self.W("lm_head")[self.code_base:self.code_base + L_ITEM * CODES]


def _layer_pre_attn(m: Model, l: int, h: np.ndarray, pos: np.ndarray):
    sp = m.spec
    H, hd, d = sp.n_heads, sp.head_dim, sp.d_model
    xg = m.rnd(h * m.W(f"layers.{l}.attn_norm"))
    qkv = (xg @ m.W(f"layers.{l}.wqkv").T) * rms_scale(h, sp.rms_eps)
    q = qkv[:, :d].reshape(-1, H, hd)
    k = qkv[:, d:2 * d].reshape(-1, H, hd)
    v = qkv[:, 2 * d:].reshape(-1, H, hd)
    q = m.rnd(rope(q, pos, sp.rope_theta))
    k = m.rnd(rope(k, pos, sp.rope_theta))
    v = m.rnd(v)
    return q, k, v


def _layer_mlp_act(m: Model, l: int, h: np.ndarray, o: np.ndarray):
    """O projection added to the residual, RMSNorm, gate/up projection and the SwiGLU product
    (the norm's scale applied to the projection's output, as in _layer_pre_attn).
    Returns (residual after the attention block, rounded SwiGLU product)."""
    sp = m.spec
    f = sp.d_ffn
    h = h + m.rnd(o).reshape(h.shape[0], -1) @ m.W(f"layers.{l}.wo").T
    x2g = m.rnd(h * m.W(f"layers.{l}.mlp_norm"))
    gu = (x2g @ m.W(f"layers.{l}.wgate_up").T) * rms_scale(h, sp.rms_eps)
    return h, m.rnd(silu(gu[:, :f]) * gu[:, f:])


def _layer_mlp_out(m: Model, l: int, h: np.ndarray, a: np.ndarray) -> np.ndarray:
    """Down projection of the SwiGLU product added to the residual."""
    return h + a @ m.W(f"layers.{l}.wdown").T


def _layer_post_attn(m: Model, l: int, h: np.ndarray, o: np.ndarray) -> np.ndarray:
    h, a = _layer_mlp_act(m, l, h, o)
    return _layer_mlp_out(m, l, h, a)


def _attend(q: np.ndarray, K: np.ndarray, V: np.ndarray, mask: Optional[np.ndarray]) -> np.ndarray:
    """q [n,H,hd], K/V [m,H,hd], mask [n,m] (True = visible) -> o [n,H,hd]."""
    hd = q.shape[-1]
    s = np.einsum("nhd,mhd->hnm", q, K) / np.sqrt(hd)
    if mask is not None:
        s = np.where(mask[None, :, :], s, -np.inf)
    p = softmax(s, axis=-1)
    return np.einsum("hnm,mhd->nhd", p, V)


def final_hidden_to_logits(m: Model, h: np.ndarray, full_vocab: bool = False) -> np.ndarray:
    x = m.rnd(rmsnorm(h, m.W("final_norm"), m.spec.rms_eps))
    rows = m.W("lm_head") if full_vocab else m.item_rows()
    return x @ rows.T


def causal_forward(m: Model, tokens: Sequence[int], full_vocab: bool = False, keep_kv: bool = False):
    """Plain causal forward of a token sequence.

    Returns (logits [S, 1024 or V] fp64, per-layer (K, V) if keep_kv else None).
    """
    tokens = np.asarray(tokens, dtype=np.int64)
    S = tokens.shape[0]
    pos = np.arange(S)
    h = m.W("embed")[tokens].copy()
    causal = np.tril(np.ones((S, S), dtype=bool))
    kv = []
    for l in range(m.spec.n_layers):
        q, k, v = _layer_pre_attn(m, l, h, pos)
        o = _attend(q, k, v, causal)
        h = _layer_post_attn(m, l, h, o)
        if keep_kv:
            kv.append((k, v))
    return final_hidden_to_logits(m, h, full_vocab), (kv if keep_kv else None)


def path_tokens(path: Sequence[int], code_base: int) -> List[int]:
    """Item codes -> token ids: code c at level l (0-based) is code_base + 256*l + c."""
    return [code_base + CODES * l + int(c) for l, c in enumerate(path)]


class PathEvaluator:
    """Logits of ``prompt + path`` for many item-code paths of one user.

    The prompt is run once (its rows do not depend on what follows under causal
    attention); each path's token rows are computed from its parent path's
    cached K/V, which equals re-running the whole causal forward.
    """

    def __init__(self, m: Model, prompt: Sequence[int], full_vocab: bool = False):
        self.m = m
        self.full = full_vocab
        self.P = len(prompt)
        logits, kv = causal_forward(m, prompt, full_vocab, keep_kv=True)
        self.prefix_kv = kv
        self.root_logits = logits[-1]
        self.cache: Dict[Tuple[int, ...], Tuple[list, np.ndarray]] = {}

    def logits(self, paths: Sequence[Tuple[int, ...]]) -> List[np.ndarray]:
        """fp64 logit rows (item-code rows, or the whole vocabulary) at the end of each path.

        Missing paths (and their missing ancestors) are computed one depth at a time, all paths of
        a depth together, so each weight matrix is read once per depth."""
        missing = set()
        for p in paths:
            p = tuple(p)
            while len(p) > 0 and p not in self.cache and p not in missing:
                missing.add(p)
                p = p[:-1]
        for t in sorted({len(p) for p in missing}):
            self._extend(sorted(p for p in missing if len(p) == t))
        return [self.root_logits if len(p) == 0 else self.cache[tuple(p)][1] for p in paths]

    def _ensure(self, path: Tuple[int, ...]) -> None:
        if len(path) == 0 or path in self.cache:
            return
        todo = []
        p = path
        while len(p) > 0 and p not in self.cache:
            todo.append(p)
            p = p[:-1]
        for p in reversed(todo):
            self._extend([p])

    def extend_level(self, paths: Sequence[Tuple[int, ...]]) -> None:
        """Compute a batch of same-length paths whose parents are cached (row-batched GEMMs)."""
        todo = [tuple(p) for p in paths if tuple(p) not in self.cache]
        for p in todo:
            if len(p) > 1:
                self._ensure(p[:-1])
        if todo:
            self._extend(todo)

    def _extend(self, paths: List[Tuple[int, ...]]) -> None:
        m = self.m
        t = len(paths[0])
        assert all(len(p) == t for p in paths)
        toks = np.array([path_tokens(p, m.code_base)[-1] for p in paths], dtype=np.int64)
        pos = np.full(len(paths), self.P + t - 1)
        parents = [self.cache[p[:-1]][0] if t > 1 else None for p in paths]
        h = m.W("embed")[toks].copy()
        new_kv = [[] for _ in paths]
        for l in range(m.spec.n_layers):
            q, k, v = _layer_pre_attn(m, l, h, pos)
            Kp, Vp = self.prefix_kv[l]
            o = np.empty_like(q)
            for i in range(len(paths)):
                if parents[i] is not None:
                    Ka, Va = parents[i][l]
                    Ki = np.concatenate([Kp, Ka, k[i:i + 1]])
                    Vi = np.concatenate([Vp, Va, v[i:i + 1]])
                else:
                    Ki = np.concatenate([Kp, k[i:i + 1]])
                    Vi = np.concatenate([Vp, v[i:i + 1]])
                o[i] = _attend(q[i:i + 1], Ki, Vi, None)[0]
                pk = parents[i][l][0] if parents[i] is not None else k[i:i + 1][:0]
                pv = parents[i][l][1] if parents[i] is not None else v[i:i + 1][:0]
                new_kv[i].append((np.concatenate([pk, k[i:i + 1]]), np.concatenate([pv, v[i:i + 1]])))
            h = _layer_post_attn(m, l, h, o)
        logits = final_hidden_to_logits(m, h, self.full)
        for i, p in enumerate(paths):
            self.cache[p] = (new_kv[i], logits[i])


def tree_mask(parents: Sequence[int]) -> np.ndarray:
    """L_f x L_f tree mask of a flattened drafted sequence (App. A.3.1, Table 6).

    ``parents[i]`` is the flattened index of node i's parent (-1 for a node whose
    parent is the shared prefix).  Row i marks node i itself and every node on
    its path back to the prefix.
    """
    n = len(parents)
    M = np.zeros((n, n), dtype=bool)
    for i in range(n):
        j = i
        while j >= 0:
            M[i, j] = True
            j = parents[j]
    return M


def forward_tree_flat(m: Model, prompt: Sequence[int], flat_codes: Sequence[int], parents: Sequence[int],
                      depths: Sequence[int], full_vocab: bool = False) -> np.ndarray:
    """Paper formulation of the verification forward: one pass over prompt + flattened tree.

    Every flattened node attends to the whole prompt and to the tree nodes its
    mask row marks; node i sits at position P + depth_i - 1.  Returns the
    logits of every flattened node.
    """
    P = len(prompt)
    n = len(flat_codes)
    toks = np.array([m.code_base + CODES * (depths[i] - 1) + int(flat_codes[i]) for i in range(n)], dtype=np.int64)
    all_tok = np.concatenate([np.asarray(prompt, dtype=np.int64), toks])
    pos = np.concatenate([np.arange(P), P + np.asarray(depths, dtype=np.int64) - 1])
    S = P + n
    mask = np.zeros((S, S), dtype=bool)
    mask[:P, :P] = np.tril(np.ones((P, P), dtype=bool))
    mask[P:, :P] = True
    mask[P:, P:] = tree_mask(parents)
    h = m.W("embed")[all_tok].copy()
    for l in range(m.spec.n_layers):
        q, k, v = _layer_pre_attn(m, l, h, pos)
        o = _attend(q, k, v, mask)
        h = _layer_post_attn(m, l, h, o)
    return final_hidden_to_logits(m, h[P:], full_vocab)
