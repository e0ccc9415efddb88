"""Workload definitions and seeded generators (inputs only).

Workloads mirror the paper's evaluation setting (Sec. 4.1, App. A.3.1): item
identifiers of L=4 codebook tokens, a LLaMA-style target and a small draft
model, gamma=4 drafted beam steps, draft beam N=40 and K in {1..20}.  The
paper's datasets (Amazon Beauty/Games) and trained weights are not available,
so every workload here is synthetic and seeded:

* weights: i.i.d. normal, std 0.02 for every matrix except the LM head
  (std 3/sqrt(d), so that unit-RMS final hidden states give logits of std ~3),
  RMSNorm gains 1 + 0.1*N(0,1); every value rounded to bf16 (RNE);
* items: ``n_items`` distinct 4-tuples of codes in [0, 256), codes drawn per
  level either uniformly or Zipf(a) over ranks mapped through a seeded
  per-level permutation (so popular codes are not all low indices);
* token id of code ``c`` at level ``l`` (0-based) = ``code_base + 256*l + c``;
* prompts: i.i.d. uniform tokens over the whole vocabulary.
"""
from __future__ import annotations

import dataclasses
import os
import zlib
from concurrent.futures import ThreadPoolExecutor
from typing import Dict, Iterator, List, Optional, Sequence, Tuple

import numpy as np

L_ITEM = 4          # codebook identifier length (paper: L = 4)
CODES = 256         # codes per level

__all__ = [
    "L_ITEM", "CODES", "ModelSpec", "Workload", "WORKLOADS", "workload",
    "bf16_round_input", "normal_bf16", "model_tensor_names", "model_tensor",
    "iter_model_tensors", "model_weights", "make_items", "make_prompts",
    "random_logits", "random_tree", "SWEEP_AXES",
]


@dataclasses.dataclass(frozen=True)
class ModelSpec:
    n_layers: int
    d_model: int
    n_heads: int
    d_ffn: int
    vocab: int
    rms_eps: float = 1e-6
    rope_theta: float = 10000.0

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_heads

    def n_params(self) -> int:
        d, f = self.d_model, self.d_ffn
        per_layer = 4 * d * d + 3 * d * f + 2 * d
        return self.n_layers * per_layer + 2 * self.vocab * d + d


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    target: ModelSpec
    draft: ModelSpec
    n_items: int
    code_dist: str            # "uniform" | "zipf"
    zipf_a: float
    code_base: int
    prompt_len: Tuple[int, int]   # inclusive range
    n_users: int
    K: int
    N: int
    gamma: int
    modes: Tuple[str, ...]
    seed: int                 # world seed (weights, items, prompts)
    philox_seed: int = 0


_T7 = ModelSpec(32, 4096, 32, 11008, 33024)
_D7 = ModelSpec(4, 768, 12, 3072, 33024)

WORKLOADS: Dict[str, Workload] = {
    # tiny: 2-layer target d=128, vocab = the 1024 item codes only
    "tiny": Workload("tiny", ModelSpec(2, 128, 4, 512, 1024), ModelSpec(1, 64, 2, 256, 1024),
                     1000, "uniform", 0.0, 0, (32, 32), 1, 5, 10, 2, ("strict",), 1),
    "mid": Workload("mid", ModelSpec(16, 2048, 32, 5632, 33024), ModelSpec(2, 512, 8, 1408, 33024),
                    20000, "zipf", 1.1, 32000, (256, 256), 1, 10, 40, 4, ("strict",), 2),
    "7b": Workload("7b", _T7, _D7, 50000, "zipf", 1.1, 32000, (512, 512), 1, 10, 40, 4,
                   ("strict", "relaxed"), 3, 0),
    "7b_b16": Workload("7b_b16", _T7, _D7, 200000, "zipf", 1.1, 32000, (256, 1024), 16, 20, 80, 4,
                       ("relaxed",), 4, 0),
    "sweep": Workload("sweep", _T7, _D7, 50000, "zipf", 1.1, 32000, (512, 512), 1, 10, 40, 4,
                      ("strict", "relaxed"), 5, 0),
}

# verify-call sweep on the 7B-shape target (K x gamma x draft-beam multiple x batch)
SWEEP_AXES = {"K": (1, 5, 10, 20), "gamma": (1, 2, 3, 4), "N_mult": (1, 2, 4), "batch": (1, 4, 16)}


def workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return dataclasses.replace(w, **overrides) if overrides else w


# ----------------------------------------------------------------------------------------------
# bf16 helpers for *input preparation* (weights are bf16 by construction)
# ----------------------------------------------------------------------------------------------

def bf16_round_input(x: np.ndarray) -> np.ndarray:
    """Round a float32 array to the nearest bf16 value (ties to even), returned as float32."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    u = u + (np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))
    u &= np.uint32(0xFFFF0000)
    return u.view(np.float32)


def _tag(*parts) -> int:
    return zlib.crc32("/".join(str(p) for p in parts).encode())


_CHUNK = 1 << 22
_POOL: Optional[ThreadPoolExecutor] = None


def _pool() -> ThreadPoolExecutor:
    global _POOL
    if _POOL is None:
        _POOL = ThreadPoolExecutor(max(1, min(32, os.cpu_count() or 1)))
    return _POOL


def normal_bf16(seed: int, tag: int, n: int, std: float, mean: float = 0.0) -> np.ndarray:
    """``n`` i.i.d. N(mean, std^2) values rounded to bf16, as float32.

    Generated in fixed chunks of 4M values, each from its own Philox-seeded numpy
    generator keyed by (seed, tag, chunk), so the result does not depend on the
    number of threads used.
    """
    out = np.empty(n, dtype=np.float32)
    nchunks = (n + _CHUNK - 1) // _CHUNK

    def fill(c: int) -> None:
        lo, hi = c * _CHUNK, min(n, (c + 1) * _CHUNK)
        rng = np.random.Generator(np.random.Philox(np.random.SeedSequence([seed, tag, c])))
        v = rng.standard_normal(hi - lo, dtype=np.float32)
        v *= np.float32(std)
        if mean:
            v += np.float32(mean)
        out[lo:hi] = bf16_round_input(v)

    if nchunks == 1:
        fill(0)
    else:
        list(_pool().map(fill, range(nchunks)))
    return out


def model_tensor_names(spec: ModelSpec) -> List[str]:
    names = ["embed", "final_norm", "lm_head"]
    for l in range(spec.n_layers):
        names += [f"layers.{l}.{k}" for k in ("attn_norm", "wqkv", "wo", "mlp_norm", "wgate_up", "wdown")]
    return names


def _tensor_shape_std(spec: ModelSpec, name: str):
    d, f, V = spec.d_model, spec.d_ffn, spec.vocab
    leaf = name.split(".")[-1]
    table = {
        "embed": ((V, d), 0.02, 0.0),
        "lm_head": ((V, d), 3.0 / np.sqrt(d), 0.0),
        "final_norm": ((d,), 0.1, 1.0),
        "attn_norm": ((d,), 0.1, 1.0),
        "mlp_norm": ((d,), 0.1, 1.0),
        "wqkv": ((3 * d, d), 0.02, 0.0),      # rows: q (d), k (d), v (d); head-major inside each
        "wo": ((d, d), 0.02, 0.0),
        "wgate_up": ((2 * f, d), 0.02, 0.0),  # rows: gate (f) then up (f)
        "wdown": ((d, f), 0.02, 0.0),
    }
    return table[leaf]


def model_tensor(spec: ModelSpec, seed: int, role: str, name: str) -> np.ndarray:
    shape, std, mean = _tensor_shape_std(spec, name)
    n = int(np.prod(shape))
    return normal_bf16(seed, _tag(role, name, spec), n, float(std), mean).reshape(shape)


def iter_model_tensors(spec: ModelSpec, seed: int, role: str) -> Iterator[Tuple[str, np.ndarray]]:
    for name in model_tensor_names(spec):
        yield name, model_tensor(spec, seed, role, name)


def model_weights(spec: ModelSpec, seed: int, role: str) -> Dict[str, np.ndarray]:
    """All weights of one model (role = "target" | "draft") as bf16-valued float32 arrays."""
    return dict(iter_model_tensors(spec, seed, role))


# ----------------------------------------------------------------------------------------------
# items and prompts
# ----------------------------------------------------------------------------------------------

def make_items(n_items: int, dist: str, zipf_a: float, seed: int, L: int = L_ITEM,
               codes: int = CODES) -> np.ndarray:
    """``n_items`` distinct L-tuples of codes (int32 [n_items, L]), in generation order."""
    rng = np.random.default_rng([seed, _tag("items")])
    if dist == "uniform":
        probs = [None] * L
        perms = [np.arange(codes)] * L
    elif dist == "zipf":
        w = np.arange(1, codes + 1, dtype=np.float64) ** (-zipf_a)
        w /= w.sum()
        probs = [w] * L
        perms = [rng.permutation(codes) for _ in range(L)]
    else:
        raise ValueError(dist)
    seen = set()
    out: List[Tuple[int, ...]] = []
    while len(out) < n_items:
        m = 2 * (n_items - len(out)) + 16
        cols = [perms[l][rng.choice(codes, size=m, p=probs[l])] for l in range(L)]
        for row in zip(*cols):
            t = tuple(int(c) for c in row)
            if t not in seen:
                seen.add(t)
                out.append(t)
                if len(out) == n_items:
                    break
    return np.asarray(out, dtype=np.int32).reshape(n_items, L)


def make_prompts(n_users: int, len_range: Tuple[int, int], vocab: int, seed: int) -> List[np.ndarray]:
    rng = np.random.default_rng([seed, _tag("prompts")])
    lens = rng.integers(len_range[0], len_range[1] + 1, size=n_users)
    return [rng.integers(0, vocab, size=int(n)).astype(np.int32) for n in lens]


# ----------------------------------------------------------------------------------------------
# kernel-level parity cases: random logits and random drafted trees built from item prefixes
# ----------------------------------------------------------------------------------------------

def random_logits(shape: Sequence[int], seed: int, std: float = 3.0) -> np.ndarray:
    rng = np.random.default_rng([seed, _tag("logits")])
    return (rng.standard_normal(size=tuple(shape)) * std).astype(np.float32)


def random_tree(items: np.ndarray, depth: int, n_in: int, levels: int, width: int, seed: int):
    """A drafted beam tree whose every beam is a prefix of some item.

    Returns ``(incoming, levels_list)`` where ``incoming`` is a list of ``n_in``
    distinct ``depth``-prefixes (the empty tuple when depth == 0) and
    ``levels_list[j]`` is a list of (parent index into the previous level, code)
    pairs, at most ``width`` per level, each extending a beam of the previous
    level by one valid code.  Pure input construction: prefixes are read off
    sampled items; no scoring is involved.
    """
    rng = np.random.default_rng([seed, _tag("tree")])
    n = items.shape[0]
    if depth == 0:
        incoming = [()]
    else:
        pref = sorted({tuple(int(c) for c in items[i, :depth]) for i in range(n)})
        pick = rng.permutation(len(pref))[:n_in]
        incoming = [pref[i] for i in sorted(pick)]
    # index items by prefix to extend beams
    prev = list(incoming)
    out = []
    for j in range(levels):
        lvl = depth + j + 1
        if lvl > items.shape[1]:
            break
        by_parent = {}
        prev_set = {p: i for i, p in enumerate(prev)}
        for i in range(n):
            p = tuple(int(c) for c in items[i, :lvl - 1])
            if p in prev_set:
                by_parent.setdefault(prev_set[p], set()).add(int(items[i, lvl - 1]))
        cands = sorted((pi, c) for pi, cs in by_parent.items() for c in cs)
        order = rng.permutation(len(cands))[:width]
        chosen = [cands[i] for i in order]          # random "draft order"
        out.append(chosen)
        prev = [prev[pi] + (c,) for pi, c in chosen]
    return incoming, out
