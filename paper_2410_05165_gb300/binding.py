"""Thin ctypes binding of ``libatspeed.so`` (the C ABI in include/atspeed.h).

Argument marshalling only: every step of the verification call runs in the CUDA library.  PyTorch
supplies device memory (weights, inputs, outputs) and the CUDA stream.  There is no CPU fallback:
if the library is missing or fails to load, every entry point raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np
import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libatspeed.so")

OK, E_ARG, E_SHAPE, E_OOM, E_CUDA, E_TIMEOUT, E_STATE, E_UNSUPPORTED = 0, -1, -2, -3, -4, -5, -6, -7
STRICT, RELAXED = 0, 1
NORM_MASKED, NORM_FULL = 0, 1
PLAIN_TOPK, PLAIN_SAMPLE, SD_STRICT, SD_RELAXED = 0, 1, 2, 3

EXPORTS = [
    "atspeed_create", "atspeed_destroy", "atspeed_last_error", "atspeed_prefill", "atspeed_begin_step",
    "atspeed_draft_step", "atspeed_verify", "atspeed_draft_step_logits", "atspeed_verify_logits",
    "atspeed_beam_search", "atspeed_set_early_reject", "atspeed_profile", "atspeed_profile_read", "atspeed_tree_shape", "atspeed_debug_tree",
    "atspeed_debug_node_logits", "atspeed_debug_node_lse", "atspeed_debug_buffer", "atspeed_set_tree", "atspeed_op_workspace_bytes", "atspeed_op_gemm",
    "atspeed_op_gemm_noalloc", "atspeed_op_status", "atspeed_op_gemm_swiglu", "atspeed_op_rmsnorm", "atspeed_op_attention_scratch", "atspeed_op_attention",
]


class AtSpeedError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"atspeed status {status}: {msg}")
        self.status = status


class ModelDesc(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("d_ffn", ctypes.c_int), ("vocab", ctypes.c_int), ("rms_eps", ctypes.c_float),
                ("rope_theta", ctypes.c_float), ("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p), ("attn_norm", ctypes.POINTER(ctypes.c_void_p)),
                ("wqkv", ctypes.POINTER(ctypes.c_void_p)), ("wo", ctypes.POINTER(ctypes.c_void_p)),
                ("mlp_norm", ctypes.POINTER(ctypes.c_void_p)), ("wgate_up", ctypes.POINTER(ctypes.c_void_p)),
                ("wdown", ctypes.POINTER(ctypes.c_void_p))]


class ItemsDesc(ctypes.Structure):
    _fields_ = [("n_items", ctypes.c_int), ("L", ctypes.c_int), ("codes_per_level", ctypes.c_int),
                ("code_base", ctypes.c_int), ("h_codes", ctypes.POINTER(ctypes.c_int32))]


class Limits(ctypes.Structure):
    _fields_ = [("max_users", ctypes.c_int), ("max_prompt", ctypes.c_int), ("max_K", ctypes.c_int),
                ("max_N", ctypes.c_int), ("max_gamma", ctypes.c_int)]


class DecodeOpts(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int), ("N", ctypes.c_int), ("gamma", ctypes.c_int), ("norm", ctypes.c_int),
                ("philox_seed", ctypes.c_uint64)]


_lib: Optional[ctypes.CDLL] = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Loads the CUDA library (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"libatspeed.so not built ({path}); run __graft_entry__.build() first")
    lib = ctypes.CDLL(path)
    vp, i32p, fp = ctypes.c_void_p, ctypes.POINTER(ctypes.c_int32), ctypes.POINTER(ctypes.c_float)
    c_int = ctypes.c_int
    sig = {
        "atspeed_create": (c_int, [ctypes.POINTER(ModelDesc), ctypes.POINTER(ModelDesc), ctypes.POINTER(ItemsDesc),
                                   ctypes.POINTER(Limits), ctypes.POINTER(vp)]),
        "atspeed_destroy": (None, [vp]),
        "atspeed_last_error": (ctypes.c_char_p, [vp]),
        "atspeed_prefill": (c_int, [vp, vp, c_int, vp, i32p]),
        "atspeed_begin_step": (c_int, [vp, vp, ctypes.POINTER(DecodeOpts)]),
        "atspeed_draft_step": (c_int, [vp, vp, ctypes.POINTER(DecodeOpts), c_int]),
        "atspeed_verify": (c_int, [vp, vp, ctypes.POINTER(DecodeOpts), c_int, vp, vp, vp, vp]),
        "atspeed_draft_step_logits": (c_int, [vp, vp, ctypes.POINTER(DecodeOpts), c_int, fp]),
        "atspeed_verify_logits": (c_int, [vp, vp, ctypes.POINTER(DecodeOpts), c_int, fp, vp, vp, vp, vp]),
        "atspeed_beam_search": (c_int, [vp, vp, c_int, vp, i32p, ctypes.POINTER(DecodeOpts), c_int, vp, vp, i32p]),
        "atspeed_set_early_reject": (c_int, [vp, c_int]),
        "atspeed_profile": (c_int, [vp, c_int]),
        "atspeed_profile_read": (c_int, [vp, c_int, i32p, ctypes.POINTER(ctypes.c_double),
                                         ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]),
        "atspeed_tree_shape": (c_int, [vp, i32p, i32p, i32p, i32p]),
        "atspeed_debug_tree": (c_int, [vp, i32p, fp, fp, i32p]),
        "atspeed_debug_node_logits": (c_int, [vp, c_int, c_int, c_int, fp]),
        "atspeed_debug_node_lse": (c_int, [vp, c_int, c_int, c_int, fp]),
        "atspeed_debug_buffer": (c_int, [vp, c_int, c_int, vp, ctypes.c_size_t]),
        "atspeed_set_tree": (c_int, [vp, vp, c_int, i32p, i32p, i32p, fp, fp]),
        "atspeed_op_workspace_bytes": (ctypes.c_size_t, []),
        "atspeed_op_gemm": (c_int, [vp, vp, vp, c_int, c_int, c_int, c_int, vp, c_int, c_int, vp]),
        "atspeed_op_gemm_noalloc": (c_int, [vp, vp, vp, c_int, c_int, c_int, c_int, vp, c_int, c_int]),
        "atspeed_op_gemm_swiglu": (c_int, [vp, vp, vp, c_int, c_int, c_int, c_int, vp, c_int, vp]),
        "atspeed_op_status": (c_int, [vp, vp]),
        "atspeed_op_rmsnorm": (c_int, [vp, vp, vp, c_int, c_int, ctypes.c_float, vp, c_int]),
        "atspeed_op_attention_scratch": (ctypes.c_size_t, [c_int, c_int, c_int, c_int]),
        "atspeed_op_attention": (c_int, [vp, vp, vp, vp, c_int, c_int, c_int, c_int, c_int, i32p, i32p, i32p, i32p,
                                         vp, vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _i32(a) -> ctypes.Array:
    a = np.ascontiguousarray(a, dtype=np.int32)
    return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def _stream(stream: Optional[torch.cuda.Stream]) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _check(status: int, ctx=None):
    if status != OK:
        lib = load()
        msg = lib.atspeed_last_error(ctx)
        raise AtSpeedError(status, msg.decode() if msg else "")


def weights_to_device(weights: Dict[str, np.ndarray], device="cuda") -> Dict[str, torch.Tensor]:
    """float32 arrays holding bf16 values -> bf16 device tensors (exact)."""
    return {k: torch.from_numpy(np.ascontiguousarray(v)).to(device=device, dtype=torch.bfloat16)
            for k, v in weights.items()}


def _model_desc(spec, w: Dict[str, torch.Tensor]):
    L = spec.n_layers
    arrs = {}
    for key in ("attn_norm", "wqkv", "wo", "mlp_norm", "wgate_up", "wdown"):
        ptrs = [w[f"layers.{l}.{key}"].data_ptr() for l in range(L)]
        arrs[key] = (ctypes.c_void_p * L)(*ptrs)
    d = ModelDesc(spec.n_layers, spec.d_model, spec.n_heads, spec.d_ffn, spec.vocab, spec.rms_eps, spec.rope_theta,
                  w["embed"].data_ptr(), w["final_norm"].data_ptr(), w["lm_head"].data_ptr(),
                  arrs["attn_norm"], arrs["wqkv"], arrs["wo"], arrs["mlp_norm"], arrs["wgate_up"], arrs["wdown"])
    return d, arrs


def opts(K: int, N: int, gamma: int, seed: int = 0, norm: int = NORM_MASKED) -> DecodeOpts:
    return DecodeOpts(K, N, gamma, norm, seed)


class Context:
    """One atspeed_ctx: borrowed device weights, the item trie and every device buffer."""

    def __init__(self, target_spec, target_w: Dict[str, torch.Tensor], draft_spec, draft_w,
                 items: np.ndarray, code_base: int, max_users: int, max_prompt: int, max_K: int, max_N: int,
                 max_gamma: int):
        lib = load()
        self._lib = lib
        self._keep = [target_w, draft_w]
        td, ta = _model_desc(target_spec, target_w)
        self._keep += [td, ta]
        dd = None
        if draft_spec is not None:
            dd, da = _model_desc(draft_spec, draft_w)
            self._keep += [dd, da]
        it = np.ascontiguousarray(items, dtype=np.int32)
        self._keep.append(it)
        idesc = ItemsDesc(it.shape[0], it.shape[1], 256, code_base, it.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)))
        lim = Limits(max_users, max_prompt, max_K, max_N, max_gamma)
        self.max_N = max_N
        out = ctypes.c_void_p()
        st = lib.atspeed_create(ctypes.byref(td), ctypes.byref(dd) if dd is not None else None, ctypes.byref(idesc),
                                ctypes.byref(lim), ctypes.byref(out))
        _check(st, None)
        self.ptr = out.value
        self.n_users = 0

    def close(self):
        if getattr(self, "ptr", None):
            self._lib.atspeed_destroy(self.ptr)
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- calls -----------------------------------------------------------------------------------
    def prefill(self, tokens: torch.Tensor, offsets: Sequence[int], stream=None):
        off, offp = _i32(offsets)
        self.n_users = len(offsets) - 1
        _check(self._lib.atspeed_prefill(self.ptr, _stream(stream), self.n_users, tokens.data_ptr(), offp), self.ptr)

    def begin_step(self, o: DecodeOpts, stream=None):
        _check(self._lib.atspeed_begin_step(self.ptr, _stream(stream), ctypes.byref(o)), self.ptr)

    def draft_step(self, o: DecodeOpts, mode: int, stream=None):
        _check(self._lib.atspeed_draft_step(self.ptr, _stream(stream), ctypes.byref(o), mode), self.ptr)

    def verify(self, o: DecodeOpts, mode: int, stream=None):
        B, K = self.n_users, o.K
        dev = torch.device("cuda")
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        depth = torch.empty(B, dtype=torch.int32, device=dev)
        beams = torch.empty(B, K, 4, dtype=torch.int32, device=dev)
        scores = torch.empty(B, K, dtype=torch.float32, device=dev)
        _check(self._lib.atspeed_verify(self.ptr, _stream(stream), ctypes.byref(o), mode, acc.data_ptr(),
                                        depth.data_ptr(), beams.data_ptr(), scores.data_ptr()), self.ptr)
        return acc, depth, beams, scores

    def draft_step_logits(self, o: DecodeOpts, mode: int, logits: np.ndarray, stream=None):
        """logits [n_users][width][1024]: draft item-code logits of the previous level's slots."""
        lg = np.ascontiguousarray(logits, np.float32)
        _check(self._lib.atspeed_draft_step_logits(self.ptr, _stream(stream), ctypes.byref(o), mode,
                                                   lg.ctypes.data_as(ctypes.POINTER(ctypes.c_float))), self.ptr)

    def verify_logits(self, o: DecodeOpts, mode: int, logits: np.ndarray, stream=None):
        """logits [n_users][K + gamma*N][1024]: target item-code logits of every node slot."""
        B, K = self.n_users, o.K
        dev = torch.device("cuda")
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        depth = torch.empty(B, dtype=torch.int32, device=dev)
        beams = torch.empty(B, K, 4, dtype=torch.int32, device=dev)
        scores = torch.empty(B, K, dtype=torch.float32, device=dev)
        lg = np.ascontiguousarray(logits, np.float32)
        _check(self._lib.atspeed_verify_logits(self.ptr, _stream(stream), ctypes.byref(o), mode,
                                               lg.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), acc.data_ptr(),
                                               depth.data_ptr(), beams.data_ptr(), scores.data_ptr()), self.ptr)
        return acc, depth, beams, scores

    def beam_search(self, tokens: torch.Tensor, offsets: Sequence[int], o: DecodeOpts, mode: int, stream=None,
                    items_out: Optional[torch.Tensor] = None, scores_out: Optional[torch.Tensor] = None):
        B = len(offsets) - 1
        self.n_users = B
        dev = torch.device("cuda")
        items = items_out if items_out is not None else torch.empty(B, o.K, 4, dtype=torch.int32, device=dev)
        scores = scores_out if scores_out is not None else torch.empty(B, o.K, dtype=torch.float32, device=dev)
        stats = np.zeros((B, 3), dtype=np.int32)
        off, offp = _i32(offsets)
        _check(self._lib.atspeed_beam_search(self.ptr, _stream(stream), B, tokens.data_ptr(), offp, ctypes.byref(o),
                                             mode, items.data_ptr(), scores.data_ptr(),
                                             stats.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))), self.ptr)
        return items, scores, stats

    def set_early_reject(self, enable: bool):
        _check(self._lib.atspeed_set_early_reject(self.ptr, 1 if enable else 0), self.ptr)

    def profile(self, enable: bool):
        _check(self._lib.atspeed_profile(self.ptr, 1 if enable else 0), self.ptr)

    def profile_read(self, kind: int):
        n = ctypes.c_int32()
        ms, by, fl = ctypes.c_double(), ctypes.c_double(), ctypes.c_double()
        _check(self._lib.atspeed_profile_read(self.ptr, kind, ctypes.byref(n), ctypes.byref(ms), ctypes.byref(by),
                                              ctypes.byref(fl)), self.ptr)
        return {"launches": n.value, "ms": ms.value, "bytes": by.value, "flops": fl.value}

    # -- introspection -----------------------------------------------------------------------------
    def tree_shape(self):
        B = self.n_users
        depth = np.zeros(B, np.int32)
        levels = np.zeros(B, np.int32)
        si = np.zeros(1, np.int32)
        sl = np.zeros(1, np.int32)
        p = lambda a: a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))
        _check(self._lib.atspeed_tree_shape(self.ptr, p(depth), p(levels), p(si), p(sl)), self.ptr)
        return depth, levels, int(si[0]), int(sl[0])

    def debug_tree(self, gamma: int):
        depth, levels, si, sl = self.tree_shape()
        B = self.n_users
        stride = si + gamma * sl
        path = np.zeros((B, stride, 4), np.int32)
        sq = np.zeros((B, stride), np.float32)
        sp = np.zeros((B, stride), np.float32)
        cnt = np.zeros((B, gamma + 1), np.int32)
        _check(self._lib.atspeed_debug_tree(self.ptr, path.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                                            sq.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                                            sp.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                                            cnt.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))), self.ptr)
        return {"path": path, "sq": sq, "sp": sp, "count": cnt, "slots_in": si, "slots_lvl": sl, "depth": depth,
                "levels": levels}

    def debug_buffer(self, which: int, buf: int, dtype, count: int) -> np.ndarray:
        out = np.zeros(count, dtype=dtype)
        _check(self._lib.atspeed_debug_buffer(self.ptr, which, buf, out.ctypes.data, out.nbytes), self.ptr)
        return out

    def node_logits(self, which: int, user: int, slot: int) -> np.ndarray:
        out = np.zeros(1024, np.float32)
        _check(self._lib.atspeed_debug_node_logits(self.ptr, which, user, slot,
                                                   out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))), self.ptr)
        return out

    def node_lse(self, which: int, user: int, slot: int) -> float:
        out = np.zeros(1, np.float32)
        _check(self._lib.atspeed_debug_node_lse(self.ptr, which, user, slot,
                                                out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))), self.ptr)
        return float(out[0])

    def set_tree(self, counts: np.ndarray, parents: np.ndarray, codes: np.ndarray, sq: np.ndarray,
                 draft_logits: Optional[np.ndarray] = None, stream=None):
        """counts [B][n_levels]; parents/codes/sq [B][n_levels][max_N]; draft_logits
        [B][n_levels][max_N][1024] (logits of the parents on levels 0 .. n_levels-1) or None."""
        n_levels = counts.shape[1]
        c, cp = _i32(counts)
        p, pp = _i32(parents)
        k, kp = _i32(codes)
        s = np.ascontiguousarray(sq, np.float32)
        dl = None if draft_logits is None else np.ascontiguousarray(draft_logits, np.float32)
        _check(self._lib.atspeed_set_tree(self.ptr, _stream(stream), n_levels, cp, pp, kp,
                                          s.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                                          None if dl is None else dl.ctypes.data_as(ctypes.POINTER(ctypes.c_float))),
               self.ptr)


# ---------------------------------------------------------------------------------------------------
# stateless operators
# ---------------------------------------------------------------------------------------------------
_ws: Dict[int, torch.Tensor] = {}


def op_workspace(device: int = 0) -> torch.Tensor:
    if device not in _ws:
        n = load().atspeed_op_workspace_bytes()
        _ws[device] = torch.zeros(n, dtype=torch.uint8, device=f"cuda:{device}")
    return _ws[device]


def op_gemm(W: torch.Tensor, X: torch.Tensor, T: int, Y: Optional[torch.Tensor] = None, accumulate=False,
            stream=None) -> torch.Tensor:
    M, K = W.shape
    if Y is None:
        Y = torch.zeros(T, M, dtype=torch.float32, device=W.device)
    _check(load().atspeed_op_gemm(_stream(stream), W.data_ptr(), X.data_ptr(), M, K, T, X.shape[0], Y.data_ptr(),
                                  Y.shape[1], 1 if accumulate else 0, op_workspace().data_ptr()))
    return Y


def op_gemm_noalloc(W: torch.Tensor, X: torch.Tensor, T: int, Y: Optional[torch.Tensor] = None, accumulate=False,
                    stream=None) -> torch.Tensor:
    """atspeed_op_gemm without a workspace argument (the library's fixed scratch array is used)."""
    M, K = W.shape
    if Y is None:
        Y = torch.zeros(T, M, dtype=torch.float32, device=W.device)
    _check(load().atspeed_op_gemm_noalloc(_stream(stream), W.data_ptr(), X.data_ptr(), M, K, T, X.shape[0],
                                          Y.data_ptr(), Y.shape[1], 1 if accumulate else 0))
    return Y


def op_status(noalloc: bool = False, stream=None) -> int:
    """atspeed_op_status: synchronises, reads and clears the device error word of the op GEMMs'
    workspace (or of the allocation-free scratch); returns the status code (0 = no device error)."""
    ws = None if noalloc else op_workspace().data_ptr()
    return int(load().atspeed_op_status(_stream(stream), ws))


def op_gemm_swiglu(W: torch.Tensor, X: torch.Tensor, T: int, stream=None) -> torch.Tensor:
    F2, K = W.shape
    out = torch.zeros(T, F2 // 2, dtype=torch.bfloat16, device=W.device)
    _check(load().atspeed_op_gemm_swiglu(_stream(stream), W.data_ptr(), X.data_ptr(), F2 // 2, K, T, X.shape[0],
                                         out.data_ptr(), out.shape[1], op_workspace().data_ptr()))
    return out


def op_rmsnorm(h: torch.Tensor, g: torch.Tensor, eps: float, stream=None) -> torch.Tensor:
    T, d = h.shape
    x = torch.zeros(T, d, dtype=torch.bfloat16, device=h.device)
    _check(load().atspeed_op_rmsnorm(_stream(stream), h.data_ptr(), g.data_ptr(), T, d, eps, x.data_ptr(), d))
    return x


def op_attention(q: torch.Tensor, kc: torch.Tensor, vc: torch.Tensor, n_heads: int, head_dim: int, P: int,
                 pages: Sequence[int], vis: Sequence[int], path_rows: Optional[np.ndarray] = None,
                 n_path: Optional[Sequence[int]] = None, stream=None) -> torch.Tensor:
    lib = load()
    T = q.shape[0]
    out = torch.zeros(T, n_heads * head_dim, dtype=torch.bfloat16, device=q.device)
    scratch = torch.empty(lib.atspeed_op_attention_scratch(T, n_heads, head_dim, P), dtype=torch.uint8,
                          device=q.device)
    pg, pgp = _i32(list(pages) if len(pages) else [0])
    vv, vvp = _i32(vis)
    pr = np.zeros((T, 4), np.int32) if path_rows is None else path_rows
    pr, prp = _i32(pr)
    npth = np.zeros(T, np.int32) if n_path is None else n_path
    npth, npp = _i32(npth)
    _check(lib.atspeed_op_attention(_stream(stream), q.data_ptr(), kc.data_ptr(), vc.data_ptr(), kc.shape[0], T,
                                    n_heads, head_dim, P, pgp, vvp, prp, npp, out.data_ptr(), scratch.data_ptr()))
    return out
