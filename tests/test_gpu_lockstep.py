"""Layer-by-layer lockstep parity of the verification call's decoder forward against the oracle
(Sec. 3.3 "Tree-based Attention", App. A.3.1: a drafted node's logits are the last-position logits
of the causal forward of prompt + path; the tree forward computes all of them in one pass).

End to end, each side runs every layer on its own previous output, so one bf16 rounding decision
that comes out the other way (fp32 tensor-core sums against the oracle's fp64) propagates through
all later layers.  Here every layer of the oracle runs on the GPU's OWN input to that layer, and
each rounding point of the layer is compared on its own:

* q, k, v after RoPE (bf16), from the GPU's residual entering the layer (the GEMM input is the
  gain-scaled residual g * h in bf16, the norm's per-token scale multiplies the GEMM output);
* the tree attention output (bf16), from the GPU's q and its K/V cache (history pages written by
  the prefill, path keys written by this forward);
* the SwiGLU product (bf16), from the GPU's attention output (O projection, residual and RMSNorm in
  fp64);
* the fp32 residual leaving the layer, from the GPU's SwiGLU product;
* the final RMSNorm (bf16) and the item-code logits, from the GPU's final residual.

The GPU's input to layer l is the residual of a context whose model holds the first l layers of
the same weights: the forward is deterministic and no work split depends on the layer count, which
the test checks by comparing the shared layers' K/V cache rows bit for bit.

Tolerance of a bf16 output: one bf16 ulp of the oracle's rounded value, plus what can move the
value before its rounding -- the fp32 accumulation of the GEMM that feeds it (4 * 2^-24 * sqrt(K) *
sum_k |a_k w_k|) and the inputs of that GEMM whose own rounding could come out either way (a bf16
input within the fp32 error of a rounding boundary, one ulp times |w|); the attention output also
absorbs the fp16 rounding of its softmax weights (2^-10 of sum p|v| / sum p).  The fp32 residual
and the logits: within the benchmark spec's 2e-2 (the measured differences are printed).
"""
import numpy as np
import pytest
import torch

import synth
from oracle.model import (Model, _attend, _layer_mlp_act, _layer_mlp_out, _layer_pre_attn,
                          final_hidden_to_logits)
from oracle.numerics import bf16, rms_scale, rmsnorm, rope_angles, silu

pytestmark = pytest.mark.gpu

U32 = 2.0 ** -24


@pytest.fixture(scope="module")
def ats():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2410_05165_gb300 as m
    return m


def _ulp(x):
    """bf16 ulp of |x| (8 significant bits), at least the smallest normal's."""
    a = np.maximum(np.abs(np.asarray(x, np.float64)), 2.0 ** -126)
    return 2.0 ** (np.floor(np.log2(a)) - 7)


def _flip_risk(r, rel):
    """1 where an fp64 value r, perturbed by rel * |r| (the other side's fp32 arithmetic), could
    round to a different bf16 value: its distance to the nearest rounding boundary is below that."""
    u = _ulp(r)
    frac = np.abs(r) / u - np.floor(np.abs(r) / u)        # position inside the ulp, rounding at 0.5
    return (np.abs(frac - 0.5) * u <= rel * np.abs(r) + 1e-30).astype(np.float64)


def _check_bf16(name, got, ref, slack):
    """|got - ref| <= ulp + slack element-wise; prints the share of exact matches."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    d = np.abs(got - ref)
    lim = np.maximum(_ulp(ref), _ulp(got)) + slack
    ratio = d / lim
    worst = np.unravel_index(np.argmax(ratio), ratio.shape)
    print(f"  {name:10s} exact {np.mean(d == 0):.4f}  within 1 ulp {np.mean(d <= np.maximum(_ulp(ref), _ulp(got))):.5f}"
          f"  max |d|/tol {ratio.max():.3f}")
    assert ratio.max() <= 1.0, (name, worst, got[worst], ref[worst], lim[worst])


def _bf16_to_f64(a_u16):
    return (np.asarray(a_u16, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


class GpuCut:
    """The verification forward of a model cut to its first `c` layers: buffers after the call."""

    def __init__(self, ats, spec, c, tw_dev, items, code_base, prompts, K, N, G, levels):
        self.spec_c = synth.ModelSpec(c, spec.d_model, spec.n_heads, spec.d_ffn, spec.vocab)
        B = len(prompts)
        ctx = ats.Context(self.spec_c, tw_dev, None, None, items, code_base, max_users=B,
                          max_prompt=max(len(p) for p in prompts), max_K=K, max_N=N, max_gamma=G)
        toks = torch.from_numpy(np.concatenate(prompts).astype(np.int32)).cuda()
        off = np.concatenate([[0], np.cumsum([len(p) for p in prompts])]).astype(np.int32)
        ctx.prefill(toks, off)
        o = ats.opts(K, N, G)
        ctx.begin_step(o)
        cnt = np.zeros((B, G), np.int32)
        par = np.zeros((B, G, N), np.int32)
        cod = np.zeros((B, G, N), np.int32)
        for u in range(B):
            for j, lvl in enumerate(levels[u]):
                cnt[u, j] = len(lvl)
                for k, (p, cc) in enumerate(lvl):
                    par[u, j, k], cod[u, j, k] = p, cc
        ctx.set_tree(cnt, par, cod, np.zeros((B, G, N), np.float32))
        ctx.verify(o, ats.STRICT)
        d, f = spec.d_model, spec.d_ffn
        rows, tcap, xrows, ppu = (int(v) for v in ctx.debug_buffer(0, 16, np.int32, 4))
        T = B * G * N                                   # every slot of levels 1..G is forwarded
        self.T, self.rows, self.ppu = T, rows, ppu
        self.h = ctx.debug_buffer(0, 0, np.float32, T * d).reshape(T, d).astype(np.float64)
        self.x = _bf16_to_f64(ctx.debug_buffer(0, 1, np.uint16, T * d).reshape(T, d))
        self.q = _bf16_to_f64(ctx.debug_buffer(0, 2, np.uint16, T * d).reshape(T, d))
        self.att = _bf16_to_f64(ctx.debug_buffer(0, 3, np.uint16, T * d).reshape(T, d))
        self.act = _bf16_to_f64(ctx.debug_buffer(0, 4, np.uint16, T * f).reshape(T, f))
        kc = ctx.debug_buffer(0, 5, np.uint16, c * rows * d).reshape(c, rows, d)
        vc = ctx.debug_buffer(0, 6, np.float16, c * rows * d).reshape(c, rows, d)
        self.kc, self.vc = kc, vc                       # all layers (raw bits / fp16)
        self.logits = ctx.debug_buffer(0, 7, np.float32, (B + T) * 1024).reshape(B + T, 1024)[B:]
        self.tok = ctx.debug_buffer(0, 11, np.int32, T)
        self.pos = ctx.debug_buffer(0, 12, np.int32, T)
        self.kvrow = ctx.debug_buffer(0, 13, np.int32, T)
        self.anc = ctx.debug_buffer(0, 14, np.int32, 4 * T).reshape(T, 4)
        self.ancn = ctx.debug_buffer(0, 15, np.int32, T)
        ctx.close()


def _run_case(ats, cfg, n_layers, prompts, K, N, G, items_n, seed_tree=5):
    w = synth.workload(cfg)
    base = w.target
    spec = synth.ModelSpec(n_layers, base.d_model, base.n_heads, base.d_ffn, base.vocab)
    tw = synth.model_weights(spec, w.seed, "target")
    tw_dev = ats.weights_to_device(tw)
    items = synth.make_items(items_n, w.code_dist, w.zipf_a, w.seed)
    B = len(prompts)
    levels = [synth.random_tree(items, 0, 1, G, N, seed=seed_tree + u)[1] for u in range(B)]
    d, H, hd, f = spec.d_model, spec.n_heads, spec.head_dim, spec.d_ffn
    m = Model(spec, tw, w.code_base)
    cuts = [GpuCut(ats, spec, c, tw_dev, items, w.code_base, prompts, K, N, G, levels)
            for c in range(1, n_layers + 1)]
    T = cuts[0].T
    users = np.repeat(np.arange(B), G * N)
    print(f"\n{cfg}: {n_layers} layers, {B} user(s), T = {T} tree tokens, histories {[len(p) for p in prompts]}")
    for c in range(1, n_layers):   # shared layers: bit-identical caches and tables
        for l in range(c):
            a, b = cuts[c - 1], cuts[c]
            np.testing.assert_array_equal(a.kc[l, a.kvrow], b.kc[l, b.kvrow])
            np.testing.assert_array_equal(a.vc[l, a.kvrow], b.vc[l, b.kvrow])
    h_in = tw["embed"][cuts[0].tok].astype(np.float64)
    for l in range(n_layers):
        g = cuts[l]
        print(f" layer {l}")
        pos = g.pos.astype(np.int64)
        # ---- q, k, v from the GPU's residual
        q_ref, k_ref, v_ref = _layer_pre_attn(m, l, h_in, pos)
        # GEMM input g * h (bf16; the fp32 product rounds first), output times the norm scale
        # s(h), which the GPU sums in fp32 from per-tile partial sums (relative error < 2^-18)
        xgr = h_in * m.W(f"layers.{l}.attn_norm")
        xg = bf16(xgr)
        rs = rms_scale(h_in, spec.rms_eps)
        W = np.asarray(tw[f"layers.{l}.wqkv"], np.float32)
        Wa = np.abs(W)
        mag = (np.abs(xg).astype(np.float32) @ Wa.T).astype(np.float64)
        slack = 4 * U32 * np.sqrt(d) * mag
        slack += (_flip_risk(xgr, 2.0 ** -23) * _ulp(xgr)).astype(np.float32) @ Wa.T
        slack = slack * rs + 2.0 ** -18 * mag * rs
        ang = rope_angles(pos, hd, spec.rope_theta)
        cs, sn = np.abs(np.cos(ang))[:, None, :], np.abs(np.sin(ang))[:, None, :]

        def rot_slack(s):
            s = s.reshape(T, H, hd)
            a, b = s[..., :hd // 2], s[..., hd // 2:]
            return np.concatenate([a * cs + b * sn, b * cs + a * sn], axis=-1).reshape(T, d)
        sq, sk, sv = slack[:, :d], slack[:, d:2 * d], slack[:, 2 * d:]
        _check_bf16("q", g.q, q_ref.reshape(T, d), rot_slack(sq))
        k_gpu = _bf16_to_f64(g.kc[l, g.kvrow])
        v_gpu = g.vc[l, g.kvrow].astype(np.float64)
        _check_bf16("k", k_gpu, k_ref.reshape(T, d), rot_slack(sk))
        _check_bf16("v", v_gpu, v_ref.reshape(T, d), sv)
        # ---- tree attention from the GPU's q and K/V cache
        qg = g.q.reshape(T, H, hd)
        o_ref = np.zeros((T, H, hd))
        pv_scale = np.zeros((T, H, hd))
        for u in range(B):
            ri = np.nonzero(users == u)[0]
            P = len(prompts[u])
            prow = u * g.ppu * 64 + np.arange(P)
            Kp = _bf16_to_f64(g.kc[l, prow]).reshape(P, H, hd)
            Vp = g.vc[l, prow].astype(np.float64).reshape(P, H, hd)
            for i in ri:
                pr = g.anc[i, :g.ancn[i]]
                Kt = np.concatenate([Kp, _bf16_to_f64(g.kc[l, pr]).reshape(-1, H, hd)])
                Vt = np.concatenate([Vp, g.vc[l, pr].astype(np.float64).reshape(-1, H, hd)])
                o_ref[i] = _attend(qg[i:i + 1], Kt, Vt, None)[0]
                s = np.einsum("hd,mhd->hm", qg[i], Kt) / np.sqrt(hd)
                p = np.exp(s - s.max(axis=1, keepdims=True))
                pv_scale[i] = np.einsum("hm,mhd->hd", p, np.abs(Vt)) / p.sum(axis=1, keepdims=True)
        _check_bf16("attention", g.att, bf16(o_ref).reshape(T, d), 2.0 ** -10 * pv_scale.reshape(T, d))
        # ---- O projection, RMSNorm, gate/up and SwiGLU from the GPU's attention output
        h_mid, a_ref = _layer_mlp_act(m, l, h_in, g.att)
        Wo = np.abs(np.asarray(tw[f"layers.{l}.wo"], np.float32))
        dh_mid = 4 * U32 * np.sqrt(d) * (np.abs(g.att).astype(np.float32) @ Wo.T).astype(np.float64)
        gn = m.W(f"layers.{l}.mlp_norm")
        x2r = h_mid * gn
        rs = rms_scale(h_mid, spec.rms_eps)
        # the GPU's residual carries the O projection's fp32 error dh_mid: into g * h, and into s(h)
        rel = (dh_mid * np.abs(gn)) / np.maximum(np.abs(x2r), 1e-30) + 2.0 ** -20
        rel_rs = np.sum(np.abs(h_mid) * dh_mid, axis=-1, keepdims=True) / np.sum(h_mid * h_mid, axis=-1, keepdims=True)
        x2 = bf16(x2r)
        Wgu = np.abs(np.asarray(tw[f"layers.{l}.wgate_up"], np.float32))
        mag = (np.abs(x2).astype(np.float32) @ Wgu.T).astype(np.float64)
        acc = 4 * U32 * np.sqrt(d) * mag
        acc += (_flip_risk(x2r, rel) * _ulp(x2r)).astype(np.float32) @ Wgu.T
        acc = acc * rs + (2.0 ** -18 + rel_rs) * mag * rs
        gu = (x2.astype(np.float32) @ np.asarray(tw[f"layers.{l}.wgate_up"], np.float32).T).astype(np.float64) * rs
        gg, uu = gu[:, :f], gu[:, f:]
        sg = 1.0 / (1.0 + np.exp(-gg))
        dsilu = sg * (1.0 + gg * (1.0 - sg))
        act_slack = np.abs(dsilu * uu) * acc[:, :f] + np.abs(silu(gg)) * acc[:, f:] + 1e-6 * np.abs(silu(gg) * uu)
        _check_bf16("swiglu", g.act, a_ref, act_slack)
        # ---- down projection into the residual from the GPU's SwiGLU product
        h_out = _layer_mlp_out(m, l, h_mid, g.act)
        dh = np.abs(g.h - h_out)
        print(f"  residual   max |d| {dh.max():.3g} (mean {dh.mean():.3g})")
        assert dh.max() <= 2e-2
        h_in = g.h
        m.drop_cache()
    # ---- final RMSNorm and item-code logits from the GPU's final residual
    g = cuts[-1]
    xr = rmsnorm(g.h, m.W("final_norm"), spec.rms_eps)
    _check_bf16("final norm", g.x, bf16(xr), _flip_risk(xr, 2.0 ** -20) * _ulp(xr))
    dl = np.abs(g.logits - final_hidden_to_logits(m, g.h))
    print(f"  logits     max |d| {dl.max():.3g} (mean {dl.mean():.3g})")
    assert dl.max() <= 2e-2
    m.drop_cache()


def test_lockstep_mid_one_user(ats):
    """Mid shape (d 2048, 32 heads of 64, FFN 5632), 2 layers, 256-token history, T = 120 (one
    128-token tile)."""
    w = synth.workload("mid")
    prompts = synth.make_prompts(1, w.prompt_len, w.target.vocab, w.seed)
    _run_case(ats, "mid", 2, prompts, 10, 40, 3, 5000)


def test_lockstep_7b_one_user(ats):
    """7B shape (d 4096, 32 heads of 128, FFN 11008), 2 layers, 512-token history, T = 120."""
    w = synth.workload("7b")
    prompts = synth.make_prompts(1, w.prompt_len, w.target.vocab, w.seed)
    _run_case(ats, "7b", 2, prompts, 10, 40, 3, 5000)


def test_lockstep_mid_three_ragged_users(ats):
    """Three users with ragged histories (256, 131, 200 tokens) in one call: T = 360 tree tokens,
    so the 256-token tile (two token tiles), per-user page tables, query tiles and attention
    splits all run."""
    w = synth.workload("mid")
    rng = np.random.default_rng(41)
    prompts = [rng.integers(0, w.target.vocab, size=n).astype(np.int32) for n in (256, 131, 200)]
    _run_case(ats, "mid", 2, prompts, 10, 40, 3, 5000)


def test_lockstep_7b_sixteen_users(ats):
    """The 16-user workload's shape: 7B, 2 layers, K 20, N 80, 3 drafted levels (T = 3 840 tree
    tokens, fifteen 256-token tiles), histories of 256..1024 tokens."""
    w = synth.workload("7b_b16")
    prompts = synth.make_prompts(16, w.prompt_len, w.target.vocab, w.seed)
    _run_case(ats, "7b_b16", 2, prompts, 20, 80, 3, 20000)
