"""Operator-level parity of the CUDA kernels against the oracle / plain fp64 references, through the
C ABI: tcgen05 GEMM (plain, accumulate, SwiGLU; ragged shapes, stream-K split tiles, the 7B
shapes), RMSNorm, and shared-prefix tree attention over a paged cache with path keys."""
import numpy as np
import pytest
import torch

import synth
from oracle.model import _attend
from oracle.numerics import bf16, rmsnorm, silu

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ats():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2410_05165_gb300 as m
    return m


def _bf16_tensor(shape, seed, std=1.0):
    a = synth.normal_bf16(seed, 77, int(np.prod(shape)), std).reshape(shape)
    return a, torch.from_numpy(a).cuda().to(torch.bfloat16)


def _x_rows(T):
    return ((T + 255) // 256) * 256


@pytest.mark.parametrize("M,K,T", [(384, 128, 20), (1000, 256, 130), (192, 64, 1), (4096, 4096, 120),
                                   (1024, 2048, 300), (12288, 4096, 120), (4096, 11008, 120), (640, 512, 128),
                                   (256, 1024, 129)])
def test_gemm_matches_fp64(ats, M, K, T):
    W, Wt = _bf16_tensor((M, K), 1 + M + K)
    X, Xt = _bf16_tensor((_x_rows(T), K), 2 + T)
    Y = ats.op_gemm(Wt, Xt, T)
    torch.cuda.synchronize()
    ref = X[:T].astype(np.float64) @ W.astype(np.float64).T
    got = Y.cpu().numpy()
    err = np.abs(got - ref)
    tol = 1e-5 * np.sqrt(K) * np.abs(W).max() * np.abs(X).max() * 4 + 1e-6
    assert err.max() <= tol, (err.max(), tol)


def test_gemm_accumulate_and_determinism(ats):
    M, K, T = 4096, 4096, 64
    W, Wt = _bf16_tensor((M, K), 11)
    X, Xt = _bf16_tensor((_x_rows(T), K), 12)
    Y0 = torch.randn(T, M, device="cuda", dtype=torch.float32)
    Y = Y0.clone()
    ats.op_gemm(Wt, Xt, T, Y=Y, accumulate=True)
    ref = Y0.cpu().numpy().astype(np.float64) + X[:T].astype(np.float64) @ W.astype(np.float64).T
    assert np.abs(Y.cpu().numpy() - ref).max() < 1e-2
    # bitwise reproducible (fixed split-K summation order)
    a = ats.op_gemm(Wt, Xt, T).cpu().numpy()
    b = ats.op_gemm(Wt, Xt, T).cpu().numpy()
    np.testing.assert_array_equal(a, b)


def test_gemm_token_columns_are_batch_invariant(ats):
    """A token's output does not depend on which other tokens share the call."""
    M, K = 4096, 4096
    W, Wt = _bf16_tensor((M, K), 21)
    X, Xt = _bf16_tensor((256, K), 22)
    full = ats.op_gemm(Wt, Xt, 120).cpu().numpy()
    few = ats.op_gemm(Wt, Xt, 10).cpu().numpy()
    np.testing.assert_array_equal(full[:10], few)


@pytest.mark.parametrize("F,K,T", [(256, 64, 5), (512, 128, 20), (11008, 4096, 120), (1408, 512, 200)])
def test_swiglu_epilogue(ats, F, K, T):
    W, Wt = _bf16_tensor((2 * F, K), 31 + F, 0.02)
    X, Xt = _bf16_tensor((_x_rows(T), K), 32 + T)
    out = ats.op_gemm_swiglu(Wt, Xt, T).float().cpu().numpy()
    gu = X[:T].astype(np.float64) @ W.astype(np.float64).T
    ref = bf16(silu(gu[:, :F]) * gu[:, F:])
    err = np.abs(out - ref)
    # one bf16 ulp of the result, plus the fp32 accumulation error of g and u (absolute, ~1e-4 at
    # K = 4096) carried through the product where g or u nearly cancels
    g, u = gu[:, :F], gu[:, F:]
    assert np.all(err <= 2.0 ** -6 * np.abs(ref) + 1e-4 * (np.abs(g) + np.abs(u) + 1.0)), err.max()
    assert np.mean(err > 0) < 0.01


@pytest.mark.parametrize("T,d", [(1, 64), (37, 128), (120, 4096), (512, 2048)])
def test_rmsnorm(ats, T, d):
    rng = np.random.default_rng(T + d)
    h = (rng.standard_normal((T, d)) * 3).astype(np.float32)
    g, gt = _bf16_tensor((d,), 5 + d, 0.1)
    g = bf16(g + 1.0).astype(np.float32)
    gt = torch.from_numpy(g).cuda().to(torch.bfloat16)
    x = ats.op_rmsnorm(torch.from_numpy(h).cuda(), gt, 1e-6).float().cpu().numpy()
    ref = bf16(rmsnorm(h.astype(np.float64), g.astype(np.float64), 1e-6))
    err = np.abs(x - ref)
    assert np.all(err <= 2.0 ** -7 * np.abs(ref) + 1e-7)   # at most one bf16 ulp
    assert np.mean(err > 0) < 0.01


@pytest.mark.parametrize("H,hd,P,T", [(4, 32, 32, 20), (32, 128, 512, 120), (8, 64, 200, 70), (12, 64, 1, 3),
                                      (2, 32, 130, 65)])
def test_tree_attention(ats, H, hd, P, T):
    rng = np.random.default_rng(H * 1000 + P)
    d = H * hd
    pages_n = (P + 63) // 64
    rows = 64 * (pages_n * 2 + 4) + 64
    # scatter the prefix over non-contiguous pages
    page_ids = list(rng.permutation(pages_n * 2 + 4)[:pages_n])
    kc = bf16(rng.standard_normal((rows, d))).astype(np.float32)
    vc = bf16(rng.standard_normal((rows, d))).astype(np.float32)
    q = bf16(rng.standard_normal((T, d))).astype(np.float32)
    n_path = rng.integers(0, 5, size=T).astype(np.int32)
    path_rows = rng.integers(0, rows, size=(T, 4)).astype(np.int32)
    vis = np.full(T, P, np.int32)
    vis[: T // 3] = rng.integers(0, P + 1, size=T // 3)   # some causal-like partial visibility
    out = ats.op_attention(torch.from_numpy(q).cuda().to(torch.bfloat16),
                           torch.from_numpy(kc).cuda().to(torch.bfloat16),
                           torch.from_numpy(vc).cuda().to(torch.float16), H, hd, P, page_ids, vis, path_rows,
                           n_path).float().cpu().numpy()
    prefix_rows = np.array([64 * page_ids[p // 64] + p % 64 for p in range(P)], dtype=np.int64)
    for t in range(T):
        keys = np.concatenate([prefix_rows[: vis[t]], path_rows[t, : n_path[t]]]).astype(np.int64)
        if keys.size == 0:
            assert np.all(out[t] == 0)
            continue
        Kt = kc[keys].reshape(-1, H, hd).astype(np.float64)
        Vt = vc[keys].reshape(-1, H, hd).astype(np.float64)
        qt = q[t].reshape(1, H, hd).astype(np.float64)
        ref = _attend(qt, Kt, Vt, None)[0].reshape(-1)
        # fp32 scores and softmax; P rounded to fp16 (unit roundoff 2^-11) for P V, so
        # |d o| <= 2^-11 * sum_k p_k |v_k| / sum_k p_k; then the final bf16 rounding of o (one ulp)
        mag = _attend(qt, Kt, np.abs(Vt), None)[0].reshape(-1)
        tol = 2.0 ** -7 * np.abs(ref) + 2.0 ** -11 * mag + 1e-6
        assert np.all(np.abs(out[t] - ref) <= tol), (t, (np.abs(out[t] - ref) - tol).max())
