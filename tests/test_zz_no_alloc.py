"""The allocation-free GEMM entry point (atspeed_op_gemm_noalloc) against the ordinary one.

Callers that cannot allocate device memory (stream capture, fixed-budget serving loops, foreign
allocators) use atspeed_op_gemm_noalloc, whose split-K scratch is a static device array of the
library.  Two calls in a row (the second one finds the first one's leftovers in that array) must
give what atspeed_op_gemm gives, within the GEMM tolerance of the other parity tests.  This file is
collected last so that a run that stops at the first failure has run every other test already."""
import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ats():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2410_05165_gb300 as m
    return m


def _bf16(shape, seed):
    a = synth.normal_bf16(seed, 91, int(np.prod(shape)), 1.0).reshape(shape)
    return a, torch.from_numpy(a).cuda().to(torch.bfloat16)


def test_noalloc_gemm_matches_workspace_gemm_twice(ats):
    for (M, K, T), seed in (((4096, 4096, 120), 1), ((1000, 256, 130), 2)):
        W, Wt = _bf16((M, K), seed)
        X, Xt = _bf16((((T + 255) // 256) * 256, K), seed + 10)
        want = ats.op_gemm(Wt, Xt, T).cpu().numpy()
        got = ats.op_gemm_noalloc(Wt, Xt, T).cpu().numpy()
        ref = X[:T].astype(np.float64) @ W.astype(np.float64).T
        tol = 1e-5 * np.sqrt(K) * np.abs(W).max() * np.abs(X).max() * 4 + 1e-6
        assert np.abs(got - want).max() <= tol
        assert np.abs(got - ref).max() <= tol
    # accumulate into an existing output, and a too-large request is refused
    W, Wt = _bf16((512, 128), 5)
    X, Xt = _bf16((256, 128), 6)
    Y0 = torch.randn(7, 512, device="cuda")
    Y = ats.op_gemm_noalloc(Wt, Xt, 7, Y=Y0.clone(), accumulate=True).cpu().numpy()
    ref = Y0.cpu().numpy().astype(np.float64) + X[:7].astype(np.float64) @ W.astype(np.float64).T
    assert np.abs(Y - ref).max() < 1e-3
    big = torch.zeros(4096 * 128 + 128, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ats.AtSpeedError):
        ats.op_gemm_noalloc(big, Xt[:, :64].contiguous(), 1)
