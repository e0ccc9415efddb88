"""The allocation-free GEMM entry point (atspeed_op_gemm_noalloc) against the ordinary one.

Some callers cannot allocate device memory: code that must not allocate while a stream is being
captured, serving loops that run inside a fixed, pre-reserved memory budget, and hosts whose device
memory belongs to another allocator.  They call atspeed_op_gemm_noalloc, whose split-K scratch is a
static device array of the library.  Two calls in a row with different data (the second one finds
the first one's partial sums and counters in that array) must each give what atspeed_op_gemm gives,
within the GEMM tolerance of the other parity tests, and leave the scratch's error word clear.
This file is collected last so that a run that stops at the first failure has run every other test
already."""
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


# (M, K, T) on the entry point's 32-CTA grid:
#   4096 x 4096 x 120: 32 tiles, one whole tile per CTA (no split);
#   1000 x 256 x 130: 8 tiles of 4 k-blocks, a ragged last weight tile, two token tiles' worth of T;
#   1000 x 4096 x 300: 16 tiles (BN = 256, two token tiles) of 64 k-blocks, every tile split over
#     two CTAs (stream-K), partial sums through the static array;
#   5120 x 4096 x 120: 40 tiles, one whole tile per CTA plus 8 tiles split four ways.
SHAPES = [(4096, 4096, 120), (1000, 256, 130), (1000, 4096, 300), (5120, 4096, 120)]


@pytest.mark.parametrize("M,K,T", SHAPES)
def test_noalloc_gemm_matches_workspace_gemm_twice(ats, M, K, T):
    assert ats.op_status(noalloc=True) == 0          # nothing left over from earlier calls
    for call in range(2):                           # different data on each call
        seed = 100 * call + M % 97 + K % 89 + T
        W, Wt = _bf16((M, K), seed)
        X, Xt = _bf16((((T + 255) // 256) * 256, K), seed + 10)
        want = ats.op_gemm(Wt, Xt, T).cpu().numpy()
        got = ats.op_gemm_noalloc(Wt, Xt, T).cpu().numpy()
        ref = X[:T].astype(np.float64) @ W.astype(np.float64).T
        tol = 1e-5 * np.sqrt(K) * np.abs(W).max() * np.abs(X).max() * 4 + 1e-6
        assert np.abs(got - want).max() <= tol, (call, np.abs(got - want).max())
        assert np.abs(got - ref).max() <= tol, (call, np.abs(got - ref).max())
        assert ats.op_status(noalloc=True) == 0     # no bounded wait gave up
        assert ats.op_status() == 0


def test_noalloc_gemm_accumulates_and_refuses_oversize(ats):
    W, Wt = _bf16((512, 128), 5)
    X, Xt = _bf16((256, 128), 6)
    Y0 = torch.randn(7, 512, device="cuda")
    Y = ats.op_gemm_noalloc(Wt, Xt, 7, Y=Y0.clone(), accumulate=True).cpu().numpy()
    ref = Y0.cpu().numpy().astype(np.float64) + X[:7].astype(np.float64) @ W.astype(np.float64).T
    assert np.abs(Y - ref).max() < 1e-3
    # more than 4096 output tiles, and K above 16384, are refused with E_SHAPE before any launch
    big = torch.zeros(4096 * 128 + 128, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ats.AtSpeedError) as e:
        ats.op_gemm_noalloc(big, Xt[:, :64].contiguous(), 1)
    assert e.value.status == ats.E_SHAPE
    wide = torch.zeros(128, 16384 + 64, dtype=torch.bfloat16, device="cuda")
    xw = torch.zeros(128, 16384 + 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ats.AtSpeedError) as e:
        ats.op_gemm_noalloc(wide, xw, 1)
    assert e.value.status == ats.E_SHAPE
    assert ats.op_status(noalloc=True) == 0
