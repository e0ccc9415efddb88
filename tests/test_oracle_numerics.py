"""Pins for oracle.numerics and oracle.philox against closed forms, library routines and
published known-answer vectors."""
import os

import numpy as np
import pytest
import torch

from oracle.numerics import bf16, rms_scale, rmsnorm, rope, silu
from oracle.philox import (draw_u32, gumbel, philox4x32_10, u_accept, u_open)

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def test_bf16_matches_torch_rne():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000),
                        [0.0, 1.0, -1.0, 1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8)]]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(bf16(x.astype(np.float64)), ref)


def test_bf16_ties_to_even():
    assert bf16(1 + 2 ** -8) == 1.0               # halfway, even neighbour is 1.0
    assert bf16(1 + 3 * 2 ** -8) == 1 + 2 ** -6    # halfway, even neighbour is above
    assert bf16(1 + 2 ** -8 + 2 ** -20) == 1 + 2 ** -7


def test_rmsnorm_closed_form():
    h = np.full((3, 64), -2.5)
    g = np.linspace(0.5, 1.5, 64)
    out = rmsnorm(h, g, 1e-6)
    np.testing.assert_allclose(out, np.broadcast_to(-2.5 / np.sqrt(6.25 + 1e-6) * g[None, :], out.shape), rtol=1e-15)
    # torch's rms_norm as an independent routine
    x = np.random.default_rng(1).standard_normal((5, 32))
    ref = torch.nn.functional.rms_norm(torch.from_numpy(x), (32,), torch.from_numpy(g[:32]), eps=1e-6).numpy()
    np.testing.assert_allclose(rmsnorm(x, g[:32], 1e-6), ref, rtol=1e-12)


def test_rms_scale_closed_form():
    """RMSNorm's per-row scale alone: exact values, and times h it is torch's gain-free rms_norm."""
    np.testing.assert_array_equal(rms_scale(np.array([[2.0, -2.0], [1.0, 1.0]]), 0.0), [[0.5], [1.0]])
    np.testing.assert_allclose(rms_scale(np.array([[3.0, 4.0]]), 0.0), [[1.0 / np.sqrt(12.5)]], rtol=1e-15)
    x = np.random.default_rng(2).standard_normal((4, 48))
    ref = torch.nn.functional.rms_norm(torch.from_numpy(x), (48,), None, eps=1e-6).numpy()
    np.testing.assert_allclose(x * rms_scale(x, 1e-6), ref, rtol=1e-12)


def test_rope_identity_norm_and_relative_position():
    rng = np.random.default_rng(2)
    q = rng.standard_normal((1, 2, 16))
    k = rng.standard_normal((1, 2, 16))
    np.testing.assert_allclose(rope(q, np.array([0]), 1e4), q, rtol=0, atol=0)
    r = rope(q, np.array([37]), 1e4)
    # rotation of pairs (i, i + hd/2) preserves each pair's norm
    n0 = q[..., :8] ** 2 + q[..., 8:] ** 2
    n1 = r[..., :8] ** 2 + r[..., 8:] ** 2
    np.testing.assert_allclose(n0, n1, rtol=1e-12)
    # <rope(q, m), rope(k, n)> depends only on m - n
    a = np.sum(rope(q, np.array([10]), 1e4) * rope(k, np.array([3]), 1e4))
    b = np.sum(rope(q, np.array([107]), 1e4) * rope(k, np.array([100]), 1e4))
    np.testing.assert_allclose(a, b, rtol=1e-10)
    # pair (0, hd/2) rotates by exactly pos radians (frequency theta^0 = 1)
    e = np.zeros((1, 1, 16)); e[0, 0, 0] = 1.0
    r = rope(e, np.array([0.75]), 1e4)
    np.testing.assert_allclose([r[0, 0, 0], r[0, 0, 8]], [np.cos(0.75), np.sin(0.75)], rtol=1e-14)


def test_silu_library():
    x = np.linspace(-20, 20, 101)
    np.testing.assert_allclose(silu(x), torch.nn.functional.silu(torch.from_numpy(x)).numpy(), rtol=1e-12)


def test_philox_weyl_constants_closed_form():
    # the key schedule adds the fixed-point fractions of the golden ratio and of sqrt(3) - 1 (SC'11)
    from oracle.philox import W0, W1
    assert W0 == int(np.floor(2.0 ** 32 * (np.sqrt(5.0) - 1.0) / 2.0))
    assert W1 == int(np.floor(2.0 ** 32 * (np.sqrt(3.0) - 1.0)))


def _philox_inverse(x, k0, k1):
    """Undo the 10 rounds, written from the round definition: (c0, c1, c2, c3) ->
    (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2), hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)).  lo(M*c) determines c
    because M is odd."""
    from oracle.philox import M0, M1, W0, W1
    inv0, inv1 = pow(M0, -1, 2 ** 32), pow(M1, -1, 2 ** 32)
    keys = []
    a, b = k0, k1
    for r in range(10):
        if r:
            a, b = (a + W0) & 0xFFFFFFFF, (b + W1) & 0xFFFFFFFF
        keys.append((a, b))
    y0, y1, y2, y3 = (int(v) for v in x)
    for a, b in reversed(keys):
        c2 = (y1 * inv1) & 0xFFFFFFFF
        c0 = (y3 * inv0) & 0xFFFFFFFF
        c1 = y0 ^ ((M1 * c2) >> 32) ^ a
        c3 = y2 ^ ((M0 * c0) >> 32) ^ b
        y0, y1, y2, y3 = c0, c1, c2, c3
    return y0, y1, y2, y3


# An independent Philox4x32-10: the one in Triton's language library (tl.philox), run by Triton's
# CPU interpreter in a child process (the interpreter is chosen by an environment variable read at
# import).  It fixes the round multipliers, which the inversion test below cannot (it inverts with
# the oracle's own multipliers), and the whole round and key schedule of Salmon et al. (SC'11).
_TRITON_PHILOX = r"""
import json, os, sys
os.environ["TRITON_INTERPRET"] = "1"
import torch, triton, triton.language as tl

@triton.jit
def kern(c_ptr, k_ptr, o_ptr, N: tl.constexpr):
    i = tl.arange(0, N)
    seed = (tl.load(k_ptr + 2 * i + 1).to(tl.uint64) << 32) | tl.load(k_ptr + 2 * i).to(tl.uint64)
    r0, r1, r2, r3 = tl.philox(seed, tl.load(c_ptr + 4 * i), tl.load(c_ptr + 4 * i + 1),
                               tl.load(c_ptr + 4 * i + 2), tl.load(c_ptr + 4 * i + 3), 10)
    tl.store(o_ptr + 4 * i, r0)
    tl.store(o_ptr + 4 * i + 1, r1)
    tl.store(o_ptr + 4 * i + 2, r2)
    tl.store(o_ptr + 4 * i + 3, r3)

rows = json.load(sys.stdin)
n = len(rows)
c = torch.tensor([x for r in rows for x in r[:4]], dtype=torch.int64).to(torch.int32)
k = torch.tensor([x for r in rows for x in r[4:]], dtype=torch.int64).to(torch.uint32)
o = torch.zeros(4 * n, dtype=torch.int32)
kern[(1,)](c, k, o, N=n)
print(json.dumps([x & 0xFFFFFFFF for x in o.tolist()]))
"""


def test_philox_matches_triton_library():
    import json
    import subprocess
    import sys
    pytest.importorskip("triton")
    rng = np.random.default_rng(17)
    rows = [[0] * 6, [0xFFFFFFFF] * 6, [1, 2, 3, 4, 5, 6]]
    rows += [[int(v) for v in rng.integers(0, 2 ** 32, size=6, dtype=np.uint64)] for _ in range(125)]
    r = subprocess.run([sys.executable, "-c", _TRITON_PHILOX], input=json.dumps(rows), capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lib = np.array(json.loads(r.stdout.strip().splitlines()[-1]), dtype=np.uint64).reshape(-1, 4)
    ours = np.stack([np.array([int(x) for x in philox4x32_10(*row)], dtype=np.uint64) for row in rows])
    np.testing.assert_array_equal(ours, lib)


def test_philox_inverts_to_its_counter():
    rng = np.random.default_rng(5)
    for _ in range(200):
        c = [int(v) for v in rng.integers(0, 2 ** 32, size=4, dtype=np.uint64)]
        k0, k1 = (int(v) for v in rng.integers(0, 2 ** 32, size=2, dtype=np.uint64))
        out = philox4x32_10(*c, k0, k1)
        assert list(_philox_inverse(out, k0, k1)) == c


def test_philox_no_collisions_and_avalanche():
    n = 1 << 16
    out = philox4x32_10(np.arange(n), 0, 0, 0, 1, 2)
    words = np.stack(out, axis=1).astype(np.uint64)
    keys = (words[:, 0] << np.uint64(32)) | words[:, 1]
    assert np.unique(keys).size == n
    # flipping one counter bit flips about half of the 128 output bits
    a = np.stack(philox4x32_10(np.arange(4096), 7, 9, 11, 3, 4), axis=1)
    b = np.stack(philox4x32_10(np.arange(4096) ^ 1, 7, 9, 11, 3, 4), axis=1)
    flips = np.unpackbits((a ^ b).view(np.uint8), axis=1).sum(axis=1)
    assert abs(flips.mean() - 64) < 1.0


def test_philox_uniform_statistics():
    w = draw_u32(1234, 1, 2, 3, 4, np.arange(200000))
    u = u_accept(w)
    assert u.min() > 0 and u.max() <= 1.0
    assert abs(u.mean() - 0.5) < 4 * np.sqrt(1 / 12 / u.size)
    hist = np.bincount((w >> np.uint32(24)).astype(np.int64), minlength=256)
    e = u.size / 256
    chi2 = np.sum((hist - e) ** 2 / e)
    assert chi2 < 255 + 6 * np.sqrt(2 * 255)
    # every value is an exact multiple of 2**-24
    assert np.all(np.floor(u * 2 ** 24) == u * 2 ** 24)
    uo = u_open(w)
    assert uo.min() > 0 and uo.max() < 1


def test_philox_streams_differ():
    a = draw_u32(0, 0, 1, 0, 0, np.arange(64))
    b = draw_u32(0, 1, 1, 0, 0, np.arange(64))
    c = draw_u32(0, 0, 1, 0, 1, np.arange(64))
    assert not np.array_equal(a, b) and not np.array_equal(a, c)
    # word selection: draws 4i..4i+3 are the four outputs of one counter
    words = philox4x32_10(0, 1, 0, 0, 0, 0)
    np.testing.assert_array_equal(a[:4], np.array([int(x) for x in words], dtype=np.uint32))


def test_gumbel_moments():
    g = gumbel(draw_u32(7, 3, 1, 0, 0, np.arange(400000))).astype(np.float64)
    assert abs(g.mean() - 0.5772156649) < 4 * np.sqrt(np.pi ** 2 / 6 / g.size)
    assert abs(g.var() - np.pi ** 2 / 6) < 0.02
