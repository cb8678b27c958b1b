"""CPU pins of the float64 restatement of the library's randomized refresh
(oracle/rsi_ref.py): the Philox4x32-10 generator against its published
known-answer vectors, the Gaussian sketch's Box-Muller mapping, and the
randomized projector against the exact TruncatedSVD where the two must agree
(a full sketch spans the whole column space; a clear spectral gap and enough
power iterations converge), Eckart-Young, and monotonicity in q."""

import os

import numpy as np
import pytest

from oracle import moara_ref as o
from oracle import rsi_ref as R

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        w = [int(x, 16) for x in line.split()]
        rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


def test_philox_known_answers():
    kat = _kat()
    assert len(kat) == 3
    for ctr, key, out in kat:
        got = R.philox4x32_10(np.array(ctr, dtype=np.uint64), key)
        assert [int(x) for x in got] == out


def test_philox_vectorised_matches_single():
    ctrs = np.array([[i, i >> 3, 7, 9] for i in range(10)], dtype=np.uint64)
    many = R.philox4x32_10(ctrs, (0x1234, 0x5678))
    for i in range(10):
        one = R.philox4x32_10(ctrs[i], (0x1234, 0x5678))
        assert [int(x) for x in one] == [int(x) for x in many[i]]


def test_sketch_box_muller_mapping():
    """Element e of the sketch comes from counter group e // 4: recompute the
    first group by hand from the generator's words."""
    key = (11, 22)
    Z = R.gaussian_sketch(3, 5, key)
    w = R.philox4x32_10(np.array([0, 0, 0x4D6F4152, 0x52616E64], dtype=np.uint64), key)
    u = [((int(x) >> 8) + 1) * 2.0 ** -24 for x in w]
    r1, r3 = np.sqrt(-2 * np.log(u[0])), np.sqrt(-2 * np.log(u[2]))
    want = [r1 * np.cos(2 * np.pi * u[1]), r1 * np.sin(2 * np.pi * u[1]),
            r3 * np.cos(2 * np.pi * u[3]), r3 * np.sin(2 * np.pi * u[3])]
    np.testing.assert_allclose(Z.reshape(-1)[:4], want, rtol=1e-15, atol=0)
    assert Z.shape == (3, 5)


def test_sketch_is_standard_normal():
    Z = R.gaussian_sketch(200, 250, R.sketch_key(0, 3, 1))
    assert abs(Z.mean()) < 0.01 and abs(Z.std() - 1.0) < 0.01
    # different module ids and refresh counts draw different streams
    assert not np.allclose(Z, R.gaussian_sketch(200, 250, R.sketch_key(0, 4, 1)))
    assert not np.allclose(Z, R.gaussian_sketch(200, 250, R.sketch_key(0, 3, 2)))


def test_full_sketch_equals_truncated_svd():
    """l = min(m, n): span(Q) is the whole column space and the
    Rayleigh-Ritz step is the exact SVD."""
    rng = np.random.default_rng(4)
    X = rng.standard_normal((40, 30)) * np.linspace(3, 1, 30)
    P = R.randomized_projector(X, 6, 100, 0, (1, 2))
    Pe, _ = o.truncated_svd(X, 6)
    np.testing.assert_allclose(P, Pe, atol=1e-10)


def test_clear_gap_converges_to_truncated_svd():
    rng = np.random.default_rng(5)
    m, n, r = 120, 90, 8
    U = np.linalg.qr(rng.standard_normal((m, n)))[0]
    W = np.linalg.qr(rng.standard_normal((n, n)))[0]
    s = np.concatenate([10 * 0.8 ** np.arange(r), 0.1 * 0.9 ** np.arange(n - r)])
    X = (U * s) @ W.T
    P = R.randomized_projector(X, r, 8, 4, (3, 4))
    Pe, _ = o.truncated_svd(X, r)
    np.testing.assert_allclose(P, Pe, atol=1e-8)


def test_eckart_young_and_more_iterations_help():
    """Captured energy never exceeds the sum of the top r squared singular
    values, and grows with the number of power iterations on a flat tail."""
    rng = np.random.default_rng(6)
    X = rng.standard_normal((150, 100))
    s = np.linalg.svd(X, compute_uv=False)
    best = np.sum(s[:20] ** 2)
    e = [R.captured_energy(R.randomized_projector(X, 20, 8, q, (9, 9)), X) for q in (0, 1, 3, 8)]
    assert all(x <= best * (1 + 1e-12) for x in e)
    assert e[0] < e[1] < e[2] < e[3]
    P = R.randomized_projector(X, 20, 8, 3, (9, 9))
    np.testing.assert_allclose(P.T @ P, np.eye(20), atol=1e-12)
