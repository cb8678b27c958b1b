"""Float64 reference of the randomized method the library uses for the
projector refresh (test infrastructure only, like the rest of ``oracle/``).

The paper refreshes the projector with TruncatedSVD(V, r) (Algorithm 1); the
exact definition is ``moara_ref.truncated_svd``.  The library computes it
approximately by randomized subspace iteration -- its own choice of method,
after Halko, Martinsson and Tropp, "Finding structure with randomness"
(SIAM Review 53, 2011), Algorithm 4.4 (randomized subspace iteration) followed
by a Rayleigh-Ritz step (their Algorithm 5.1 in the form "SVD of Q^T V").
This module restates that method in float64 so that tests can separate two
questions: does the device compute what the method computes (compare with
``randomized_projector``), and how far is the method from the exact top-r
subspace (compare ``randomized_projector`` with ``truncated_svd``).

Steps, for V (m x n), rank r, oversampling p, power iterations q:

1. Omega (n x l), l = min(r + p, min(m, n)): standard normals from
   Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11), the counter-based
   generator the library also uses, turned into normals by Box-Muller.
2. Q = orth(V Omega).
3. q times:  Z = orth(V^T Q);  Q = orth(V Z).
4. Rayleigh-Ritz: Z = V^T Q, C = Z^T Z (l x l), X = eigenvectors of C by
   decreasing eigenvalue; P = Q X[:, :r].
5. Sign convention of ``moara_ref.fix_signs``.

``orth`` is any orthonormal basis of the column span (here a Householder QR);
the span, not the basis, is what each step passes on.
"""

from __future__ import annotations

import numpy as np

from . import moara_ref as o

# Philox4x32-10 constants (Salmon et al., SC'11): round multipliers and the
# Weyl increments of the key schedule.
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
MASK32 = 0xFFFFFFFF


def philox4x32_10(ctr, key):
    """Philox4x32 with 10 rounds.  ctr: uint64 array (..., 4) of 32-bit words,
    key: two 32-bit words.  Each round multiplies words 0 and 2 by M0 and M1
    (64-bit products split into high and low halves) and mixes: new words =
    (hi(M1 c2) ^ c1 ^ k0, lo(M1 c2), hi(M0 c0) ^ c3 ^ k1, lo(M0 c0)); the key
    then advances by the Weyl increments."""
    c = np.asarray(ctr, dtype=np.uint64) & MASK32
    k0, k1 = int(key[0]) & MASK32, int(key[1]) & MASK32
    for _ in range(10):
        p0 = c[..., 0] * np.uint64(PHILOX_M0)
        p1 = c[..., 2] * np.uint64(PHILOX_M1)
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(MASK32)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(MASK32)
        c = np.stack([hi1 ^ c[..., 1] ^ np.uint64(k0), lo1, hi0 ^ c[..., 3] ^ np.uint64(k1), lo0], axis=-1)
        k0 = (k0 + PHILOX_W0) & MASK32
        k1 = (k1 + PHILOX_W1) & MASK32
    return c


def sketch_key(seed: int, module_id: int, refresh_count: int) -> tuple[int, int]:
    """The 64-bit key of one module's sketch at one refresh (the library's
    stream assignment: seed mixed with the module id and the refresh count by
    odd 64-bit constants), as two 32-bit words (low, high)."""
    m64 = (1 << 64) - 1
    k = (seed ^ ((0x9E3779B97F4A7C15 * (module_id + 1)) & m64) ^ ((refresh_count * 0xD1B54A32D192ED03) & m64)) & m64
    return k & MASK32, k >> 32


def gaussian_sketch(rows: int, cols: int, key) -> np.ndarray:
    """rows x cols standard normals, row-major element e = i * cols + j: group
    g = e // 4 uses counter (g_lo, g_hi, 0x4D6F4152, 0x52616E64); its four words
    give uniforms u = (x >> 8 + 1) 2^-24 in (0, 1], and Box-Muller turns
    (u1, u2), (u3, u4) into (R1 cos 2 pi u2, R1 sin 2 pi u2, R3 cos 2 pi u4,
    R3 sin 2 pi u4) with R = sqrt(-2 ln u)."""
    count = rows * cols
    groups = (count + 3) // 4
    g = np.arange(groups, dtype=np.uint64)
    ctr = np.stack([g & np.uint64(MASK32), g >> np.uint64(32),
                    np.full_like(g, 0x4D6F4152), np.full_like(g, 0x52616E64)], axis=-1)
    w = philox4x32_10(ctr, key)
    u = ((w >> np.uint64(8)).astype(np.float64) + 1.0) * 2.0 ** -24
    ra = np.sqrt(-2.0 * np.log(u[:, 0]))
    rb = np.sqrt(-2.0 * np.log(u[:, 2]))
    z = np.stack([ra * np.cos(2 * np.pi * u[:, 1]), ra * np.sin(2 * np.pi * u[:, 1]),
                  rb * np.cos(2 * np.pi * u[:, 3]), rb * np.sin(2 * np.pi * u[:, 3])], axis=-1)
    return z.reshape(-1)[:count].reshape(rows, cols)


def _orth(Y):
    q, _ = np.linalg.qr(Y)
    return q


def randomized_projector(X, r: int, p: int, q: int, key) -> np.ndarray:
    """Steps 1-5 above for X (m x n); returns P (m x r) with orthonormal
    columns in decreasing Rayleigh quotient order, signed like
    ``moara_ref.truncated_svd``."""
    X = np.asarray(X, dtype=np.float64)
    m, n = X.shape
    l = min(r + p, min(m, n))
    Q = _orth(X @ gaussian_sketch(n, l, key))
    for _ in range(q):
        Z = _orth(X.T @ Q)
        Q = _orth(X @ Z)
    Z = X.T @ Q
    w, U = np.linalg.eigh(Z.T @ Z)
    order = np.argsort(-w, kind="stable")
    P = Q @ U[:, order[:r]]
    return o.fix_signs(P)


def captured_energy(P, X) -> float:
    """||P^T X||_F^2, the energy of X that span(P) captures."""
    return float(np.sum((np.asarray(P).T @ np.asarray(X, dtype=np.float64)) ** 2))
