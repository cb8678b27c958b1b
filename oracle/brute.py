"""Loop-only twin of the oracle for tiny matrices (TEST INFRASTRUCTURE ONLY).

Written independently of ``moara_ref`` (no NumPy arithmetic, no shared
helpers): explicit Python loops over lists of floats.  The truncated SVD is
replaced by the cyclic Jacobi eigenvalue method (Jacobi 1846; Golub & Van Loan,
Matrix Computations, §8.5) applied to X X^T, whose eigenvectors are the left
singular vectors of X.  Used only to pin the oracle on inputs of a few rows.

Same readings as the oracle: refresh when (t - 1) mod T == 0, Adam in the
torch.optim.Adam form, eigenvector columns signed so that their largest
magnitude entry is positive.
"""

from __future__ import annotations

import math


def _zeros(rows, cols):
    return [[0.0] * cols for _ in range(rows)]


def decompose(G, B, eps=1e-12):
    """Block magnitudes and directions of §3.1 / App. B.1 with loops."""
    m = len(G)
    n = len(G[0])
    k = (n + B - 1) // B
    M = _zeros(m, k)
    V = _zeros(m, n)
    for i in range(m):
        for b in range(k):
            ss = 0.0
            for c in range(b * B, (b + 1) * B):
                x = G[i][c] if c < n else 0.0       # zero padding
                ss += x * x
            mag = math.sqrt(ss)
            M[i][b] = mag
            for c in range(b * B, min((b + 1) * B, n)):   # cropped
                V[i][c] = G[i][c] / (mag + eps)
    return M, V


def jacobi_eigh(A, sweeps=100, tol=1e-30):
    """Cyclic Jacobi on a symmetric matrix: returns (eigenvalues, vectors).

    Each rotation zeroes A[p][q]; the product of rotations gives the
    eigenvectors as columns.
    """
    n = len(A)
    A = [row[:] for row in A]
    Q = _zeros(n, n)
    for i in range(n):
        Q[i][i] = 1.0
    for _ in range(sweeps):
        off = 0.0
        for p in range(n):
            for q in range(p + 1, n):
                off += A[p][q] * A[p][q]
        if off <= tol:
            break
        for p in range(n - 1):
            for q in range(p + 1, n):
                apq = A[p][q]
                if apq == 0.0:
                    continue
                theta = (A[q][q] - A[p][p]) / (2.0 * apq)
                tt = (1.0 if theta >= 0 else -1.0) / (abs(theta) + math.sqrt(theta * theta + 1.0))
                c = 1.0 / math.sqrt(tt * tt + 1.0)
                s = tt * c
                for k in range(n):          # A <- A J (columns p, q)
                    akp, akq = A[k][p], A[k][q]
                    A[k][p] = c * akp - s * akq
                    A[k][q] = s * akp + c * akq
                for k in range(n):          # A <- J^T A (rows p, q)
                    apk, aqk = A[p][k], A[q][k]
                    A[p][k] = c * apk - s * aqk
                    A[q][k] = s * apk + c * aqk
                for k in range(n):          # Q <- Q J
                    qkp, qkq = Q[k][p], Q[k][q]
                    Q[k][p] = c * qkp - s * qkq
                    Q[k][q] = s * qkp + c * qkq
    return [A[i][i] for i in range(n)], Q


def top_left_singular(X, r):
    """Top-r left singular vectors of X via Jacobi on X X^T, sign-fixed."""
    m = len(X)
    n = len(X[0])
    C = _zeros(m, m)
    for i in range(m):
        for j in range(m):
            acc = 0.0
            for c in range(n):
                acc += X[i][c] * X[j][c]
            C[i][j] = acc
    vals, vecs = jacobi_eigh(C)
    order = sorted(range(m), key=lambda j: -vals[j])[:r]
    P = _zeros(m, r)
    for jj, j in enumerate(order):
        big = 0
        for i in range(m):
            if abs(vecs[i][j]) > abs(vecs[big][j]):
                big = i
        sgn = -1.0 if vecs[big][j] < 0 else 1.0
        for i in range(m):
            P[i][jj] = sgn * vecs[i][j]
    return P


def _adam(g, mom1, mom2, t, b1, b2, eps):
    rows, cols = len(g), len(g[0])
    out = _zeros(rows, cols)
    for i in range(rows):
        for j in range(cols):
            mom1[i][j] = b1 * mom1[i][j] + (1.0 - b1) * g[i][j]
            mom2[i][j] = b2 * mom2[i][j] + (1.0 - b2) * g[i][j] * g[i][j]
            mhat = mom1[i][j] / (1.0 - b1 ** t)
            vhat = mom2[i][j] / (1.0 - b2 ** t)
            out[i][j] = mhat / (math.sqrt(vhat) + eps)
    return out


def run(W, grads, r, lr, B, T, beta1=0.9, beta2=0.999, adam_eps=1e-6,
        scale=0.25, decompose_on=True, refresh_src="V", P=None,
        auto_refresh=True):
    """Run len(grads) steps of Algorithm 1 on one weight; returns (W, P)."""
    m = len(W)
    n = len(W[0])
    k = (n + B - 1) // B
    W = [row[:] for row in W]
    P = [row[:] for row in P] if P is not None else _zeros(m, r)
    ea, eas = _zeros(r, n), _zeros(r, n)
    ma, mas = _zeros(m, k), _zeros(m, k)
    for idx, G in enumerate(grads):
        t = idx + 1
        if decompose_on:
            M, V = decompose(G, B)
        else:
            M, V = None, G
        if auto_refresh and (t - 1) % T == 0:
            P = top_left_singular(V if refresh_src == "V" else G, r)
        R = _zeros(r, n)
        for a in range(r):
            for j in range(n):
                acc = 0.0
                for i in range(m):
                    acc += P[i][a] * V[i][j]
                R[a][j] = acc
        Nn = _adam(R, ea, eas, t, beta1, beta2, adam_eps)
        dM = _adam(M, ma, mas, t, beta1, beta2, adam_eps) if decompose_on else None
        for i in range(m):
            for j in range(n):
                acc = 0.0
                for a in range(r):
                    acc += P[i][a] * Nn[a][j]
                mult = dM[i][j // B] if decompose_on else 1.0
                W[i][j] -= lr * scale * mult * acc
    return W, P
