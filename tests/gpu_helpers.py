"""Shared helpers of the GPU tests: run the oracle and the library on the same
seeded inputs and measure their disagreement."""

import numpy as np

import synth
from oracle import moara_ref as o


def rel_err(got, ref):
    """max |got - ref| / max |ref|  (the relative error of W)."""
    return float(np.max(np.abs(got - ref)) / np.max(np.abs(ref)))


def delta_err(got, ref, W0):
    """||dW_got - dW_ref||_F / ||dW_ref||_F with dW = W_final - W0."""
    d_ref = ref - W0
    return float(np.linalg.norm((got - W0) - d_ref) / max(np.linalg.norm(d_ref), 1e-300))


def principal_angles(A, B):
    """Principal angles (radians) between span(A) and span(B), orthonormal columns."""
    s = np.linalg.svd(A.T @ B, compute_uv=False)
    return np.arccos(np.clip(s, -1.0, 1.0))


def gap_index(S, r, ratio=1.5):
    """Largest k <= r with S[k-1] / S[k] >= ratio (0 if none)."""
    best = 0
    for k in range(1, min(r, len(S) - 1) + 1):
        if S[k] > 0 and S[k - 1] / S[k] >= ratio:
            best = k
    return best


def make_inputs(shapes, B, steps, bf16, seed=0, sigma0=10.0, noise=0.01, noise_rel=True,
                signal_rank=8):
    """Per module: list of float64 grads (bf16- or fp32-representable) and W0."""
    grads, W0 = [], []
    for idx, (m, n, r) in enumerate(shapes):
        s = min(signal_rank, m, n)
        grads.append(synth.grads_for_steps(m, n, s, sigma0, noise, steps, seed=seed,
                                           module=idx, noise_rel=noise_rel, bf16=bf16))
        W0.append(synth.init_weight(m, n, seed=seed, module=idx))
    return grads, W0


def oracle_projector(G, r, B, decompose=True, src="V"):
    X = o.decompose(G, B)[1] if (decompose and src == "V") else G
    return o.truncated_svd(X, r)[0]


def top_subspace(X, r):
    """Top-r left singular vectors of X and all its squared singular values
    (decreasing), through the eigen-decomposition of the smaller Gram matrix:
    the same subspace as the SVD of TruncatedSVD, faster on tall weights."""
    X = np.asarray(X, dtype=np.float64)
    m, n = X.shape
    if m <= n:
        w, U = np.linalg.eigh(X @ X.T)
        w, U = w[::-1], U[:, ::-1]
        return U[:, :r], np.maximum(w, 0.0)
    w, Wv = np.linalg.eigh(X.T @ X)
    w, Wv = w[::-1], Wv[:, ::-1]
    U = X @ Wv[:, :r]
    U /= np.linalg.norm(U, axis=0)
    return U, np.maximum(w, 0.0)


def check_refresh(P, X, r, p, q, key, exact_bar=None, tol_angle=1e-2, rsi_slack=3e-4, rsi_frac=0.25):
    """Checks a device projector P (m x r) refreshed from X (m x n).

    * P^T P = I within 1e-5.
    * Principal angles <= tol_angle against the exact top subspace on the
      leading directions up to the spectral gap k_gap (largest k <= r with
      sigma_k / sigma_{k+1} >= 1.5).
    * Captured energy against the float64 randomized subspace iteration
      (oracle/rsi_ref.py) with the same Philox sketch, p and q: the device may
      lose at most rsi_slack of the optimum plus rsi_frac of the method's own
      deficit more (its Rayleigh-Ritz step takes a few orthogonal iterations
      instead of an exact eigensolve, and its intermediate iterates are bf16;
      the measured excess on the test shapes is 0.7e-4 to 7e-4).
    * With exact_bar: captured energy >= (1 - exact_bar) of the optimum
      sum_{i<=r} sigma_i^2 (exact TruncatedSVD).
    Returns the deficits (1 - energy / optimum) of the device and of the
    float64 method, k_gap, and max |P^T P - I|."""
    from oracle import rsi_ref as R
    P = np.asarray(P, dtype=np.float64)
    X = np.asarray(X, dtype=np.float64)
    orth = float(np.abs(P.T @ P - np.eye(r)).max())
    assert orth <= 1e-5, orth
    U, w = top_subspace(X, r)
    k = gap_index(np.sqrt(w), r)
    if k > 0:
        ang = principal_angles(P[:, :k], U[:, :k])
        assert ang.max() <= tol_angle, (k, ang.max())
    e_opt = float(np.sum(w[:r]))
    e_dev = R.captured_energy(P, X)
    e_rsi = R.captured_energy(R.randomized_projector(X, r, p, q, key), X)
    d_dev, d_rsi = 1.0 - e_dev / e_opt, 1.0 - e_rsi / e_opt
    assert e_dev >= e_rsi - (rsi_slack + rsi_frac * d_rsi) * e_opt, (d_dev, d_rsi)
    if exact_bar is not None:
        assert e_dev >= (1.0 - exact_bar) * e_opt, d_dev
    return {"k_gap": k, "deficit": d_dev, "deficit_rsi": d_rsi, "orth": orth}
