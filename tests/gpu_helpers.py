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
