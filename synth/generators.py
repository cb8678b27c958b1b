"""Seeded random inputs: low-rank-plus-noise gradients, weights, projectors.

Recipe (one module, m x n):
    G_t = sum_{i < s} sigma_i u_i v_i^T + nu * Z_t,  sigma_i = sigma0 * 0.7^i
u (m x s) and v (n x s) are Gaussian factors with orthonormalised columns,
drawn once from seed ``seed``; Z_t is standard Gaussian noise redrawn at every
step from the stream (seed, module index, step).  nu is ``noise`` or, with
``noise_rel``, noise * sigma0 / sqrt(n).  W_0 ~ N(0, 0.02^2).

NumPy's PCG64 drives the host generators; ``lowrank_grad_torch`` builds the
same recipe on a torch device for workloads too large for the host (its
values differ from the NumPy ones; both sides of a comparison then read the
same device tensor).
"""

from __future__ import annotations

import numpy as np


def _rng(*key):
    return np.random.Generator(np.random.PCG64(list(key)))


def _orthonormal_columns(X):
    q, rr = np.linalg.qr(X)
    # make the factorisation unique (positive diagonal of R)
    d = np.sign(np.diag(rr))
    d[d == 0] = 1.0
    return q * d


def lowrank_factors(m, n, s, seed=0, module=0):
    g = _rng(seed, module, 0xF00D)
    u = _orthonormal_columns(g.standard_normal((m, s)))
    v = _orthonormal_columns(g.standard_normal((n, s)))
    return u, v


def lowrank_grad(m, n, s, sigma0, noise, step, seed=0, module=0,
                 noise_rel=False, factors=None):
    """float64 (m x n) gradient of the recipe above at step ``step``."""
    u, v = factors if factors is not None else lowrank_factors(m, n, s, seed, module)
    sig = sigma0 * 0.7 ** np.arange(s)
    nu = noise * sigma0 / np.sqrt(n) if noise_rel else noise
    z = _rng(seed, module, 1 + step).standard_normal((m, n))
    return (u * sig) @ v.T + nu * z


def to_bf16_exact(x):
    """Round float64/float32 values to bfloat16 (nearest-even) and return them
    as float64, so that the bf16 tensor and its float64 copy hold the same
    numbers."""
    f = np.asarray(x, dtype=np.float32)
    bits = f.view(np.uint32).astype(np.uint64)
    lsb = (bits >> 16) & 1
    rounded = ((bits + 0x7FFF + lsb) >> 16) << 16
    out = rounded.astype(np.uint32).view(np.float32)
    nan = np.isnan(f)
    out = np.where(nan, np.float32(np.nan), out)
    return out.astype(np.float64)


def grads_for_steps(m, n, s, sigma0, noise, steps, seed=0, module=0,
                    noise_rel=False, bf16=False):
    """Gradients for steps 1..steps (list of float64 arrays)."""
    fac = lowrank_factors(m, n, s, seed, module)
    out = []
    for t in range(1, steps + 1):
        G = lowrank_grad(m, n, s, sigma0, noise, t, seed, module, noise_rel, fac)
        out.append(to_bf16_exact(G) if bf16 else G.astype(np.float32).astype(np.float64))
    return out


def init_weight(m, n, seed=0, module=0, std=0.02):
    """W_0 ~ N(0, std^2), returned as float32-representable float64."""
    w = _rng(seed, module, 0xBEEF).standard_normal((m, n)) * std
    return w.astype(np.float32).astype(np.float64)


def random_orthonormal(m, r, seed=0, module=0):
    """A random m x r matrix with orthonormal columns (Gaussian + QR)."""
    return _orthonormal_columns(_rng(seed, module, 0xCAFE).standard_normal((m, r)))


def signed_permutation(m, r, seed=0):
    """First r columns of a random signed m x m permutation matrix."""
    g = _rng(seed, 0x5151)
    perm = g.permutation(m)
    signs = g.choice([-1.0, 1.0], size=m)
    P = np.zeros((m, m))
    P[perm, np.arange(m)] = signs
    return P[:, :r]


def lowrank_grad_torch(m, n, s, sigma0, noise, step, seed=0, module=0,
                       noise_rel=False, device="cuda", dtype=None):
    """The same recipe on a torch device (for workloads too large for the
    host): the factors come from ``lowrank_factors`` (NumPy), the noise from
    torch's generator on ``device`` seeded by (seed, module, step)."""
    import torch
    dtype = torch.bfloat16 if dtype is None else dtype
    u, v = lowrank_factors(m, n, s, seed, module)
    sig = sigma0 * 0.7 ** np.arange(s)
    ut = torch.tensor(u * sig, dtype=torch.float32, device=device)
    vt = torch.tensor(v, dtype=torch.float32, device=device)
    nu = noise * sigma0 / (n ** 0.5) if noise_rel else noise
    gen = torch.Generator(device=device)
    gen.manual_seed((seed * 1_000_003 + module * 7919 + 104729 * (1 + step)) & 0x7FFFFFFF)
    g = ut @ vt.T
    g.add_(torch.randn(m, n, generator=gen, device=device, dtype=torch.float32), alpha=nu)
    return g.to(dtype)
