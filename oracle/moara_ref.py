"""Plain float64 reference of the MoARa-on-GaLore optimizer step (the oracle).

TEST INFRASTRUCTURE ONLY.  The test-suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module; the product path (the
CUDA library under ``paper_2609_15037_gb300`` and its binding) never does, and
this module imports nothing from it.

Everything is float64 NumPy.  Library primitives used as single steps: ``@``
(matrix product), ``np.sqrt`` and LAPACK's SVD (``np.linalg.svd``).  The steps
follow the paper in its order and notation:

* ``decompose``      -- Decompose(G, B): §3.1 and Appendix B.1 (padding, block
                        norms, eps = 1e-12 in the denominator only, cropping).
* ``rep_b``          -- Rep_B of §3.1, cropped back to n columns (App. B.1).
* ``adam``           -- Optimizer_V / Optimizer_M of Algorithm 1: Adam with
                        bias correction and zero weight decay (App. D.2).
* ``truncated_svd``  -- TruncatedSVD(V, r) of Algorithm 1 (top-r left singular
                        vectors).
* ``step``           -- one pass of Algorithm 1's training-phase body for one
                        target weight, with the GaLore scale alpha (App. D.2).
* ``rank_table``     -- Phase 3 of Algorithm 1 (§3.2, App. C final allocation).
* ``clip_grads``     -- the global-norm gradient clipping of the 7B runs
                        (App. D.2), in torch.nn.utils.clip_grad_norm_ form.
* ``flatten_shape``  -- the N-D flatten rule of App. B (row axis kept, the
                        remaining axes flattened into columns).
* ``moment_bytes``   -- optimizer-state memory model of Appendix G.

Readings of the paper where it is silent:

* Step index: Algorithm 1 refreshes when ``s mod T_SVD == 0``; we take
  s = t - 1 with the 1-based Adam step t, so the first step always computes P.
* Adam: the update is (m / bc1) / (sqrt(v / bc2) + eps) with bc_i = 1 - beta_i^t
  (the torch.optim.Adam form); moments are not reset at a refresh.
* Optimizer_M returns Adam's normalised update of M (not M itself).
* The GaLore scale alpha multiplies the whole update.
* Singular-vector signs: an SVD fixes them only up to sign; each column of P is
  signed so that its entry of largest magnitude is positive (lowest index wins
  a tie).
* Projection side: the left projector P (m x r) of §3.1 for every module.
"""

from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

# Appendix B.1: "We use eps = 1e-12 in all experiments" (normalisation only).
DECOMP_EPS = 1e-12

# Algorithm 1 / §3.2: the seven target module types of a decoder layer.
MODULE_TYPES = ("q", "k", "v", "o", "gate", "up", "down")


# ---------------------------------------------------------------------------
# Decomposition (§3.1, Appendix B.1)
# ---------------------------------------------------------------------------

def num_blocks(n: int, B: int) -> int:
    """k = n_pad / B with n_pad = B * ceil(n / B)  (Appendix B.1)."""
    if B < 1 or n < 0:
        raise ValueError("block size must be >= 1 and n >= 0")
    return -(-n // B)


def decompose(G, B: int, eps: float = DECOMP_EPS):
    """Decompose(G, B) of Algorithm 1, as defined in §3.1 / Appendix B.1.

    1. right-zero-pad every row of G (m x n) to n_pad = B*ceil(n/B);
    2. split each padded row into k contiguous 1 x B blocks g_{i,b};
    3. m_{i,b} = ||g_{i,b}||_2 and v_{i,b} = g_{i,b} / (m_{i,b} + eps);
    4. discard the padded columns of V.

    Returns (M, V) with M of shape (m, k) and V of shape (m, n).
    """
    G = np.asarray(G, dtype=np.float64)
    m, n = G.shape
    k = num_blocks(n, B)
    n_pad = k * B
    G_pad = np.zeros((m, n_pad), dtype=np.float64)
    G_pad[:, :n] = G
    M = np.empty((m, k), dtype=np.float64)
    V_pad = np.empty((m, n_pad), dtype=np.float64)
    for b in range(k):
        g = G_pad[:, b * B:(b + 1) * B]
        mag = np.sqrt(np.sum(g * g, axis=1))
        M[:, b] = mag
        V_pad[:, b * B:(b + 1) * B] = g / (mag[:, None] + eps)
    V = V_pad[:, :n].copy()
    return M, V


def rep_b(X, B: int, n: int):
    """Rep_B(X) of §3.1: repeat every entry of X (m x k) over its B columns.

    The result has n_pad = k*B columns; as in Appendix B.1 the padded columns
    are cropped, giving an (m x n) matrix.
    """
    X = np.asarray(X, dtype=np.float64)
    m, k = X.shape
    out = np.empty((m, k * B), dtype=np.float64)
    for b in range(k):
        out[:, b * B:(b + 1) * B] = X[:, b:b + 1]
    return out[:, :n]


# ---------------------------------------------------------------------------
# Optimizer_V / Optimizer_M (Algorithm 1; Adam hyper-parameters of App. D.2)
# ---------------------------------------------------------------------------

def adam(grad, exp_avg, exp_avg_sq, t: int, beta1: float, beta2: float,
         eps: float):
    """One Adam step on ``grad`` with bias correction and no weight decay.

    Returns (update, new_exp_avg, new_exp_avg_sq) where
    update = (exp_avg / (1 - beta1^t)) / (sqrt(exp_avg_sq / (1 - beta2^t)) + eps).
    """
    grad = np.asarray(grad, dtype=np.float64)
    exp_avg = beta1 * exp_avg + (1.0 - beta1) * grad
    exp_avg_sq = beta2 * exp_avg_sq + (1.0 - beta2) * grad * grad
    bc1 = 1.0 - beta1 ** t
    bc2 = 1.0 - beta2 ** t
    update = (exp_avg / bc1) / (np.sqrt(exp_avg_sq / bc2) + eps)
    return update, exp_avg, exp_avg_sq


# ---------------------------------------------------------------------------
# Projector refresh (Algorithm 1, TruncatedSVD; GaLore projection of §3.1)
# ---------------------------------------------------------------------------

def fix_signs(P):
    """Sign each column so that its largest-magnitude entry is positive."""
    P = np.array(P, dtype=np.float64, copy=True)
    for j in range(P.shape[1]):
        i = int(np.argmax(np.abs(P[:, j])))
        if P[i, j] < 0:
            P[:, j] = -P[:, j]
    return P


def truncated_svd(X, r: int):
    """TruncatedSVD(X, r): the top-r left singular vectors of X (m x n).

    fp64 LAPACK SVD; columns in descending singular-value order, signs fixed
    by ``fix_signs``.  Returns (P, singular_values).
    """
    X = np.asarray(X, dtype=np.float64)
    U, S, _ = np.linalg.svd(X, full_matrices=False)
    return fix_signs(U[:, :r]), S


def bf16_round(x):
    """Nearest bf16 value (8 significant bits, ties to even) of each entry,
    from float64: x = f * 2^e with 0.5 <= |f| < 1, f rounded to a multiple of
    2^-8.  Zeros, infinities and NaNs pass through; the bf16 range is that
    of fp32, so no entry here over- or underflows it."""
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)
    return np.ldexp(np.rint(f * 256.0), e - 8)


def is_refresh_step(t: int, T: int) -> bool:
    """Algorithm 1 refreshes when s mod T_SVD == 0, read with s = t - 1."""
    return (t - 1) % T == 0


# ---------------------------------------------------------------------------
# One training-phase step of Algorithm 1 for one target weight
# ---------------------------------------------------------------------------

@dataclass
class Hparams:
    """Algorithm 1 "Require" and Appendix D.2 defaults."""
    beta1: float = 0.9
    beta2: float = 0.999
    adam_eps: float = 1e-6
    decomp_eps: float = DECOMP_EPS
    scale: float = 0.25          # GaLore scale alpha
    block_size: int = 128        # B
    refresh_interval: int = 200  # T_SVD
    decompose: bool = True       # False: plain GaLore (no magnitude branch)
    refresh_src: str = "V"       # "V" (Algorithm 1) or "G"
    state_bf16: bool = False     # W and the direction moments stored in bf16
    proj_rule: str = "left"      # "left": P (m x r) for every weight; "smaller":
                                 # GaLore's rule, a right projector Q (n x r) when m > n


@dataclass
class ModuleState:
    """Per-weight state: W, projector P and both Adam branches."""
    W: np.ndarray
    P: np.ndarray
    exp_avg: np.ndarray
    exp_avg_sq: np.ndarray
    mag_avg: np.ndarray
    mag_avg_sq: np.ndarray
    extras: dict = field(default_factory=dict)

    def copy(self):
        return replace(self, W=self.W.copy(), P=self.P.copy(),
                       exp_avg=self.exp_avg.copy(),
                       exp_avg_sq=self.exp_avg_sq.copy(),
                       mag_avg=self.mag_avg.copy(),
                       mag_avg_sq=self.mag_avg_sq.copy(), extras={})


def is_right(m: int, n: int, proj_rule: str) -> bool:
    """GaLore's smaller-side rule: project the column space (right projector
    Q, n x r) of a tall weight (m > n); the paper's memory numbers assume it
    (App. G, d_W = max(m, n))."""
    return proj_rule == "smaller" and m > n


def init_state(W, r: int, B: int, P=None, proj_rule: str = "left") -> ModuleState:
    """Zero Adam moments for weight W (m x n): r x n with a left projector P
    (m x r), m x r with a right projector Q (n x r, stored in ``P``); m x k
    magnitude moments."""
    W = np.array(W, dtype=np.float64, copy=True)
    m, n = W.shape
    k = num_blocks(n, B)
    right = is_right(m, n, proj_rule)
    shape = (n, r) if right else (m, r)
    if P is None:
        P = np.zeros(shape, dtype=np.float64)
    P = np.array(P, dtype=np.float64, copy=True)
    if P.shape != shape:
        raise ValueError(f"projector must be {shape[0]} x {shape[1]}")
    mom = (m, r) if right else (r, n)
    return ModuleState(W=W, P=P,
                       exp_avg=np.zeros(mom), exp_avg_sq=np.zeros(mom),
                       mag_avg=np.zeros((m, k)), mag_avg_sq=np.zeros((m, k)))


def step(state: ModuleState, G, t: int, lr: float, hp: Hparams,
         refresh: bool) -> ModuleState:
    """Algorithm 1, training-phase body, for one weight at Adam step t.

    M, V <- Decompose(G, B)
    if refresh: P <- TruncatedSVD(V, r)              (V, or G if refresh_src=G)
    Vt <- P^T V ; dVt <- Optimizer_V(Vt) ; dV <- P dVt
    dM <- Optimizer_M(M)
    W  <- W - lr * alpha * (Rep_B(dM) (.) dV)

    With ``hp.decompose`` False the step is plain GaLore: R = P^T G,
    W <- W - lr * alpha * P Adam(R).  Returns the new state; intermediates are
    kept in ``extras`` for tests.
    """
    G = np.asarray(G, dtype=np.float64)
    m, n = G.shape
    B = hp.block_size
    s = state.copy()
    r = s.P.shape[1]
    if hp.decompose:
        M, V = decompose(G, B, hp.decomp_eps)
    else:
        M, V = None, G
    right = is_right(m, n, hp.proj_rule)
    if refresh:
        src = V if hp.refresh_src == "V" else G
        # right projector: the top-r right singular vectors of the source
        s.P, _ = truncated_svd(src.T if right else src, r)
    R = V @ s.P if right else s.P.T @ V
    N, s.exp_avg, s.exp_avg_sq = adam(R, s.exp_avg, s.exp_avg_sq, t,
                                      hp.beta1, hp.beta2, hp.adam_eps)
    if hp.state_bf16:
        # the paper's runs keep 2-byte direction states (App. G memory model,
        # App. D.2): the update uses the new moments, which are then stored
        # rounded to bf16
        s.exp_avg, s.exp_avg_sq = bf16_round(s.exp_avg), bf16_round(s.exp_avg_sq)
    dV = N @ s.P.T if right else s.P @ N
    if hp.decompose:
        dM, s.mag_avg, s.mag_avg_sq = adam(M, s.mag_avg, s.mag_avg_sq, t,
                                           hp.beta1, hp.beta2, hp.adam_eps)
        U = rep_b(dM, B, n) * dV
    else:
        dM = None
        U = dV
    s.W = s.W - lr * hp.scale * U
    if hp.state_bf16:
        # App. D.2: the recomposed update is applied to bf16 weights
        s.W = bf16_round(s.W)
    s.extras = {"M": M, "V": V, "R": R, "N": N, "dV": dV, "dM": dM, "U": U}
    return s


def run(state: ModuleState, grads, lr: float, hp: Hparams, t0: int = 1,
        auto_refresh: bool = True) -> ModuleState:
    """Apply ``step`` for t = t0, t0+1, ... over the list ``grads``."""
    for i, G in enumerate(grads):
        t = t0 + i
        refresh = auto_refresh and is_refresh_step(t, hp.refresh_interval)
        state = step(state, G, t, lr, hp, refresh)
    return state


# ---------------------------------------------------------------------------
# Global-norm gradient clipping (App. D.2) and the N-D flatten rule (App. B)
# ---------------------------------------------------------------------------

def clip_grads(grads, max_norm: float, extra_sq: float = 0.0):
    """The 7B runs clip gradients at global norm 1.0 (App. D.2); the paper
    gives no formula, so this is torch.nn.utils.clip_grad_norm_: the total
    norm over every gradient (plus the squared norm of gradients outside this
    list), coefficient min(1, max_norm / (norm + 1e-6)), every gradient scaled
    by it.  Returns (scaled gradients, total norm, coefficient)."""
    total_sq = float(extra_sq)
    for G in grads:
        G = np.asarray(G, dtype=np.float64)
        total_sq += float(np.sum(G * G))
    norm = np.sqrt(total_sq)
    coef = min(1.0, max_norm / (norm + 1e-6))
    return [coef * np.asarray(G, dtype=np.float64) for G in grads], norm, coef


def flatten_shape(shape):
    """App. B: a gradient of shape (s_0, ..., s_{k-1}) is treated as the
    matrix with m = s_0 rows and n = s_1 * ... * s_{k-1} columns."""
    shape = [int(s) for s in shape]
    if len(shape) < 1 or min(shape) < 1:
        raise ValueError("shape must have at least one positive extent")
    n = 1
    for s in shape[1:]:
        n *= s
    return shape[0], n


# ---------------------------------------------------------------------------
# Alignment diagnostic S(W, t) (§3.2)
# ---------------------------------------------------------------------------

def alignment(G, P, B: int, eps: float = DECOMP_EPS, right: bool = False) -> float:
    """S(W,t) = cos(G, G_recon) with G_recon = Rep_B(M) (.) (P P^T V)  (§3.2);
    with a right projector Q (n x r, passed as P) the projected direction is
    V Q Q^T."""
    G = np.asarray(G, dtype=np.float64)
    M, V = decompose(G, B, eps)
    proj = (V @ P) @ P.T if right else P @ (P.T @ V)
    G_recon = rep_b(M, B, G.shape[1]) * proj
    num = float(np.sum(G * G_recon))
    den = float(np.sqrt(np.sum(G * G)) * np.sqrt(np.sum(G_recon * G_recon)))
    return num / den if den > 0 else 0.0


# ---------------------------------------------------------------------------
# Phase 3 rank reallocation (§3.2; App. C "Final rank allocation")
# ---------------------------------------------------------------------------

def rank_table(r_base: int, donors, receivers, delta_r: int):
    """Budget-preserving reallocation of Algorithm 1, Phase 3.

    donors get r_base - delta_r, receivers r_base + delta_r*|D|/|R|, the rest
    r_base.  When |R| does not divide delta_r*|D| the quotient is floored and
    the remainder handed out one by one to receivers in module order, so the
    total stays 7*r_base.  Returns a dict {module_type: rank}.
    """
    donors = [d for d in MODULE_TYPES if d in set(donors)]
    receivers = [x for x in MODULE_TYPES if x in set(receivers)]
    if set(donors) & set(receivers):
        raise ValueError("a module cannot be both donor and receiver")
    if donors and not receivers:
        raise ValueError("donors need at least one receiver")
    if not 0 <= delta_r < r_base:
        raise ValueError("need 0 <= delta_r < r_base")
    ranks = {t: r_base for t in MODULE_TYPES}
    for d in donors:
        ranks[d] = r_base - delta_r
    if receivers:
        moved = delta_r * len(donors)
        share, rem = divmod(moved, len(receivers))
        for i, x in enumerate(receivers):
            ranks[x] = r_base + share + (1 if i < rem else 0)
    return ranks


# ---------------------------------------------------------------------------
# Optimizer-state memory model (Appendix G)
# ---------------------------------------------------------------------------

def moment_bytes(m: int, n: int, r: int, B: int, b_V: int, b_M: int,
                 d_rule: str = "n", decompose: bool = True) -> int:
    """Adam-state bytes of one target matrix, Appendix G.

    Direction branch 2*b_V*r*d_W and magnitude branch 2*b_M*m*ceil(n/B).
    d_rule "n": d_W = n (left projector, R is r x n);
    d_rule "max": d_W = max(m, n) (the smaller side is projected, as GaLore
    does for tall matrices).
    """
    d = n if d_rule == "n" else max(m, n)
    total = 2 * b_V * r * d
    if decompose:
        total += 2 * b_M * m * num_blocks(n, B)
    return total
