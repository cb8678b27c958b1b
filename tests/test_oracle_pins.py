"""Pins of the oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: special
cases the paper states, closed forms computed with a different routine, a
library optimiser (torch.optim.Adam), the paper's printed numbers, and a
loop-only twin on tiny inputs.
"""

import math
import os

import numpy as np
import pytest

from oracle import moara_ref as o
from oracle import brute
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- decompose

@pytest.mark.parametrize("m,n,B", [(5, 12, 4), (7, 10, 3), (3, 16, 16), (6, 9, 1)])
def test_recomposition_exact_without_eps(m, n, B):
    """§3.1: G_pad = Rep_B(M) (.) V_pad exactly as eps -> 0."""
    G = _rng(1).standard_normal((m, n))
    M, V = o.decompose(G, B, eps=0.0)
    np.testing.assert_allclose(o.rep_b(M, B, n) * V, G, rtol=1e-14, atol=1e-15)


def test_recomposition_with_eps_closed_form():
    """App. B.1: m*v = ||g|| / (||g|| + eps) * g for finite eps."""
    eps = 1e-3
    G = _rng(2).standard_normal((4, 10)) * 1e-2
    B = 4
    M, V = o.decompose(G, B, eps=eps)
    Gp = np.zeros((4, 12))
    Gp[:, :10] = G
    norms = np.linalg.norm(Gp.reshape(4, 3, 4), axis=2)
    factor = np.repeat(norms / (norms + eps), 4, axis=1)[:, :10]
    np.testing.assert_allclose(o.rep_b(M, B, 10) * V, factor * G, rtol=1e-13)


def test_zero_block_gives_zero_direction():
    """App. B.3: a zero block has v = 0 (automatic with eps > 0)."""
    G = _rng(3).standard_normal((3, 8))
    G[1, 4:8] = 0.0
    M, V = o.decompose(G, 4)
    assert M[1, 1] == 0.0
    assert np.all(V[1, 4:8] == 0.0)
    Mz, Vz = o.decompose(np.zeros((2, 5)), 2)
    assert np.all(Mz == 0) and np.all(Vz == 0)


def test_block_size_one_is_sign():
    """App. B.3 small-B regime: B = 1 gives M = |G| and V = sign(G)."""
    G = _rng(4).standard_normal((6, 7))
    G[2, 3] = 0.0
    with np.errstate(invalid="ignore"):
        M, V = o.decompose(G, 1, eps=0.0)
    np.testing.assert_array_equal(M, np.abs(G))
    np.testing.assert_array_equal(np.nan_to_num(V), np.sign(G))
    M, V = o.decompose(G, 1)
    np.testing.assert_array_equal(M, np.abs(G))
    dev = np.abs(V - np.sign(G))
    assert np.all(dev <= 1e-12 / np.maximum(np.abs(G), 1e-300) + 1e-15)


def test_block_size_n_is_row_normalisation():
    """§3.1: a single block per row is the row-wise decomposition."""
    G = _rng(5).standard_normal((5, 11))
    M, V = o.decompose(G, 11)
    rn = np.linalg.norm(G, axis=1)
    np.testing.assert_allclose(M[:, 0], rn, rtol=1e-14)
    np.testing.assert_allclose(V, G / rn[:, None], rtol=1e-11)


def test_blocks_run_along_columns():
    """§3.1 / App. B.1: rows are kept, blocks are contiguous column ranges."""
    G = _rng(6).standard_normal((3, 12))
    M, _ = o.decompose(G, 4)
    assert M.shape == (3, 3)
    for i in range(3):
        for b in range(3):
            assert M[i, b] == pytest.approx(np.linalg.norm(G[i, 4 * b:4 * b + 4]), rel=1e-14)


@pytest.mark.parametrize("n,B", [(10, 4), (2736, 32), (13, 5), (7, 8)])
def test_padding_invariance(n, B):
    """App. B.1: zero padding does not change the last block's magnitude;
    decomposing G equals decomposing the explicitly padded G, then cropping."""
    m = 3
    G = _rng(7).standard_normal((m, n))
    k = -(-n // B)
    Gp = np.zeros((m, k * B))
    Gp[:, :n] = G
    M1, V1 = o.decompose(G, B)
    M2, V2 = o.decompose(Gp, B)
    np.testing.assert_array_equal(M1, M2)
    np.testing.assert_array_equal(V1, V2[:, :n])
    last = np.linalg.norm(G[:, (k - 1) * B:], axis=1)
    np.testing.assert_allclose(M1[:, -1], last, rtol=1e-14)


def test_proposition_1_block_cosine():
    """App. B.3, Proposition 1: cos(G_b, m_b * vt_b) = cos(v_b, vt_b)."""
    m, n, B, r = 16, 24, 6, 5
    G = _rng(8).standard_normal((m, n))
    M, V = o.decompose(G, B)
    P = synth.random_orthonormal(m, r, seed=3)
    Vt = P @ (P.T @ V)
    for i in range(m):
        for b in range(n // B):
            gb = G[i, b * B:(b + 1) * B]
            vb = V[i, b * B:(b + 1) * B]
            tb = Vt[i, b * B:(b + 1) * B]
            c1 = gb @ (M[i, b] * tb) / (np.linalg.norm(gb) * np.linalg.norm(M[i, b] * tb))
            c2 = vb @ tb / (np.linalg.norm(vb) * np.linalg.norm(tb))
            assert c1 == pytest.approx(c2, rel=1e-12, abs=1e-14)


# ------------------------------------------------- Adam reductions (library)

def _torch_adam_trajectory(W0, grads, lr, beta1, beta2, eps):
    torch = pytest.importorskip("torch")
    p = torch.nn.Parameter(torch.tensor(W0, dtype=torch.float64))
    opt = torch.optim.Adam([p], lr=lr, betas=(beta1, beta2), eps=eps,
                           weight_decay=0.0)
    for G in grads:
        p.grad = torch.tensor(G, dtype=torch.float64)
        opt.step()
    return p.detach().numpy()


@pytest.mark.parametrize("m,n", [(6, 9), (8, 8)])
def test_galore_full_rank_signed_permutation_is_adam(m, n):
    """Decomposition off, P a signed permutation with r = m <= n: the GaLore
    step is plain Adam (torch.optim.Adam with lr * alpha)."""
    hp = o.Hparams(decompose=False, scale=0.25, adam_eps=1e-8, block_size=3)
    lr = 1e-2
    P = synth.signed_permutation(m, m, seed=11)
    grads = [_rng(20 + t).standard_normal((m, n)) for t in range(10)]
    W0 = _rng(19).standard_normal((m, n)) * 0.02
    st = o.run(o.init_state(W0, m, 3, P=P), grads, lr, hp, auto_refresh=False)
    ref = _torch_adam_trajectory(W0, grads, lr * hp.scale, hp.beta1, hp.beta2, hp.adam_eps)
    np.testing.assert_allclose(st.W, ref, rtol=1e-12, atol=1e-15)


def test_galore_partial_permutation_updates_selected_rows_only():
    """r < m with P = r columns of a signed permutation: selected rows follow
    Adam, the other rows are untouched."""
    m, n, r = 7, 5, 3
    hp = o.Hparams(decompose=False, scale=1.0, adam_eps=1e-8, block_size=5)
    P = synth.signed_permutation(m, r, seed=4)
    rows = [int(np.flatnonzero(P[:, j])[0]) for j in range(r)]
    grads = [_rng(40 + t).standard_normal((m, n)) for t in range(6)]
    W0 = _rng(39).standard_normal((m, n))
    st = o.run(o.init_state(W0, r, 5, P=P), grads, 1e-2, hp, auto_refresh=False)
    ref = _torch_adam_trajectory(W0, grads, 1e-2, hp.beta1, hp.beta2, hp.adam_eps)
    other = [i for i in range(m) if i not in rows]
    np.testing.assert_allclose(st.W[rows], ref[rows], rtol=1e-12)
    np.testing.assert_array_equal(st.W[other], W0[other])


def test_identity_projector_is_adam_of_v_times_adam_of_m():
    """Decomposition on and P = I: the update is Rep_B(Adam(M)) (.) Adam(V),
    with both Adams run by torch.optim.Adam and M, V from np.linalg.norm."""
    torch = pytest.importorskip("torch")
    m, n, B = 5, 10, 4
    k = 3
    hp = o.Hparams(decompose=True, scale=0.25, adam_eps=1e-6, block_size=B)
    lr = 3e-3
    grads = [_rng(60 + t).standard_normal((m, n)) for t in range(8)]
    W0 = _rng(59).standard_normal((m, n)) * 0.02
    st = o.run(o.init_state(W0, m, B, P=np.eye(m)), grads, lr, hp, auto_refresh=False)

    pv = torch.nn.Parameter(torch.zeros(m, n, dtype=torch.float64))
    pm = torch.nn.Parameter(torch.zeros(m, k, dtype=torch.float64))
    ov = torch.optim.Adam([pv], lr=1.0, betas=(hp.beta1, hp.beta2), eps=hp.adam_eps)
    om = torch.optim.Adam([pm], lr=1.0, betas=(hp.beta1, hp.beta2), eps=hp.adam_eps)
    W = W0.copy()
    for G in grads:
        Gp = np.zeros((m, k * B))
        Gp[:, :n] = G
        Mg = np.linalg.norm(Gp.reshape(m, k, B), axis=2)
        Vg = G / (np.repeat(Mg, B, axis=1)[:, :n] + hp.decomp_eps)
        before_v, before_m = pv.detach().clone(), pm.detach().clone()
        pv.grad = torch.tensor(Vg)
        pm.grad = torch.tensor(Mg)
        ov.step()
        om.step()
        dV = (before_v - pv.detach()).numpy()
        dM = (before_m - pm.detach()).numpy()
        W = W - lr * hp.scale * np.repeat(dM, B, axis=1)[:, :n] * dV
    np.testing.assert_allclose(st.W, W, rtol=1e-11, atol=1e-14)


def test_projector_column_sign_flip_invariance():
    """Flipping the sign of projector columns leaves the trajectory unchanged."""
    m, n, r, B = 12, 16, 4, 4
    hp = o.Hparams(block_size=B, adam_eps=1e-8)
    P = synth.random_orthonormal(m, r, seed=9)
    Pf = P * np.array([1, -1, -1, 1])
    grads = [_rng(80 + t).standard_normal((m, n)) for t in range(5)]
    W0 = _rng(79).standard_normal((m, n))
    a = o.run(o.init_state(W0, r, B, P=P), grads, 1e-3, hp, auto_refresh=False)
    b = o.run(o.init_state(W0, r, B, P=Pf), grads, 1e-3, hp, auto_refresh=False)
    np.testing.assert_allclose(a.W, b.W, rtol=1e-13, atol=1e-16)


def test_projector_rotation_changes_update():
    """Adam is elementwise, so a general rotation of P does change the step:
    the P = I reduction above needs a signed permutation."""
    m, n = 6, 6
    hp = o.Hparams(decompose=False, block_size=3)
    Q = synth.random_orthonormal(m, m, seed=2)
    G = _rng(90).standard_normal((m, n))
    W0 = np.zeros((m, n))
    a = o.step(o.init_state(W0, m, 3, P=np.eye(m)), G, 1, 1e-2, hp, refresh=False)
    b = o.step(o.init_state(W0, m, 3, P=Q), G, 1, 1e-2, hp, refresh=False)
    assert np.max(np.abs(a.W - b.W)) > 1e-4


# ---------------------------------------------------------------- refresh

def test_fix_signs_convention_by_hand():
    """Singular vectors are defined up to sign; the projector fixes it so that
    each column's largest-magnitude entry is positive, the lowest row winning
    a tie of magnitudes.  Checked on hand-made columns."""
    P = np.array([[-0.5, 0.5, 0.0, -0.25],
                  [0.5, -0.5, 0.0, 0.75],
                  [0.1, 0.2, 0.0, -0.75]])
    F = o.fix_signs(P)
    # column 0: tie of 0.5 between rows 0 (negative) and 1: row 0 wins, flip
    np.testing.assert_array_equal(F[:, 0], [0.5, -0.5, -0.1])
    # column 1: the same tie, row 0 positive: unchanged
    np.testing.assert_array_equal(F[:, 1], P[:, 1])
    # column 2: all zero stays zero
    np.testing.assert_array_equal(F[:, 2], P[:, 2])
    # column 3: tie of 0.75 between rows 1 (positive) and 2: unchanged
    np.testing.assert_array_equal(F[:, 3], P[:, 3])
    # idempotent, and a sign flip of the input gives the same output
    np.testing.assert_array_equal(o.fix_signs(F), F)
    np.testing.assert_array_equal(o.fix_signs(-P), F)


def test_refresh_orthonormal_and_eckart_young():
    """TruncatedSVD: P^T P = I, and the captured energy ||P^T V||_F^2 equals
    the sum of the top-r squared singular values (Eckart-Young), more than
    any other orthonormal P."""
    m, n, r = 30, 40, 6
    G = synth.lowrank_grad(m, n, 8, 10.0, 0.01, 1, seed=1)
    _, V = o.decompose(G, 8)
    P, S = o.truncated_svd(V, r)
    np.testing.assert_allclose(P.T @ P, np.eye(r), atol=1e-12)
    e = np.sum((P.T @ V) ** 2)
    assert e == pytest.approx(np.sum(S[:r] ** 2), rel=1e-12)
    for s in range(5):
        Q = synth.random_orthonormal(m, r, seed=100 + s)
        assert np.sum((Q.T @ V) ** 2) < e


def test_refresh_step_index():
    """Algorithm 1 refreshes at s mod T == 0 with s = t - 1."""
    assert o.is_refresh_step(1, 200)
    assert not o.is_refresh_step(200, 200)
    assert o.is_refresh_step(201, 200)
    assert [t for t in range(1, 11) if o.is_refresh_step(t, 3)] == [1, 4, 7, 10]


# -------------------------------------------------- brute-force twin on 8x8

def _gap_ok(X, r, rel=1e-6):
    S = np.linalg.svd(np.asarray(X), compute_uv=False)
    if r >= len(S):
        return S[-1] > rel * S[0]
    return (S[r - 1] - S[r]) > rel * S[0]


CASES = [
    # (m, n, B, r, decompose, src)
    (8, 8, 1, 3, True, "V"), (8, 8, 2, 5, True, "V"), (8, 8, 3, 4, True, "V"),
    (8, 8, 4, 8, True, "V"), (8, 8, 8, 1, True, "V"), (8, 8, 4, 2, True, "G"),
    (8, 8, 2, 6, False, "V"), (8, 11, 3, 7, True, "V"), (6, 8, 4, 6, True, "V"),
    (8, 5, 2, 5, True, "V"),
]


@pytest.mark.parametrize("m,n,B,r,dec,src", CASES)
def test_oracle_matches_loop_twin(m, n, B, r, dec, src):
    T = 3
    grads = [list(map(list, _rng(300 + t).standard_normal((m, n)))) for t in range(10)]
    W0 = _rng(299).standard_normal((m, n)) * 0.02
    hp = o.Hparams(block_size=B, refresh_interval=T, decompose=dec,
                   refresh_src=src, adam_eps=1e-6, scale=0.25)
    for t in range(1, 11):
        if o.is_refresh_step(t, T):
            Gt = np.array(grads[t - 1])
            X = o.decompose(Gt, B)[1] if (dec and src == "V") else Gt
            if not _gap_ok(X, r):
                pytest.skip("degenerate spectrum at the truncation rank")
    st = o.run(o.init_state(W0, r, B), [np.array(g) for g in grads], 1e-2, hp)
    Wb, Pb = brute.run([list(row) for row in W0], grads, r, 1e-2, B, T,
                       decompose_on=dec, refresh_src=src, adam_eps=1e-6,
                       scale=0.25)
    np.testing.assert_allclose(np.array(Pb), st.P, atol=1e-9)
    np.testing.assert_allclose(np.array(Wb), st.W, rtol=1e-9, atol=1e-12)


# ------------------------------------------------------- rank table (Phase 3)

def _golden_rows(name):
    rows = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                p = line.split()
                rows[p[0]] = p[1:]
    return rows


def test_rank_table_matches_final_allocation():
    """App. C: D = {q, k}, R = {down}, delta_r = r_base/2 at r_base = 256."""
    ours = [int(x) for x in _golden_rows("rank_allocations.txt")["Ours"]]
    got = o.rank_table(256, ["q", "k"], ["down"], 128)
    assert [got[t] for t in o.MODULE_TYPES] == ours


def test_rank_tables_preserve_budget():
    """Every allocation in the paper's table (and every output of the rule,
    including uneven splits) keeps sum_tau r_tau = 7 r_base."""
    for run, vals in _golden_rows("rank_allocations.txt").items():
        assert sum(int(v) for v in vals) == 7 * 256, run
    for donors, recv, dr in [(["q", "k", "v"], ["up", "down"], 100),
                             (["q"], ["gate", "up", "down"], 64),
                             ([], [], 0), (["o", "k"], ["q"], 255)]:
        got = o.rank_table(512, donors, recv, dr)
        assert sum(got.values()) == 7 * 512
    uneven = o.rank_table(512, ["q", "k", "v"], ["up", "down"], 101)
    assert (uneven["up"], uneven["down"]) == (512 + 152, 512 + 151)


# ------------------------------------------------ memory model (Appendix G)

@pytest.mark.parametrize("model", ["350M", "1B", "7B"])
def test_memory_model_reproduces_printed_table(model):
    """Appendix G: 2 b_V r d_W + 2 b_M m ceil(n/B) summed over the target
    matrices reproduces all printed optimizer-state MiB values, with
    b_V = 2, b_M = 4 (fp32 magnitude branch, App. D.2), d_W = max(m, n),
    plus untied 32000-token embedding/head with full Adam in 2-byte states
    and fp32 norm weights."""
    row = _golden_rows("memory_table.txt")[model]
    h, f, L, B, rb = (int(x) for x in row[:5])
    printed = [float(x) for x in row[5:]]
    shp = {"q": (h, h), "k": (h, h), "v": (h, h), "o": (h, h),
           "gate": (f, h), "up": (f, h), "down": (h, f)}
    uni = {t: rb for t in shp}
    aware = o.rank_table(rb, ["q", "k"], ["down"], rb // 2)
    other = 2 * 32000 * h * 2 * 2 + (2 * L + 1) * h * 4

    def total(ranks, dec):
        return L * sum(o.moment_bytes(m, n, ranks[t], B, 2, 4, "max", dec)
                       for t, (m, n) in shp.items()) + other

    got = [total(uni, False), total(uni, True), total(aware, False), total(aware, True)]
    for g, p in zip(got, printed):
        assert round(g / 2 ** 20, 2) == pytest.approx(p, abs=1e-9)


def test_alignment_full_rank_projection_is_one():
    """§3.2: with P spanning the whole column space, G_recon = Rep_B(M) (.) V,
    so S(W, t) = 1 up to the eps of the decomposition."""
    G = _rng(12).standard_normal((6, 9))
    assert o.alignment(G, np.eye(6), 3) == pytest.approx(1.0, abs=1e-12)
    P = synth.random_orthonormal(6, 2, seed=1)
    assert o.alignment(G, P, 3) < 0.99

def test_alignment_rank_one_closed_form():
    """§3.2 with one block per row (B = n) and G = u v^T: V = sign(u) v^T/||v||,
    so with P = u/||u|| the reconstruction is |u_i| u_i (sum|u|) v_j / ||u||^2 and
    S = sum|u_i|^3 / (||u|| sqrt(sum u_i^4)); with P along sign(u), S = 1."""
    rng = _rng(31)
    u, v = rng.standard_normal(7), rng.standard_normal(5)
    G = np.outer(u, v)
    S = o.alignment(G, (u / np.linalg.norm(u))[:, None], 5)
    closed = np.sum(np.abs(u) ** 3) / (np.linalg.norm(u) * np.sqrt(np.sum(u ** 4)))
    assert S == pytest.approx(closed, rel=1e-12)
    sg = np.sign(u)
    assert o.alignment(G, (sg / np.linalg.norm(sg))[:, None], 5) == pytest.approx(1.0, abs=1e-12)


def test_alignment_loop_twin_and_invariances():
    """The alignment against a pure-loop evaluation of its definition (block
    norms, V, P P^T V, Rep_B, cosine) on a ragged 5 x 7 case with B = 3, and
    its invariance under column sign flips of P and positive scaling of G."""
    rng = _rng(32)
    m, n, r, B = 5, 7, 2, 3
    G = rng.standard_normal((m, n))
    P = synth.random_orthonormal(m, r, seed=4)
    eps = 1e-12
    kb = -(-n // B)
    M = [[0.0] * kb for _ in range(m)]
    V = [[0.0] * n for _ in range(m)]
    for i in range(m):
        for b in range(kb):
            cols = range(b * B, min(n, (b + 1) * B))
            M[i][b] = sum(G[i][j] ** 2 for j in cols) ** 0.5
            for j in cols:
                V[i][j] = G[i][j] / (M[i][b] + eps)
    R = [[sum(P[i][a] * V[i][j] for i in range(m)) for j in range(n)] for a in range(r)]
    num = den_g = den_r = 0.0
    for i in range(m):
        for j in range(n):
            rec = M[i][j // B] * sum(P[i][a] * R[a][j] for a in range(r))
            num += G[i][j] * rec
            den_g += G[i][j] ** 2
            den_r += rec ** 2
    assert o.alignment(G, P, B) == pytest.approx(num / (den_g * den_r) ** 0.5, rel=1e-12)
    flip = P * np.array([-1.0, 1.0])
    assert o.alignment(G, flip, B) == pytest.approx(o.alignment(G, P, B), rel=1e-12)
    assert o.alignment(3.0 * G, P, B) == pytest.approx(o.alignment(G, P, B), rel=1e-9)


def test_clip_closed_forms():
    """App. D.2 clipping: constant gradients with sum of squares 6*9 + 4*4 = 70;
    below the threshold nothing changes; the extra term of other parameters
    enters the norm (70 + 30 = 100, norm 10)."""
    g1, g2 = np.full((2, 3), 3.0), np.full((4, 1), -2.0)
    out, norm, coef = o.clip_grads([g1, g2], 1.0)
    assert norm == pytest.approx(np.sqrt(70.0), rel=1e-15)
    assert coef == pytest.approx(1.0 / (np.sqrt(70.0) + 1e-6), rel=1e-15)
    assert out[0][0, 0] == pytest.approx(3.0 * coef, rel=1e-15)
    assert out[1][3, 0] == pytest.approx(-2.0 * coef, rel=1e-15)
    clipped = np.sqrt(sum(float(np.sum(x * x)) for x in out))
    assert clipped == pytest.approx(np.sqrt(70.0) / (np.sqrt(70.0) + 1e-6), rel=1e-14)
    out, norm, coef = o.clip_grads([g1, g2], 100.0)
    assert coef == 1.0 and np.array_equal(out[0], g1) and np.array_equal(out[1], g2)
    _, norm, coef = o.clip_grads([g1, g2], 1.0, extra_sq=30.0)
    assert norm == pytest.approx(10.0, rel=1e-15)
    assert coef == pytest.approx(1.0 / (10.0 + 1e-6), rel=1e-15)


def test_clip_scales_magnitude_not_direction():
    """§3.1: Decompose(c G) = (c M, V) for c > 0 up to the eps of the block
    normalisation, so clipping reaches only the magnitude branch when the
    decomposition is on."""
    G = _rng(41).standard_normal((6, 10))
    M, V = o.decompose(G, 4)
    Mc, Vc = o.decompose(0.3 * G, 4)
    np.testing.assert_allclose(Mc, 0.3 * M, rtol=1e-14)
    np.testing.assert_allclose(Vc, V, rtol=1e-10)


def test_flatten_rule():
    """App. B flatten: the row axis is kept and the others are flattened."""
    assert o.flatten_shape((8, 3, 3, 3)) == (8, 27)
    assert o.flatten_shape((4096, 11008)) == (4096, 11008)
    assert o.flatten_shape((5,)) == (5, 1)
    G = np.arange(2 * 3 * 4, dtype=np.float64).reshape(2, 3, 4)
    m, n = o.flatten_shape(G.shape)
    flat = G.reshape(m, n)
    assert flat[1, 5] == G[1, 1, 1]
    with pytest.raises(ValueError):
        o.flatten_shape((3, 0))


def test_bf16_round_matches_torch_and_ties_to_even():
    """bf16_round against torch's float32 -> bfloat16 conversion (a library
    routine) on fp32-representable inputs, and the tie rule by hand:
    1 + 2^-8 lies halfway between 1 and 1 + 2^-7 and rounds to the even 1;
    1 + 3 * 2^-8 rounds up to 1 + 2^-6."""
    torch = pytest.importorskip("torch")
    x = (_rng(51).standard_normal(10000) * np.exp(_rng(52).uniform(-20, 20, 10000))).astype(np.float32)
    ref = torch.tensor(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(o.bf16_round(x.astype(np.float64)), ref)
    assert o.bf16_round(np.array([1.0 + 2.0 ** -8]))[0] == 1.0
    assert o.bf16_round(np.array([1.0 + 3 * 2.0 ** -8]))[0] == 1.0 + 2.0 ** -6
    assert o.bf16_round(np.array([-(1.0 + 2.0 ** -8)]))[0] == -1.0
    assert o.bf16_round(np.array([0.0]))[0] == 0.0


def test_bf16_state_step_stores_rounded_states():
    """With bf16 states the step's W and direction moments are bf16 values
    and differ from the fp32-state step by rounding only."""
    rng = _rng(53)
    m, n, r, B = 16, 24, 4, 8
    G = rng.standard_normal((m, n))
    W0 = o.bf16_round(rng.standard_normal((m, n)) * 0.02)
    P = np.linalg.qr(rng.standard_normal((m, r)))[0]
    hp32, hp16 = o.Hparams(block_size=B), o.Hparams(block_size=B, state_bf16=True)
    s32 = o.step(o.init_state(W0, r, B, P=P), G, 1, 1e-3, hp32, False)
    s16 = o.step(o.init_state(W0, r, B, P=P), G, 1, 1e-3, hp16, False)
    for x in (s16.W, s16.exp_avg, s16.exp_avg_sq):
        assert np.array_equal(o.bf16_round(x), x)
    np.testing.assert_array_equal(s16.W, o.bf16_round(s32.W))
    np.testing.assert_array_equal(s16.exp_avg, o.bf16_round(s32.exp_avg))


def test_right_projection_is_the_transposed_left_step():
    """GaLore's rule for a tall weight: without the decomposition the step
    with the right projector Q on G (m x n) is the left-projector step on
    G^T (n x m) with P = Q, transposed back (same Adam moments, transposed)."""
    rng = _rng(61)
    m, n, r = 12, 7, 3
    hpR = o.Hparams(block_size=4, decompose=False, proj_rule="smaller")
    hpL = o.Hparams(block_size=4, decompose=False)
    W0 = rng.standard_normal((m, n)) * 0.02
    Q = np.linalg.qr(rng.standard_normal((n, r)))[0]
    sR, sL = o.init_state(W0, r, 4, P=Q, proj_rule="smaller"), o.init_state(W0.T, r, 4, P=Q)
    for t in range(1, 4):
        G = rng.standard_normal((m, n))
        sR = o.step(sR, G, t, 1e-3, hpR, False)
        sL = o.step(sL, G.T, t, 1e-3, hpL, False)
    np.testing.assert_allclose(sR.W, sL.W.T, rtol=0, atol=1e-15)
    np.testing.assert_allclose(sR.exp_avg, sL.exp_avg.T, rtol=0, atol=1e-15)


def test_right_projector_refresh_and_full_rank():
    """The smaller-side refresh takes the top-r right singular vectors (the
    row space of V); with r = n the projector spans everything and, as with
    P = I for the left rule, the direction branch is Adam on V itself."""
    rng = _rng(62)
    m, n, B = 10, 6, 3
    G = rng.standard_normal((m, n))
    hp = o.Hparams(block_size=B, proj_rule="smaller")
    st = o.step(o.init_state(np.zeros((m, n)), 2, B, proj_rule="smaller"), G, 1, 1e-3, hp, True)
    V = o.decompose(G, B)[1]
    _, S, Vt = np.linalg.svd(V)
    cos = np.abs(np.sum(st.P * Vt[:2].T, axis=0))
    np.testing.assert_allclose(cos, 1.0, atol=1e-12)
    # full rank, Q = I: R = V, so the step equals the P = I left-rule step on V's rows
    st_r = o.step(o.init_state(np.zeros((m, n)), n, B, P=np.eye(n), proj_rule="smaller"), G, 1, 1e-3, hp, False)
    np.testing.assert_allclose(st_r.extras["R"], V, atol=1e-15)
    # square and wide weights keep the left projector under the smaller-side rule
    assert not o.is_right(6, 6, "smaller") and not o.is_right(4, 9, "smaller") and o.is_right(9, 4, "smaller")


def test_alignment_right_projector_is_the_transposed_case_without_blocks():
    """With one block per row and a rank-one G = u v^T, V = sign(u) v^T / ||v||
    lies in the row space span(v): a right projector along v reconstructs V
    exactly (S = 1), one orthogonal to v gives S = 0."""
    rng = _rng(63)
    u, v = rng.standard_normal(7), rng.standard_normal(5)
    G = np.outer(u, v)
    q = (v / np.linalg.norm(v))[:, None]
    assert o.alignment(G, q, 5, right=True) == pytest.approx(1.0, abs=1e-12)
    w = rng.standard_normal(5)
    w -= q[:, 0] * (q[:, 0] @ w)
    assert o.alignment(G, (w / np.linalg.norm(w))[:, None], 5, right=True) == pytest.approx(0.0, abs=1e-12)
