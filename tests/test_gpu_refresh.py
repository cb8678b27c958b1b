"""GPU projector refresh (TruncatedSVD of Algorithm 1, computed by the
library's randomized subspace iteration) against the float64 references.

Every refreshed projector is checked for P^T P = I within 1e-5, principal
angles <= 1e-2 rad against the exact top-r subspace on the leading
directions up to the spectral gap k_gap (largest k <= r with
sigma_k / sigma_{k+1} >= 1.5), and captured energy against the float64
restatement of the same randomized method with the same Philox sketch
(oracle/rsi_ref.py; the device may lose at most 3e-4 of the optimum plus a
quarter of the method's own deficit more).  On inputs with a clear gap at r
the energy must also reach (1 - 1e-3) of the exact optimum and every
singular vector must match individually, in order.  The decomposed V of
the rank-32-plus-noise gradients has a flat noise bulk around r; there the
method's own deficit against the exact SVD is measured and reported (the
flat-bulk figures are recorded with the design notes), not hidden behind a
looser bar.
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import principal_angles, gap_index, make_inputs, check_refresh, top_subspace
from oracle import rsi_ref as R

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def _dev(G, bf16=True):
    t = torch.tensor(G, dtype=torch.float32)
    return (t.to(torch.bfloat16) if bf16 else t).cuda()


def _check(g, mid, P, X, r, exact_bar=None):
    hp = g.hp
    return check_refresh(P, X, r, hp.oversample, hp.power_iters, R.sketch_key(hp.seed, mid, 0),
                         exact_bar=exact_bar)


@pytest.mark.parametrize("src", ["V", "G"])
def test_refresh_llama300m_attention_and_mlp(M, src):
    shapes = [(1024, 1024, 128), (2816, 1024, 256), (1024, 2816, 256)]
    B = 64
    grads, W0 = make_inputs(shapes, B, 1, True, signal_rank=32)
    g = M.MoaraGroup(block_size=B, refresh_src=(M.MOARA_REFRESH_SRC_V if src == "V"
                                                 else M.MOARA_REFRESH_SRC_G))
    for (m, n, r) in shapes:
        g.add(m, n, r, "bf16")
    g.refresh([_dev(grads[i][0]) for i in range(len(shapes))])
    torch.cuda.synchronize()
    assert g.status() == 0
    for i, (m, n, r) in enumerate(shapes):
        P = g.modules[i].P.double().cpu().numpy()
        X = o.decompose(grads[i][0], B)[1] if src == "V" else grads[i][0]
        res = _check(g, g.ids[i], P, X, r)
        print(f"{m}x{n} r={r} src={src}: deficit {res['deficit']:.2e} (float64 method {res['deficit_rsi']:.2e}), |P^T P - I| {res['orth']:.1e}")
        Pb = g.modules[i].P_bf16.view(torch.bfloat16).float().cpu().numpy()
        np.testing.assert_allclose(Pb, P, rtol=2 ** -8, atol=1e-30)
    g.close()


def test_refresh_clear_gap_all_directions(M):
    """Signal sigma_i = 10 * 0.7^i of rank r + 8 with a drop after r: all r
    directions, each singular vector individually (consecutive ratio 1/0.7)."""
    m, n, r = 384, 512, 16
    u, v = synth.lowrank_factors(m, n, r + 8, seed=5)
    sig = np.concatenate([10.0 * 0.7 ** np.arange(r), 0.01 * 0.7 ** np.arange(8)])
    G = (u * sig) @ v.T + 1e-4 * np.random.default_rng(1).standard_normal((m, n))
    G = G.astype(np.float32).astype(np.float64)
    g = M.MoaraGroup(block_size=64, refresh_src=M.MOARA_REFRESH_SRC_G)
    g.add(m, n, r, "f32")
    g.refresh([_dev(G, bf16=False)])
    torch.cuda.synchronize()
    P = g.modules[0].P.double().cpu().numpy()
    U = np.linalg.svd(G, full_matrices=False)[0][:, :r]
    assert principal_angles(P, U).max() <= 1e-2
    Po = o.truncated_svd(G, r)[0]
    # columns come in descending order with the oracle's sign convention
    assert np.min(np.sum(P * Po, axis=0)) >= 0.9999
    _check(g, g.ids[0], P, G, r, exact_bar=1e-3)
    g.close()


def test_auto_refresh_step_equals_refresh_then_step(M):
    """Refresh and step on the same step (t = 1, (t-1) mod T = 0) equals the
    two calls made one after the other."""
    shapes = [(512, 256, 64), (256, 512, 32)]
    grads, W0 = make_inputs(shapes, 64, 2, True)
    outs = []
    for mode in ("auto", "manual"):
        g = M.MoaraGroup(block_size=64)
        for i, (m, n, r) in enumerate(shapes):
            g.add(m, n, r, "bf16", W0=W0[i])
        Gs = [_dev(grads[i][0]) for i in range(len(shapes))]
        if mode == "auto":
            g.step(Gs, 1, 1e-3, auto_refresh=True)
        else:
            g.refresh(Gs)
            g.step(Gs, 1, 1e-3, auto_refresh=False)
        torch.cuda.synchronize()
        outs.append([(b.W.clone(), b.P.clone()) for b in g.modules])
        g.close()
    for (wa, pa), (wb, pb) in zip(*outs):
        assert torch.equal(pa, pb) and torch.equal(wa, wb)


def test_refresh_interval(M):
    """auto_refresh runs the refresh exactly when (t - 1) mod T == 0."""
    B = M.binding
    g = M.MoaraGroup(block_size=32, refresh_interval=3)
    g.add(128, 96, 8, "bf16")
    G = _dev(make_inputs([(128, 96, 8)], 32, 1, True)[0][0][0])
    counts = []
    for t in range(1, 8):
        before = B.moara_launch_count(g.ctx)
        g.step([G], t, 1e-3, auto_refresh=True)
        counts.append(B.moara_launch_count(g.ctx) - before)
    torch.cuda.synchronize()
    plain = min(counts)
    assert [c > plain for c in counts] == [True, False, False, True, False, False, True]
    g.close()


def test_refresh_qwen2_7b_gqa_modules_with_step(M):
    """Qwen2-7B shapes with heterogeneous ranks (k/v 512 x 3584 at r = 256,
    q 3584 x 3584 at r = 896): refresh and step on the same step."""
    shapes = [(3584, 3584, 896), (512, 3584, 256), (512, 3584, 256)]
    B = 128
    grads, W0 = make_inputs(shapes, B, 1, True, signal_rank=32)
    g = M.MoaraGroup(block_size=B)
    for i, (m, n, r) in enumerate(shapes):
        g.add(m, n, r, "bf16", W0=W0[i])
    g.step([_dev(grads[i][0]) for i in range(len(shapes))], 1, 1e-3, auto_refresh=True)
    torch.cuda.synchronize()
    assert g.status() == 0
    for i, (m, n, r) in enumerate(shapes):
        P = g.modules[i].P.double().cpu().numpy()
        X = o.decompose(grads[i][0], B)[1]
        res = _check(g, g.ids[i], P, X, r)
        print(f"{m}x{n} r={r}: deficit {res['deficit']:.2e} (float64 method {res['deficit_rsi']:.2e}), |P^T P - I| {res['orth']:.1e}")
        assert np.all(np.isfinite(g.modules[i].W.cpu().numpy()))
    g.close()


def test_refresh_workspace_too_small(M):
    B = M.binding
    g = M.MoaraGroup(block_size=32)
    mid = g.add(128, 128, 16, "bf16")
    tiny = torch.empty(1024, dtype=torch.uint8, device="cuda")
    B.moara_set_refresh_workspace(g.ctx, tiny.data_ptr(), 1024)
    G = torch.zeros(128, 128, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(B.MoaraError) as e:
        B.moara_refresh_projector(g.ctx, [mid], [G.data_ptr()])
    assert e.value.code == B.MOARA_ERR_WORKSPACE
    g.close()


@pytest.mark.parametrize("m", [384, 390])
@pytest.mark.parametrize("src", ["V", "G"])
def test_refresh_clear_gap_bf16_tensor_cores(M, src, m):
    """bf16 gradient: the refresh products run on tensor cores (V = V_hi + V_lo
    in bf16, Q and Z in bf16).  Same clear-gap spectrum as above, exact in
    bf16; all r directions and each singular vector individually, in order and
    with the oracle's sign convention.  m = 390 (not a multiple of 8) takes
    the fp32 CholeskyQR2 of the tall Q instead of the split-precision pass."""
    n, r, B = 512, 16, 64
    u, v = synth.lowrank_factors(m, n, r + 8, seed=5)
    sig = np.concatenate([10.0 * 0.7 ** np.arange(r), 0.01 * 0.7 ** np.arange(8)])
    G = (u * sig) @ v.T + 1e-4 * np.random.default_rng(1).standard_normal((m, n))
    G = synth.to_bf16_exact(G)
    g = M.MoaraGroup(block_size=B, refresh_src=(M.MOARA_REFRESH_SRC_V if src == "V"
                                                 else M.MOARA_REFRESH_SRC_G))
    g.add(m, n, r, "bf16")
    M.moara_profile_enable(g.ctx, True)
    g.refresh([_dev(G)])
    torch.cuda.synchronize()
    prof = M.moara_profile_read(g.ctx)
    assert g.status() == 0
    assert prof["tc_refresh"][1] > 0          # the products ran on tensor cores
    X = o.decompose(G, B)[1] if src == "V" else G
    P = g.modules[0].P.double().cpu().numpy()
    Po = o.truncated_svd(X, r)[0]
    if src == "G":
        np.testing.assert_allclose(P.T @ P, np.eye(r), atol=1e-5)
        assert principal_angles(P, Po).max() <= 1e-2
        assert np.min(np.sum(P * Po, axis=0)) >= 0.9999
        _check(g, g.ids[0], P, X, r, exact_bar=1e-3)
    else:
        # the block normalisation bends V's spectrum: the generic checks, then
        # each vector individually up to the spectral gap
        res = _check(g, g.ids[0], P, X, r)
        assert res["k_gap"] > 0
        k = res["k_gap"]
        assert np.min(np.sum(P[:, :k] * Po[:, :k], axis=0)) >= 0.9999
    g.close()


@pytest.mark.parametrize("m,n,r", [(4096, 11008, 2048), (11008, 4096, 1024)])
def test_refresh_llama2_7b_full_size_modules(M, m, n, r):
    """The refresh at the sizes the bench times: down (4096 x 11008, r = 2048,
    sketch width l = r + p) and gate / up (11008 x 4096, r = 1024); B = 128,
    bf16 G, the bench's recipe (rank-32 signal plus noise)."""
    B = 128
    G = synth.to_bf16_exact(synth.lowrank_grad(m, n, 32, 10.0, 0.01, 1, seed=0, module=3, noise_rel=True))
    g = M.MoaraGroup(block_size=B)
    mid = g.add(m, n, r, "bf16")
    g.refresh([_dev(G)])
    torch.cuda.synchronize()
    assert g.status() == 0
    P = g.modules[0].P.double().cpu().numpy()
    X = o.decompose(G, B)[1]
    res = _check(g, mid, P, X, r)
    print(f"{m}x{n} r={r}: deficit {res['deficit']:.2e} (float64 method {res['deficit_rsi']:.2e}), k_gap {res['k_gap']}, |P^T P - I| {res['orth']:.1e}")
    g.close()
