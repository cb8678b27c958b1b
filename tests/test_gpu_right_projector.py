"""GPU parity of the smaller-side projection rule (GaLore's rule; the
paper's memory model): under MOARA_PROJ_SMALLER a tall weight (m > n) takes
a right projector Q (n x r), R = V Q (m x r) with m x r moments and
dV = N Q^T; square and wide weights keep the left projector, and one grouped
launch mixes both.  Bars as for the left rule: max relative error of W <=
2e-3 (bf16 G, fp32 states) after the steps; the refresh's Q against the
oracle's top-r right singular vectors of V by principal angles <= 1e-2 rad
with Q^T Q = I to 1e-5; the host pipeline bit-identical to the device call.
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import rel_err, make_inputs, principal_angles, gap_index

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def _dev(G):
    return torch.tensor(G, dtype=torch.float32).to(torch.bfloat16).cuda()


def _projector(G, r, B, decompose, right):
    X = o.decompose(G, B)[1] if decompose else G
    return o.truncated_svd(X.T if right else X, r)[0]


def _run(M, shapes, B, steps, decompose=1, state="f32", lr=1e-3, seed=5):
    grads, W0 = make_inputs(shapes, B, steps, True, seed=seed, signal_rank=8)
    hp_o = o.Hparams(block_size=B, adam_eps=1e-6, scale=0.25, decompose=bool(decompose),
                     proj_rule="smaller", state_bf16=(state == "bf16"))
    kw = dict(block_size=B, adam_eps=1e-6, scale=0.25, decompose=decompose, precision=M.MOARA_PREC_BF16_TC,
              proj_rule=M.MOARA_PROJ_SMALLER)
    if state == "bf16":
        kw["state_dtype"] = M.MOARA_DTYPE_BF16
    g = M.MoaraGroup(**kw)
    refs = []
    for i, (m, n, r) in enumerate(shapes):
        right = m > n
        W = o.bf16_round(W0[i]) if state == "bf16" else W0[i]
        P0 = synth.to_bf16_exact(_projector(grads[i][0], r, B, decompose, right))
        refs.append(o.run(o.init_state(W, r, B, P=P0, proj_rule="smaller"), grads[i], lr, hp_o, auto_refresh=False))
        mid = g.add(m, n, r, "bf16", W0=W)
        g.load_projector(mid, P0)
        assert g.modules[i].P.shape == (n if right else m, r)
    for t in range(1, steps + 1):
        g.step([_dev(grads[i][t - 1]) for i in range(len(shapes))], t, lr)
    torch.cuda.synchronize()
    assert g.status() == 0
    out = [b.W.double().cpu().numpy() for b in g.modules]
    g.close()
    return out, refs


MIXED = [(640, 256, 64), (392, 136, 40), (1024, 512, 128), (256, 640, 64), (320, 320, 32)]


def test_right_projector_mixed_group(M):
    out, refs = _run(M, MIXED, 64, 4)
    for i, (w, ref) in enumerate(zip(out, refs)):
        assert rel_err(w, ref.W) <= 2e-3, MIXED[i]


def test_right_projector_galore_mode(M):
    shapes = [(640, 256, 64), (392, 136, 40)]
    out, refs = _run(M, shapes, 64, 4, decompose=0)
    for i, (w, ref) in enumerate(zip(out, refs)):
        assert rel_err(w, ref.W) <= 2e-3, shapes[i]


def test_right_projector_bf16_states(M):
    shapes = [(640, 256, 64), (256, 640, 64)]
    out, refs = _run(M, shapes, 128, 3, state="bf16")
    for i, (w, ref) in enumerate(zip(out, refs)):
        tol = 2e-3 * np.max(np.abs(ref.W)) + 2 * np.exp2(np.floor(np.log2(np.maximum(np.abs(ref.W), 1e-30))) - 7)
        assert np.all(np.abs(w - ref.W) <= tol), shapes[i]


def test_right_projector_refresh(M):
    """A tall gradient with signal sigma_i = 10 * 0.7^i of rank r + 8 and a
    drop after r (refresh source G): the refresh of V^T finds the top-r right
    singular vectors, each one individually, in order, with the oracle's
    sign convention."""
    m, n, r = 768, 256, 16
    u, v = synth.lowrank_factors(m, n, r + 8, seed=5)
    sig = np.concatenate([10.0 * 0.7 ** np.arange(r), 0.01 * 0.7 ** np.arange(8)])
    G = synth.to_bf16_exact((u * sig) @ v.T + 1e-4 * np.random.default_rng(1).standard_normal((m, n)))
    g = M.MoaraGroup(block_size=64, precision=M.MOARA_PREC_BF16_TC, proj_rule=M.MOARA_PROJ_SMALLER,
                     refresh_src=M.MOARA_REFRESH_SRC_G)
    g.add(m, n, r, "bf16")
    g.refresh([_dev(G)])
    torch.cuda.synchronize()
    Q = g.modules[0].P.double().cpu().numpy()
    assert g.status() == 0
    g.close()
    assert Q.shape == (n, r)
    np.testing.assert_allclose(Q.T @ Q, np.eye(r), atol=1e-5)
    Vt = np.linalg.svd(G, full_matrices=False)[2][:r].T
    assert principal_angles(Q, Vt).max() <= 1e-2
    Qo = o.truncated_svd(G.T, r)[0]
    assert np.min(np.sum(Q * Qo, axis=0)) >= 0.9999


def test_right_projector_host_pipeline_bitwise(M):
    m, n, r, B = 640, 256, 64, 64
    grads, W0 = make_inputs([(m, n, r)], B, 3, True, seed=12)
    outs = []
    for host in (False, True):
        g = M.MoaraGroup(block_size=B, precision=M.MOARA_PREC_BF16_TC, proj_rule=M.MOARA_PROJ_SMALLER)
        mid = g.add(m, n, r, "bf16", W0=W0[0])
        g.load_projector(mid, synth.to_bf16_exact(synth.random_orthonormal(n, r, seed=2)))
        for t in range(1, 4):
            G = _dev(grads[0][t - 1])
            if host:
                g.step_host([G.cpu().pin_memory()], t, 1e-3, chunk_bytes=1 << 18)
            else:
                g.step([G], t, 1e-3)
        torch.cuda.synchronize()
        outs.append(g.modules[0].W.clone())
        g.close()
    assert torch.equal(outs[0], outs[1])


def test_right_projector_refusals(M):
    g = M.MoaraGroup(block_size=64, proj_rule=M.MOARA_PROJ_SMALLER)
    with pytest.raises(M.MoaraError) as ei:
        g.add(128, 64, 8, "f32")
    assert ei.value.code == M.MOARA_ERR_UNSUPPORTED
    g.close()
