"""GPU parity of the alignment diagnostic S(W, t) (§3.2) against the oracle.

S = cos(G, Rep_B(M) (.) (P P^T V)) computed on tensor cores: V enters as
V_hi + V_lo and R^T = V^T P as two bf16 planes, so the product P P^T V
carries about 16 significant bits; the reduction runs in fp32 per thread and
fp64 across threads.  Both sides take the same bf16-exact projector (the
module's bf16 copy is what the tensor-core path applies).  Bar: |S_gpu -
S_oracle| <= 1e-4.  Shapes cover ragged row tiles (m not a multiple of 256,
nor of 8), ragged column tiles, a padded last block, B = 32 / 64 / 128, a
projector spanning the top directions of V (S near 1) and a random one.
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import oracle_projector

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

TOL = 1e-4


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def _dev(G):
    return torch.tensor(G, dtype=torch.float32).to(torch.bfloat16).cuda()


def _case(M, shapes, B, P_mode, seed=0):
    g = M.MoaraGroup(block_size=B, precision=M.MOARA_PREC_BF16_TC)
    grads, refs = [], []
    for i, (m, n, r) in enumerate(shapes):
        G = synth.to_bf16_exact(synth.lowrank_grad(m, n, min(16, m, n), 10.0, 0.01, 0, seed=seed, module=i,
                                                   noise_rel=True))
        if P_mode == "svd":
            P = synth.to_bf16_exact(oracle_projector(G, r, B))
        else:
            P = synth.to_bf16_exact(synth.random_orthonormal(m, r, seed=seed, module=i))
        mid = g.add(m, n, r, "bf16")
        g.load_projector(mid, P)
        grads.append(_dev(G))
        refs.append(o.alignment(G, P, B))
    S = g.alignment(grads).cpu().numpy()
    status = g.status()
    g.close()
    return S, np.array(refs), status


@pytest.mark.parametrize("P_mode", ["svd", "random"])
def test_alignment_small_shapes(M, P_mode):
    shapes = [(192, 320, 24), (196, 328, 40), (520, 264, 64), (64, 1024, 16)]
    S, ref, status = _case(M, shapes, 64, P_mode)
    assert status == 0
    assert np.max(np.abs(S - ref)) <= TOL, (S, ref)
    if P_mode == "svd":
        assert np.all(ref > 0.9)


@pytest.mark.parametrize("B", [32, 128])
def test_alignment_block_sizes(M, B):
    shapes = [(384, 512, 64), (136, 392, 32)]
    S, ref, status = _case(M, shapes, B, "svd", seed=3)
    assert status == 0
    assert np.max(np.abs(S - ref)) <= TOL, (S, ref)


def test_alignment_full_size_module(M):
    """One Llama-2-7B q projection (4096 x 4096, r = 512, B = 128)."""
    S, ref, status = _case(M, [(4096, 4096, 512)], 128, "svd", seed=5)
    assert status == 0
    assert abs(S[0] - ref[0]) <= TOL, (S, ref)


def test_alignment_right_projectors(M):
    """Under the smaller-side rule a tall module's S uses V Q Q^T (its right
    projector); a wide one keeps P P^T V; both in one call."""
    B = 64
    shapes = [(640, 256, 64), (256, 640, 64), (392, 136, 40)]
    g = M.MoaraGroup(block_size=B, precision=M.MOARA_PREC_BF16_TC, proj_rule=M.MOARA_PROJ_SMALLER)
    grads, refs = [], []
    for i, (m, n, r) in enumerate(shapes):
        right = m > n
        G = synth.to_bf16_exact(synth.lowrank_grad(m, n, 16, 10.0, 0.01, 0, seed=9, module=i, noise_rel=True))
        V = o.decompose(G, B)[1]
        P = synth.to_bf16_exact(o.truncated_svd(V.T if right else V, r)[0])
        mid = g.add(m, n, r, "bf16")
        g.load_projector(mid, P)
        grads.append(_dev(G))
        refs.append(o.alignment(G, P, B, right=right))
    S = g.alignment(grads).cpu().numpy()
    assert g.status() == 0
    g.close()
    assert np.max(np.abs(S - np.array(refs))) <= TOL, (S, refs)


def test_alignment_errors(M):
    g = M.MoaraGroup(block_size=64)
    mid = g.add(64, 64, 8, "f32")
    G = torch.zeros(64, 64, dtype=torch.float32, device="cuda")
    with pytest.raises(M.MoaraError) as ei:
        g.alignment([G], ids=[mid])
    assert ei.value.code == M.MOARA_ERR_UNSUPPORTED
    assert g.alignment([], ids=[]).numel() == 0
    assert g.status() == 0
    g.close()
