"""GPU parity of the tensor-core (tcgen05) step kernels against the oracle.

bf16 operands with fp32 accumulation and fp32 states: the bar is max
relative error of W <= 2e-3 after the given steps, on the same seeded inputs
and projector as the oracle.  On this path the projector is applied in bf16,
so the tests hand both sides a bf16-representable P; the projection keeps
V = V_hi + V_lo (two bf16 tiles), so R = P^T V carries about 16 significant
bits and the sign-like first Adam step does not amplify rounding.  Shapes cover K tails (m not a multiple
of 64), partial rank tiles (r not a multiple of 128 / 256), partial column
tiles, the last block padded (B does not divide n), every supported B and the
plain GaLore mode.
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import rel_err, make_inputs, oracle_projector

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


def run_tc(M, shapes, B, steps, lr=1e-3, decompose=1, P_mode="svd", seed=0, check_tc=True):
    hp_o = o.Hparams(block_size=B, adam_eps=1e-6, scale=0.25, decompose=bool(decompose))
    grads, W0 = make_inputs(shapes, B, steps, True, seed=seed, signal_rank=8)
    g = M.MoaraGroup(block_size=B, adam_eps=1e-6, scale=0.25, decompose=decompose,
                     precision=M.MOARA_PREC_BF16_TC)
    refs = []
    for i, (m, n, r) in enumerate(shapes):
        if P_mode == "svd":
            P0 = oracle_projector(grads[i][0], r, B, bool(decompose))
        else:
            P0 = synth.random_orthonormal(m, r, seed=seed, module=i)
        P0 = synth.to_bf16_exact(P0)
        refs.append(o.run(o.init_state(W0[i], r, B, P=P0), grads[i], lr, hp_o, auto_refresh=False))
        mid = g.add(m, n, r, "bf16", W0=W0[i])
        g.load_projector(mid, P0)
    M.moara_profile_enable(g.ctx, True)
    for t in range(1, steps + 1):
        g.step([_dev(grads[i][t - 1]) for i in range(len(shapes))], t, lr)
    torch.cuda.synchronize()
    prof = M.moara_profile_read(g.ctx)
    assert g.status() == 0
    if check_tc:
        assert prof["tc_project"][1] == steps and prof["tc_backproject"][1] == steps
        assert prof["project"][1] == 0 and prof["backproject"][1] == 0
    out = [b.W.double().cpu().numpy() for b in g.modules]
    extra = [(b.mag_avg.double().cpu().numpy(), b.exp_avg.double().cpu().numpy()) for b in g.modules]
    g.close()
    return out, refs, extra


def test_tc_llama300m_layer(M):
    """One Llama-style 300M layer (q/k r = 128, others 256, B = 64), 10 steps."""
    wl = synth.workload("llama300m_layer")
    shapes = [(md.m, md.n, md.r) for md in wl["modules"]]
    out, refs, extra = run_tc(M, shapes, 64, 10)
    for i in range(len(shapes)):
        assert rel_err(out[i], refs[i].W) <= 2e-3, wl["modules"][i].name
        # magnitude moments come from fp32 norms of bf16-exact G: tight
        np.testing.assert_allclose(extra[i][0], refs[i].mag_avg, rtol=2e-5, atol=1e-7)


TC_SHAPES = [
    # (m, n, r, B)
    (200, 136, 24, 8),      # K tail, partial rank half, partial column tile
    (200, 392, 136, 16),    # second accumulator half with 8 valid rows
    (300, 200, 200, 128),   # B does not divide n: padded last block
    (520, 512, 256, 32),    # K tail, exactly one rank tile
    (600, 640, 520, 64),    # three rank tiles, last one partial
    (64, 1024, 64, 128),    # a single K stage
]


@pytest.mark.parametrize("m,n,r,B", TC_SHAPES)
def test_tc_ragged_shapes(M, m, n, r, B):
    out, refs, _ = run_tc(M, [(m, n, r)], B, 4, P_mode="random")
    assert rel_err(out[0], refs[0].W) <= 2e-3


def test_tc_update_chunk_layouts_in_one_group(M):
    """One launch group mixing the two ways K2 hands an fp32 update to W: in
    64-row x 64-column chunks through the 3-D view of W (n a multiple of 64;
    here also n = 64, a partial last column tile of 192 columns, and rows
    past m in the second row half of the last row tile) and in 128-row x
    32-column chunks (n not a multiple of 64), with B = 64, three steps."""
    shapes = [(136, 192, 64), (200, 136, 32), (64, 64, 16), (300, 448, 128), (72, 200, 24)]
    out, refs, _ = run_tc(M, shapes, 64, 3, P_mode="random", seed=3)
    for i in range(len(shapes)):
        assert rel_err(out[i], refs[i].W) <= 2e-3, shapes[i]


def test_tc_galore_mode(M):
    """Decomposition off: R = P^T G, W -= lr * alpha * P Adam(R)."""
    shapes = [(384, 256, 64), (256, 512, 128)]
    out, refs, _ = run_tc(M, shapes, 64, 4, decompose=0, P_mode="random")
    for i in range(len(shapes)):
        assert rel_err(out[i], refs[i].W) <= 2e-3


def test_tc_matches_fp32_path_closely(M):
    """The tensor-core and fp32 paths agree on one step of a 7B-like module
    slice (bf16 rounding of V, P and N only)."""
    m, n, r, B = 1024, 1024, 256, 128
    grads, W0 = make_inputs([(m, n, r)], B, 1, True)
    P0 = synth.to_bf16_exact(synth.random_orthonormal(m, r))
    outs = []
    for prec in (M.MOARA_PREC_FP32, M.MOARA_PREC_BF16_TC):
        g = M.MoaraGroup(block_size=B, precision=prec)
        mid = g.add(m, n, r, "bf16", W0=W0[0])
        g.load_projector(mid, P0)
        g.step([_dev(grads[0][0])], 1, 1e-3)
        torch.cuda.synchronize()
        outs.append(g.modules[0].W.double().cpu().numpy() - W0[0])
        g.close()
    dW32, dWtc = outs
    assert np.linalg.norm(dWtc - dW32) / np.linalg.norm(dW32) <= 2e-3
