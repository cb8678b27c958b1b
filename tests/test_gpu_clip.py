"""GPU parity of global-norm gradient clipping (App. D.2) against the oracle.

The library computes the total norm of the call's gradients (plus the
caller's extra term) on the device, then the step of the clipped gradients:
with the decomposition on, clipping scales only the block magnitudes (the
direction V of c G is that of G), without it the projection R.  The oracle
clips first (torch.nn.utils.clip_grad_norm_ form) and runs each module's step
on the clipped gradients.  Bars as for the unclipped step: max relative error
of W <= 2e-3 (bf16 G, fp32 states) / 1e-5 (all fp32); the norm and the
coefficient of the last step to 1e-5 relative; a coefficient of 1 leaves the
step bit-identical to the unclipped one.
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


def _dev(G, bf16):
    t = torch.tensor(G, dtype=torch.float32)
    return (t.to(torch.bfloat16) if bf16 else t).cuda()


def _run(M, shapes, B, steps, bf16, clip_norm, decompose=1, extra_sq=0.0, lr=1e-3, precision=None,
         adam_eps=1e-6):
    grads, W0 = make_inputs(shapes, B, steps, bf16, seed=2)
    hp_o = o.Hparams(block_size=B, adam_eps=adam_eps, scale=0.25, decompose=bool(decompose))
    Ps = []
    for i, (m, n, r) in enumerate(shapes):
        P0 = oracle_projector(grads[i][0], r, B, bool(decompose))
        Ps.append(synth.to_bf16_exact(P0) if bf16 else P0)
    # oracle: clip each step's gradients over all modules, then step each module
    states = [o.init_state(W0[i], r, B, P=Ps[i]) for i, (m, n, r) in enumerate(shapes)]
    norm = coef = None
    for t in range(1, steps + 1):
        gs = [grads[i][t - 1] for i in range(len(shapes))]
        if clip_norm > 0:
            gs, norm, coef = o.clip_grads(gs, clip_norm, extra_sq)
        states = [o.step(states[i], gs[i], t, lr, hp_o, False) for i in range(len(shapes))]
    kw = dict(block_size=B, adam_eps=adam_eps, scale=0.25, decompose=decompose, clip_norm=clip_norm)
    if precision is not None:
        kw["precision"] = precision
    g = M.MoaraGroup(**kw)
    for i, (m, n, r) in enumerate(shapes):
        mid = g.add(m, n, r, "bf16" if bf16 else "f32", W0=W0[i])
        g.load_projector(mid, Ps[i])
    if extra_sq:
        g.set_clip_extra(torch.tensor([extra_sq], dtype=torch.float32, device="cuda"))
    for t in range(1, steps + 1):
        g.step([_dev(grads[i][t - 1], bf16) for i in range(len(shapes))], t, lr)
    torch.cuda.synchronize()
    state = g.clip_state().cpu().numpy().copy()
    assert g.status() == 0
    W = [b.W.double().cpu().numpy() for b in g.modules]
    g.close()
    return W, [s.W for s in states], state, norm, coef


SHAPES = [(256, 320, 32), (192, 512, 64), (320, 256, 48)]


@pytest.mark.parametrize("decompose", [1, 0])
def test_clip_tensor_cores(M, decompose):
    W, ref, state, norm, coef = _run(M, SHAPES, 64, 4, True, 1.0, decompose=decompose,
                                     precision=M.MOARA_PREC_BF16_TC)
    assert coef < 0.5                              # the clip is active
    assert state[0] == pytest.approx(norm, rel=1e-5)
    assert state[1] == pytest.approx(coef, rel=1e-5)
    for w, r in zip(W, ref):
        assert rel_err(w, r) <= 2e-3


def test_clip_fp32_path_with_extra_term(M):
    """All-fp32 path (Adam eps 1e-8 as in the fp32 256 x 256 workload)."""
    W, ref, state, norm, coef = _run(M, SHAPES, 64, 4, False, 2.0, extra_sq=25.0,
                                     precision=M.MOARA_PREC_FP32, adam_eps=1e-8)
    assert coef < 0.5
    assert state[0] == pytest.approx(norm, rel=1e-5)
    assert state[1] == pytest.approx(coef, rel=1e-5)
    for w, r in zip(W, ref):
        assert rel_err(w, r) <= 1e-5


def test_clip_inactive_is_bit_identical(M):
    """A threshold above the norm gives coefficient 1: the same bits as no clipping."""
    Wc, _, state, norm, coef = _run(M, SHAPES, 64, 3, True, 1e6, precision=M.MOARA_PREC_BF16_TC)
    W0, _, _, _, _ = _run(M, SHAPES, 64, 3, True, 0.0, precision=M.MOARA_PREC_BF16_TC)
    assert coef == 1.0 and state[1] == 1.0
    for a, b in zip(Wc, W0):
        assert np.array_equal(a, b)


def test_clip_refused_where_the_step_is_split(M):
    g = M.MoaraGroup(block_size=64, clip_norm=1.0)
    mid = g.add(64, 64, 8, "bf16")
    host = torch.zeros(64, 64, dtype=torch.bfloat16).pin_memory()
    with pytest.raises(M.MoaraError) as ei:
        g.step_host([host], 1, 1e-3)
    assert ei.value.code == M.MOARA_ERR_UNSUPPORTED
    g.close()
    hp = M.moara_default_hparams()
    hp.clip_norm = 1.0
    z = torch.zeros(64 * 64, dtype=torch.float32, device="cuda")
    rc = M.moara_step_static_scratch(hp, 64, 64, 8, M.MOARA_DTYPE_F32, z.data_ptr(), z.data_ptr(),
                                     z.data_ptr(), z.data_ptr(), z.data_ptr(), z.data_ptr(), z.data_ptr(),
                                     1, 1e-3)
    assert rc == M.MOARA_ERR_UNSUPPORTED
