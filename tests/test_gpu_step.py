"""GPU parity of the optimizer step through the C ABI against the oracle.

Tolerances: max relative error of W (max |W_gpu - W_ref| / max |W_ref|)
<= 1e-5 for the all-fp32 path and <= 2e-3 for bf16 gradients with fp32
states, after 10 steps, on the same seeded inputs and the same projector.
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import rel_err, delta_err, make_inputs, oracle_projector

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def _to_dev(G, bf16):
    t = torch.tensor(G, dtype=torch.float32)
    return (t.to(torch.bfloat16) if bf16 else t).cuda()


def run_both(M, shapes, B, steps, bf16, lr=1e-3, precision=None, seeds=0, hp_kw=None,
             P_mode="svd", grads=None, W0=None):
    hp_kw = dict(hp_kw or {})
    hp_o = o.Hparams(block_size=B, **{k: v for k, v in hp_kw.items()
                                     if k in ("adam_eps", "scale", "decompose", "beta1", "beta2")})
    if grads is None:
        grads, W0 = make_inputs(shapes, B, steps, bf16, seed=seeds)
    ref, Ps = [], []
    for i, (m, n, r) in enumerate(shapes):
        if P_mode == "svd":
            P0 = oracle_projector(grads[i][0], r, B, hp_o.decompose)
        else:
            P0 = synth.random_orthonormal(m, r, seed=seeds, module=i)
        Ps.append(P0)
        ref.append(o.run(o.init_state(W0[i], r, B, P=P0), grads[i], lr, hp_o, auto_refresh=False))
    kw = dict(block_size=B, **hp_kw)
    if precision is not None:
        kw["precision"] = precision
    g = M.MoaraGroup(**kw)
    for i, (m, n, r) in enumerate(shapes):
        mid = g.add(m, n, r, "bf16" if bf16 else "f32", W0=W0[i])
        g.load_projector(mid, Ps[i])
    for t in range(1, steps + 1):
        g.step([_to_dev(grads[i][t - 1], bf16) for i in range(len(shapes))], t, lr)
    torch.cuda.synchronize()
    assert g.status() == 0
    out = [b.W.double().cpu().numpy() for b in g.modules]
    g.close()
    return out, ref, W0


def test_fp32_single_module_256(M):
    """256 x 256 fp32 module, rank-8 signal (10 * 0.7^i) + N(0, 0.01^2) noise,
    r = 32, B = 64, eps 1e-8, lr 1e-3, alpha 0.25, 10 steps, P from the SVD
    of the first G, no refresh: max relative error <= 1e-5."""
    wl = synth.workload("single_fp32_256")
    mod = wl["modules"][0]
    grads = [synth.grads_for_steps(256, 256, 8, 10.0, 0.01, 10, seed=0, noise_rel=False)]
    W0 = [synth.init_weight(256, 256, seed=0)]
    P0 = o.truncated_svd(grads[0][0], 32)[0]        # SVD of the first G
    hp_o = o.Hparams(block_size=64, adam_eps=1e-8, scale=0.25)
    ref = o.run(o.init_state(W0[0], 32, 64, P=P0), grads[0], 1e-3, hp_o, auto_refresh=False)
    g = M.MoaraGroup(block_size=64, adam_eps=1e-8, scale=0.25, precision=M.MOARA_PREC_FP32)
    mid = g.add(mod.m, mod.n, mod.r, "f32", W0=W0[0])
    g.load_projector(mid, P0)
    for t in range(1, 11):
        g.step([_to_dev(grads[0][t - 1], False)], t, 1e-3)
    torch.cuda.synchronize()
    W = g.modules[0].W.double().cpu().numpy()
    g.close()
    assert rel_err(W, ref.W) <= 1e-5
    assert delta_err(W, ref.W, W0[0]) <= 1e-3


@pytest.mark.parametrize("precision", ["fp32"])
def test_bf16_llama300m_layer(M, precision):
    """One Llama-style 300M layer (hidden 1024, MLP 2816), ranks q/k 128,
    others 256, B = 64, bf16 G, fp32 W/states, 10 steps: <= 2e-3."""
    wl = synth.workload("llama300m_layer")
    shapes = [(md.m, md.n, md.r) for md in wl["modules"]]
    prec = M.MOARA_PREC_FP32 if precision == "fp32" else M.MOARA_PREC_BF16_TC
    out, ref, W0 = run_both(M, shapes, 64, 10, True, precision=prec,
                            hp_kw=dict(adam_eps=1e-6, scale=0.25))
    for i in range(len(shapes)):
        assert rel_err(out[i], ref[i].W) <= 2e-3, wl["modules"][i].name


RAGGED = [
    # (m, n, r, B, bf16, decompose)
    (130, 333, 17, 24, True, True),     # padding (333 = 13*24 + 21), ragged tiles
    (257, 129, 129, 64, False, True),   # r = min(m, n), 129 % 64 != 0
    (40, 70, 5, 1, True, True),         # B = 1: V = sign(G)
    (33, 50, 33, 50, False, True),      # B = n: row normalisation, r = m
    (200, 96, 30, 32, True, False),     # plain GaLore (decomposition off)
    (1, 17, 1, 5, False, True),         # a single row
]


@pytest.mark.parametrize("m,n,r,B,bf16,dec", RAGGED)
def test_ragged_and_degenerate_shapes(M, m, n, r, B, bf16, dec):
    out, ref, W0 = run_both(M, [(m, n, r)], B, 4, bf16, precision=M.MOARA_PREC_FP32,
                            hp_kw=dict(adam_eps=1e-8, decompose=int(dec)), P_mode="random")
    assert rel_err(out[0], ref[0].W) <= 1e-5


def test_zero_gradient_blocks(M):
    """A zero block (v = 0) and an all-zero gradient stay finite and match."""
    m, n, r, B = 64, 96, 8, 32
    grads, W0 = make_inputs([(m, n, r), (m, n, r)], B, 3, False)
    for t in range(3):
        grads[0][t][5, 32:64] = 0.0
        grads[1][t][:] = 0.0
    out, ref, _ = run_both(M, [(m, n, r), (m, n, r)], B, 3, False, precision=M.MOARA_PREC_FP32,
                           hp_kw=dict(adam_eps=1e-8), P_mode="random", grads=grads, W0=W0)
    for i in range(2):
        assert np.all(np.isfinite(out[i]))
        assert rel_err(out[i], ref[i].W) <= 1e-5
    np.testing.assert_array_equal(out[1], W0[1].astype(np.float32))


def _group_run(M, shapes, B, grads, W0, Ps, steps, t0=1, g=None, bf16=True, **kw):
    if g is None:
        g = M.MoaraGroup(block_size=B, **kw)
        for i, (m, n, r) in enumerate(shapes):
            mid = g.add(m, n, r, "bf16" if bf16 else "f32", W0=W0[i])
            g.load_projector(mid, Ps[i])
    for t in range(t0, t0 + steps):
        g.step([_to_dev(grads[i][t - 1], bf16) for i in range(len(shapes))], t, 1e-3)
    torch.cuda.synchronize()
    return g


def test_determinism_bitwise(M):
    shapes = [(300, 200, 20), (128, 256, 64)]
    grads, W0 = make_inputs(shapes, 32, 3, True)
    Ps = [synth.random_orthonormal(m, r, module=i) for i, (m, n, r) in enumerate(shapes)]
    a = _group_run(M, shapes, 32, grads, W0, Ps, 3)
    b = _group_run(M, shapes, 32, grads, W0, Ps, 3)
    for x, y in zip(a.modules, b.modules):
        for k in ("W", "exp_avg", "exp_avg_sq", "mag_avg", "mag_avg_sq"):
            assert torch.equal(getattr(x, k), getattr(y, k)), k
    a.close()
    b.close()


def test_checkpoint_resume_bitwise(M):
    """State (W, P, both moment pairs, t) saved mid-run and restored into a
    fresh context continues exactly as an uninterrupted run."""
    shapes = [(192, 160, 24), (96, 256, 16)]
    grads, W0 = make_inputs(shapes, 32, 6, True)
    Ps = [synth.random_orthonormal(m, r, module=i) for i, (m, n, r) in enumerate(shapes)]
    full = _group_run(M, shapes, 32, grads, W0, Ps, 6)
    half = _group_run(M, shapes, 32, grads, W0, Ps, 3)
    saved = [b.state_dict() for b in half.modules]
    half.close()
    g = M.MoaraGroup(block_size=32)
    for i, (m, n, r) in enumerate(shapes):
        g.add(m, n, r, "bf16")
        g.modules[i].load_state_dict(saved[i])
    _group_run(M, shapes, 32, grads, W0, Ps, 3, t0=4, g=g)
    for x, y in zip(full.modules, g.modules):
        for k in ("W", "exp_avg", "exp_avg_sq", "mag_avg", "mag_avg_sq"):
            assert torch.equal(getattr(x, k), getattr(y, k)), k
    full.close()
    g.close()


def test_invalid_arguments_launch_nothing(M):
    B = M.binding
    g = M.MoaraGroup(block_size=32)
    mid = g.add(64, 64, 8, "bf16")
    before = B.moara_launch_count(g.ctx)
    buf = g.modules[0]
    d = buf.desc()
    d.r = 65
    with pytest.raises(B.MoaraError) as e:
        B.moara_init_module(g.ctx, d)
    assert e.value.code == B.MOARA_ERR_RANK
    d = buf.desc()
    d.W = d.W + 4
    with pytest.raises(B.MoaraError) as e:
        B.moara_init_module(g.ctx, d)
    assert e.value.code == B.MOARA_ERR_ALIGN
    d = buf.desc()
    d.workspace_bytes = 16
    with pytest.raises(B.MoaraError) as e:
        B.moara_init_module(g.ctx, d)
    assert e.value.code == B.MOARA_ERR_WORKSPACE
    G = torch.zeros(64, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(B.MoaraError) as e:
        B.moara_step_grouped(g.ctx, [mid + 5], [G.data_ptr()], 1, 1e-3)
    assert e.value.code == B.MOARA_ERR_UNKNOWN_MODULE
    with pytest.raises(B.MoaraError) as e:
        B.moara_step_grouped(g.ctx, [mid], [G.data_ptr() + 2], 1, 1e-3)
    assert e.value.code == B.MOARA_ERR_ALIGN
    with pytest.raises(B.MoaraError) as e:
        B.moara_step_grouped(g.ctx, [mid], [G.data_ptr()], 0, 1e-3)
    assert e.value.code == B.MOARA_ERR_INVALID_ARG
    with pytest.raises(B.MoaraError) as e:
        B.moara_step_grouped(g.ctx, [mid, mid], [G.data_ptr(), G.data_ptr()], 1, 1e-3)
    assert e.value.code == B.MOARA_ERR_INVALID_ARG
    with pytest.raises(B.MoaraError) as e:
        B.moara_refresh_projector(g.ctx, [mid], [G.data_ptr()])
    assert e.value.code == B.MOARA_ERR_WORKSPACE
    assert B.moara_launch_count(g.ctx) == before
    g.close()


@pytest.mark.parametrize("dec", [1, 0])
def test_nan_in_gradient_propagates_as_documented(M, dec):
    """A NaN at G[i, j] makes every column of j's block non-finite (through the
    direction projection), and with decomposition off only column j."""
    m, n, r, Bs = 64, 128, 8, 32
    g = M.MoaraGroup(block_size=Bs, decompose=dec)
    mid = g.add(m, n, r, "bf16", W0=np.zeros((m, n)))
    g.load_projector(mid, synth.random_orthonormal(m, r))
    G = torch.randn(m, n, device="cuda").to(torch.bfloat16)
    G[7, 40] = float("nan")
    g.step([G], 1, 1e-3)
    torch.cuda.synchronize()
    bad = ~torch.isfinite(g.modules[0].W)
    cols = torch.nonzero(bad.any(dim=0)).flatten().tolist()
    if dec:
        assert cols == list(range(32, 64))
    else:
        assert cols == [40]
    g.close()
