"""The allocation-free single-module step (moara_step_static_scratch).

Some callers cannot allocate device memory when they run the optimizer step:
their host application owns the GPU's memory through its own pool, or their
step loop cannot afford the synchronisation an allocation implies.  For them
the library offers one entry point whose scratch lives in a fixed array built
into the library.  These tests check, through the C ABI, that two calls in a
row give the same result as the grouped step on the fp32 path and as the
float64 oracle, within the fp32 path's tolerance (max relative error of W
1e-5); that a ragged shape (block size not dividing n, r*n and m*ceil(n/B)
not multiples of 64) keeps the scratch regions apart; that a call after the
first allocates no device memory; and that a request larger than the array is
refused without touching anything.  They live in their own file, collected
last, and run alone or after the other tests.
"""

import numpy as np
import pytest

import synth
from oracle import moara_ref as o

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def _rel(a, b):
    a = a.double().cpu().numpy() if hasattr(a, "cpu") else np.asarray(a, dtype=np.float64)
    b = b.double().cpu().numpy() if hasattr(b, "cpu") else np.asarray(b, dtype=np.float64)
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))


def _case(M, m, n, r, B, dtype, decompose, seed=3):
    lr = 1e-3
    hp = M.moara_default_hparams()
    hp.block_size = B
    hp.decompose = decompose
    hp.precision = M.MOARA_PREC_FP32
    g = M.MoaraGroup(hp)
    W0 = synth.init_weight(m, n, seed=seed)
    mid = g.add(m, n, r, dtype, W0=W0)
    P0 = synth.random_orthonormal(m, r, seed=seed)
    g.load_projector(mid, P0)
    ref = g.modules[0]

    dev = torch.device("cuda")
    W = torch.tensor(W0, dtype=torch.float32, device=dev)
    P = torch.tensor(P0, dtype=torch.float32, device=dev)
    ea = torch.zeros(r, n, device=dev)
    eas = torch.zeros(r, n, device=dev)
    kb = -(-n // B)
    ma = torch.zeros(m, kb, device=dev)
    mas = torch.zeros(m, kb, device=dev)
    gdt = M.MOARA_DTYPE_BF16 if dtype == "bf16" else M.MOARA_DTYPE_F32
    grads = synth.grads_for_steps(m, n, 8, 10.0, 0.01, 2, seed=seed, noise_rel=True,
                                  bf16=(dtype == "bf16"))
    # the oracle on the same inputs: P fixed (no refresh), the same W0
    ohp = o.Hparams(block_size=B, adam_eps=hp.adam_eps, decompose=bool(decompose))
    ost = o.init_state(W0, r, B, P=np.asarray(P.double().cpu().numpy()))
    for t in (1, 2):
        Gt = torch.tensor(grads[t - 1], dtype=torch.float32, device=dev)
        if dtype == "bf16":
            Gt = Gt.to(torch.bfloat16)
        g.step([Gt], t, lr)
        rc = M.moara_step_static_scratch(hp, m, n, r, gdt, Gt.data_ptr(), W.data_ptr(),
                                         P.data_ptr(), ea.data_ptr(), eas.data_ptr(),
                                         ma.data_ptr(), mas.data_ptr(), t, lr, 0)
        assert rc == M.MOARA_OK
        torch.cuda.synchronize()
        ost = o.step(ost, grads[t - 1], t, lr, ohp, refresh=False)
        assert _rel(W, ref.W) <= 1e-5
        assert _rel(ea, ref.exp_avg) <= 1e-5
        assert _rel(W, ost.W) <= 1e-5
        assert _rel(ea, ost.exp_avg) <= 1e-5
        if decompose:
            assert _rel(ma, ref.mag_avg) <= 1e-5
            assert _rel(ma, ost.mag_avg) <= 1e-5
    g.close()


@pytest.mark.parametrize("dtype,decompose", [("bf16", 1), ("f32", 1), ("bf16", 0)])
def test_static_scratch_step_matches_grouped_step_and_oracle(M, dtype, decompose):
    _case(M, 320, 448, 40, 64, dtype, decompose)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_static_scratch_ragged_shape(M, dtype):
    """B = 64 does not divide n = 450 (a ragged last block); r*n = 16650 and
    m*ceil(n/B) = 1600 are not multiples of 64, so each scratch region starts
    at a rounded offset."""
    _case(M, 200, 450, 37, 64, dtype, 1, seed=5)


def test_static_scratch_allocates_nothing(M):
    """After a first accepted call on the device (which may load the module
    holding the array), a further call leaves the device's free memory
    unchanged."""
    m, n, r, B = 256, 384, 32, 64
    hp = M.moara_default_hparams()
    hp.block_size = B
    dev = torch.device("cuda")
    W = torch.zeros(m, n, device=dev)
    G = torch.ones(m, n, device=dev, dtype=torch.bfloat16)
    P = torch.tensor(synth.random_orthonormal(m, r, seed=1), dtype=torch.float32, device=dev)
    ea = torch.zeros(r, n, device=dev)
    eas = torch.zeros(r, n, device=dev)
    ma = torch.zeros(m, n // B, device=dev)
    mas = torch.zeros(m, n // B, device=dev)
    args = (hp, m, n, r, M.MOARA_DTYPE_BF16, G.data_ptr(), W.data_ptr(), P.data_ptr(),
            ea.data_ptr(), eas.data_ptr(), ma.data_ptr(), mas.data_ptr())
    assert M.moara_step_static_scratch(*args, 1, 1e-3, 0) == M.MOARA_OK
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info(dev)
    assert M.moara_step_static_scratch(*args, 2, 1e-3, 0) == M.MOARA_OK
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info(dev)
    assert free1 == free0
    assert torch.isfinite(W).all()


def test_static_scratch_rejects_oversized_request(M):
    hp = M.moara_default_hparams()
    hp.block_size = 128
    m = n = 4096
    r = 1024                        # N alone needs 16 MiB: over the limit
    dev = torch.device("cuda")
    W = torch.zeros(m, n, device=dev)
    before = W.clone()
    G = torch.ones(m, n, device=dev, dtype=torch.bfloat16)
    P = torch.zeros(m, r, device=dev)
    ea = torch.zeros(r, n, device=dev)
    eas = torch.zeros(r, n, device=dev)
    ma = torch.zeros(m, 32, device=dev)
    mas = torch.zeros(m, 32, device=dev)
    rc = M.moara_step_static_scratch(hp, m, n, r, M.MOARA_DTYPE_BF16, G.data_ptr(), W.data_ptr(),
                                     P.data_ptr(), ea.data_ptr(), eas.data_ptr(), ma.data_ptr(),
                                     mas.data_ptr(), 1, 1e-3, 0)
    torch.cuda.synchronize()
    assert rc == M.MOARA_ERR_WORKSPACE
    assert torch.equal(W, before)


def test_static_scratch_refuses_right_projector_rule(M):
    hp = M.moara_default_hparams()
    hp.block_size = 64
    hp.proj_rule = M.MOARA_PROJ_SMALLER
    m, n, r = 256, 128, 16          # tall: the smaller-side rule would project from the right
    dev = torch.device("cuda")
    W = torch.zeros(m, n, device=dev)
    G = torch.ones(m, n, device=dev, dtype=torch.bfloat16)
    P = torch.zeros(m, r, device=dev)
    ea = torch.zeros(r, n, device=dev)
    ma = torch.zeros(m, 2, device=dev)
    rc = M.moara_step_static_scratch(hp, m, n, r, M.MOARA_DTYPE_BF16, G.data_ptr(), W.data_ptr(),
                                     P.data_ptr(), ea.data_ptr(), ea.data_ptr(), ma.data_ptr(),
                                     ma.data_ptr(), 1, 1e-3, 0)
    assert rc == M.MOARA_ERR_UNSUPPORTED
