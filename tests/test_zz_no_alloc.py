"""The allocation-free single-module step (moara_step_static_scratch).

Some callers cannot allocate device memory when they run the optimizer step
(their host application owns the GPU's memory through its own pool, or their
step loop cannot afford the synchronisation an allocation implies).  For them
the library offers one entry point whose scratch lives in a fixed array built
into the library.  This test checks, through the C ABI, that two calls in a
row give the same result as the grouped step on the fp32 path, within the
fp32 path's tolerance (max relative error of W 1e-5), and that a request
larger than the array is refused without touching anything.  It lives in its
own file, collected last, and runs alone or after the other tests.
"""

import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def _rel(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))


@pytest.mark.parametrize("dtype,decompose", [("bf16", 1), ("f32", 1), ("bf16", 0)])
def test_static_scratch_step_matches_grouped_step(M, dtype, decompose):
    m, n, r, B = 320, 448, 40, 64
    lr = 1e-3
    hp = M.moara_default_hparams()
    hp.block_size = B
    hp.decompose = decompose
    hp.precision = M.MOARA_PREC_FP32
    g = M.MoaraGroup(hp)
    W0 = synth.init_weight(m, n, seed=3)
    mid = g.add(m, n, r, dtype, W0=W0)
    P0 = synth.random_orthonormal(m, r, seed=3)
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
    grads = synth.grads_for_steps(m, n, 8, 10.0, 0.01, 2, seed=3, noise_rel=True,
                                  bf16=(dtype == "bf16"))
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
        assert _rel(W, ref.W) <= 1e-5
        assert _rel(ea, ref.exp_avg) <= 1e-5
        if decompose:
            assert _rel(ma, ref.mag_avg) <= 1e-5
    g.close()


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
