"""The host-gradient step (moara_step_grouped_host) against the device one.

Both run the same kernels on the same gradients; the host variant only adds
the chunked upload from page-locked host memory into two staging buffers on
a copy stream.  So the weights, moments and projectors after a few steps must
be bit-identical, with chunk sizes that put one module, several modules and
all modules in a chunk, with and without the refresh at t = 1.
"""

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


SHAPES = [(256, 320, 32), (384, 256, 64), (200, 136, 24), (512, 512, 128)]


def _run(M, host, chunk_bytes, auto_refresh, steps=3, dtype="bf16"):
    g = M.MoaraGroup(block_size=64)
    grads = []
    for i, (m, n, r) in enumerate(SHAPES):
        g.add(m, n, r, dtype, W0=synth.init_weight(m, n, seed=i))
        if not auto_refresh:
            g.load_projector(i, synth.to_bf16_exact(synth.random_orthonormal(m, r, seed=i)))
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    for t in range(1, steps + 1):
        gs = [synth.lowrank_grad_torch(m, n, 8, 10.0, 0.01, 1, seed=t, module=i, noise_rel=True,
                                       device=torch.device("cuda")).to(tdt)
              for i, (m, n, r) in enumerate(SHAPES)]
        if host:
            hs = [x.cpu().pin_memory() for x in gs]
            g.step_host(hs, t, 1e-3, auto_refresh=auto_refresh, chunk_bytes=chunk_bytes)
            torch.cuda.synchronize()
            grads.append(hs)
        else:
            g.step(gs, t, 1e-3, auto_refresh=auto_refresh)
            torch.cuda.synchronize()
            grads.append(gs)
    assert g.status() == 0
    out = [(b.W.clone(), b.exp_avg.clone(), b.mag_avg.clone(), b.P.clone()) for b in g.modules]
    g.close()
    return out


@pytest.mark.parametrize("chunk_bytes", [1, 300_000, 1 << 30])
@pytest.mark.parametrize("auto_refresh", [False, True])
def test_host_step_equals_device_step(M, chunk_bytes, auto_refresh):
    ref = _run(M, False, None, auto_refresh)
    got = _run(M, True, chunk_bytes, auto_refresh)
    for a, b in zip(ref, got):
        for x, y in zip(a, b):
            assert torch.equal(x, y)


def test_host_step_fp32_gradients(M):
    ref = _run(M, False, None, False, dtype="f32")
    got = _run(M, True, 400_000, False, dtype="f32")
    for a, b in zip(ref, got):
        for x, y in zip(a, b):
            assert torch.equal(x, y)
