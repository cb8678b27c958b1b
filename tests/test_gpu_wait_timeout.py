"""Failure detection on the device: a bounded wait that runs out.

Every mbarrier wait in the library's kernels is bounded.  When the bound
passes without progress, the kernel records MOARA_ERR_DEVICE_TIMEOUT in the
context's status word, waits (with the default bound) for its own copies and
tensor-core work in flight, frees its tensor memory and returns, so that the
context stays usable.  moara_set_wait_limit lowers the bound of the
single-CTA tensor-core product kernels (the refresh's and the alignment
diagnostic's) to a few hundred cycles -- shorter than any TMA copy takes --
so that their waits give up on purpose.  Nothing faults: no flag is missing
for ever, the waits simply stop early, and the host reads the status.
"""

import numpy as np
import pytest

from gpu_helpers import make_inputs

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


def test_bounded_wait_runs_out_and_context_recovers(M):
    shapes = [(256, 512, 64), (384, 256, 32)]
    B = 64
    grads, W0 = make_inputs(shapes, B, 2, True)
    g = M.MoaraGroup(block_size=B)
    for i, (m, n, r) in enumerate(shapes):
        g.add(m, n, r, "bf16", W0=W0[i])
    G1 = [_dev(grads[i][0]) for i in range(len(shapes))]
    G2 = [_dev(grads[i][1]) for i in range(len(shapes))]
    g.step(G1, 1, 1e-3, auto_refresh=True)
    S_ref = g.alignment(G1).cpu().numpy()
    torch.cuda.synchronize()
    assert g.status() == 0

    M.moara_set_wait_limit(g.ctx, 200)           # far below a TMA copy's latency
    g.alignment(G1)
    torch.cuda.synchronize()
    assert g.status() == M.MOARA_ERR_DEVICE_TIMEOUT

    M.moara_set_wait_limit(g.ctx, 0)             # the default bound again
    S = g.alignment(G1).cpu().numpy()
    torch.cuda.synchronize()
    assert g.status() == 0
    np.testing.assert_allclose(S, S_ref, rtol=0, atol=1e-6)
    # the step kernels and the refresh still run on the same context
    g.refresh(G2)
    g.step(G2, 2, 1e-3)
    torch.cuda.synchronize()
    assert g.status() == 0
    for b in g.modules:
        assert bool(torch.isfinite(b.W).all())
    g.close()
