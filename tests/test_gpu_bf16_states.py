"""GPU parity of the bf16-state mode (W and the direction moments in bf16,
the magnitude moments in fp32: the paper's runs, App. D.2 / App. G) against
the oracle with the same storage rounding.

Both sides compute each update in higher precision and store it rounded to
the nearest bf16; the device's update carries the bf16-operand error of the
tensor-core path (about 2^-9 of the update), so an entry can land on the
other side of a bf16 rounding boundary, which moves it by one bf16 unit
(2^-8 to 2^-7 of the entry), and such moves can meet over the steps.  Bar:
every W entry within the fp32-state bar (2e-3 of max |W|, the operand error
of the update) plus two bf16 units of the entry, and at most a quarter of
the entries different at all; the moments within two bf16 units plus 1e-3
of their largest entry (their inputs carry the same operand error).  Shapes
cover ragged rank and column tiles, B = 32 / 64 / 128, the first step (V_lo
plane) and later steps; the host pipeline gives the same bits as the device
call.
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import make_inputs, oracle_projector

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


def _run(M, shapes, B, steps, lr=1e-3, seed=4):
    grads, W0 = make_inputs(shapes, B, steps, True, seed=seed, signal_rank=8)
    hp_o = o.Hparams(block_size=B, adam_eps=1e-6, scale=0.25, state_bf16=True)
    g = M.MoaraGroup(block_size=B, adam_eps=1e-6, scale=0.25, precision=M.MOARA_PREC_BF16_TC,
                     state_dtype=M.MOARA_DTYPE_BF16)
    refs = []
    for i, (m, n, r) in enumerate(shapes):
        W0b = o.bf16_round(W0[i])
        P0 = synth.to_bf16_exact(oracle_projector(grads[i][0], r, B))
        refs.append(o.run(o.init_state(W0b, r, B, P=P0), grads[i], lr, hp_o, auto_refresh=False))
        mid = g.add(m, n, r, "bf16", W0=W0b)
        g.load_projector(mid, P0)
    for t in range(1, steps + 1):
        g.step([_dev(grads[i][t - 1]) for i in range(len(shapes))], t, lr)
    torch.cuda.synchronize()
    assert g.status() == 0
    out = [(b.W.double().cpu().numpy(), b.exp_avg.double().cpu().numpy(), b.exp_avg_sq.double().cpu().numpy())
           for b in g.modules]
    g.close()
    return out, refs


def _ulp(a, b):
    """One bf16 unit of max(|a|, |b|) entrywise (8 significant bits)."""
    x = np.maximum(np.maximum(np.abs(a), np.abs(b)), 1e-30)
    return np.exp2(np.floor(np.log2(x)) - 7)


def _check(got, ref, label):
    W, ea, es = got
    dW = np.abs(W - ref.W)
    tol = 2e-3 * np.max(np.abs(ref.W)) + 2 * _ulp(W, ref.W)
    assert np.all(dW <= tol), (label, float(np.max(dW / tol)))
    assert np.mean(dW > 0) <= 0.25, (label, float(np.mean(dW > 0)))
    for x, y in ((ea, ref.exp_avg), (es, ref.exp_avg_sq)):
        assert np.all(np.abs(x - y) <= 2 * _ulp(x, y) + 1e-3 * np.max(np.abs(y))), label


@pytest.mark.parametrize("B", [64, 128])
def test_bf16_states_shapes(M, B):
    shapes = [(256, 320, 32), (192, 512, 64), (136, 264, 40)]
    out, refs = _run(M, shapes, B, 4)
    for i, (got, ref) in enumerate(zip(out, refs)):
        assert np.array_equal(o.bf16_round(got[0]), got[0])      # W is stored as bf16
        _check(got, ref, shapes[i])


def test_bf16_states_block32_llama300m_attention(M):
    shapes = [(1024, 1024, 128), (1024, 1024, 256)]
    out, refs = _run(M, shapes, 32, 6, seed=7)
    for i, (got, ref) in enumerate(zip(out, refs)):
        _check(got, ref, shapes[i])


def test_bf16_states_host_pipeline_bitwise(M):
    m, n, r, B = 256, 512, 64, 64
    grads, W0 = make_inputs([(m, n, r)], B, 3, True, seed=9)
    outs = []
    for host in (False, True):
        g = M.MoaraGroup(block_size=B, precision=M.MOARA_PREC_BF16_TC, state_dtype=M.MOARA_DTYPE_BF16)
        mid = g.add(m, n, r, "bf16", W0=o.bf16_round(W0[0]))
        g.load_projector(mid, synth.to_bf16_exact(synth.random_orthonormal(m, r, seed=1)))
        for t in range(1, 4):
            G = _dev(grads[0][t - 1])
            if host:
                g.step_host([G.cpu().pin_memory()], t, 1e-3, chunk_bytes=1 << 20)
            else:
                g.step([G], t, 1e-3)
        torch.cuda.synchronize()
        outs.append(g.modules[0].W.clone())
        g.close()
    assert torch.equal(outs[0], outs[1])


def test_bf16_states_refused_off_the_tensor_core_path(M):
    g = M.MoaraGroup(block_size=64, state_dtype=M.MOARA_DTYPE_BF16)
    with pytest.raises(M.MoaraError) as ei:
        g.add(64, 64, 8, "f32")
    assert ei.value.code == M.MOARA_ERR_UNSUPPORTED
    g.close()
    g = M.MoaraGroup(block_size=16, state_dtype=M.MOARA_DTYPE_BF16)
    with pytest.raises(M.MoaraError) as ei:
        g.add(64, 64, 8, "bf16")
    assert ei.value.code == M.MOARA_ERR_UNSUPPORTED
    g.close()
