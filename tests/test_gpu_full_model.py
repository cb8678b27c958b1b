"""Full-size parity: the 224-matrix Llama-2-7B module-aware model (q/k 512,
v/o/gate/up 1024, down 2048; B = 128; bf16 G, fp32 W and states) in the
launch configuration the bench times -- one grouped call over every module,
hence 16 module parts with the decomposition of later parts overlapped with
K1 / K2 of earlier ones -- for ten Adam steps (the first with the V_lo
plane).  The oracle recomputes three sampled modules one by one in float64 on
the same inputs, one step at a time: the first module of the first part
(layer0.q), one in the middle (layer15.gate) and the last module of the last
part (layer31.down).  The other 221 modules get device-drawn gradients (drawn
anew every step) and projectors; modules do not interact, and every W must
stay finite with the device status 0.
Bar: max relative error of W <= 2e-3 on the sampled modules.
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import rel_err

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

SAMPLED = ("layer0.q", "layer15.gate", "layer31.down")
STEPS = 10
LR = 1e-3


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def test_full_model_sampled_modules(M):
    wl = synth.workload("llama2_7b_full_module_aware")
    mods, B = wl["modules"], wl["block_size"]
    assert len(mods) == 224
    g = M.MoaraGroup(block_size=B, adam_eps=wl["adam_eps"], scale=0.25, precision=M.MOARA_PREC_BF16_TC)
    hp_o = o.Hparams(block_size=B, adam_eps=wl["adam_eps"], scale=0.25)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(11)
    states = {}
    for i, md in enumerate(mods):
        if md.name in SAMPLED:
            W0 = synth.init_weight(md.m, md.n, seed=0, module=i)
            P = synth.to_bf16_exact(synth.random_orthonormal(md.m, md.r, seed=0, module=i))
            mid = g.add(md.m, md.n, md.r, "bf16", W0=W0)
            g.load_projector(mid, P)
            states[i] = o.init_state(W0, md.r, B, P=P)
        else:
            mid = g.add(md.m, md.n, md.r, "bf16")
            g.modules[i].W.normal_(0.0, 0.02, generator=gen)
            Q = torch.linalg.qr(torch.randn(md.m, md.r, device="cuda", generator=gen))[0]
            g.load_projector(mid, Q)
    for t in range(1, STEPS + 1):
        grads, host = [], {}
        for i, md in enumerate(mods):
            if i in states:
                G = synth.to_bf16_exact(synth.lowrank_grad(md.m, md.n, 32, 10.0, 0.01, t, seed=0, module=i,
                                                           noise_rel=True))
                host[i] = G
                grads.append(torch.tensor(G, dtype=torch.float32).to(torch.bfloat16).cuda())
            else:
                grads.append((torch.randn(md.m, md.n, device="cuda", generator=gen) * 0.05).to(torch.bfloat16))
        g.step(grads, t, LR)
        for i, G in host.items():
            states[i] = o.step(states[i], G, t, LR, hp_o, refresh=False)
        torch.cuda.synchronize()
        del grads
    assert g.status() == 0
    for i, md in enumerate(mods):
        if i not in states:
            assert bool(torch.isfinite(g.modules[i].W).all()), md.name
    for i, st in states.items():
        W = g.modules[i].W.double().cpu().numpy()
        assert rel_err(W, st.W) <= 2e-3, mods[i].name
    g.close()
