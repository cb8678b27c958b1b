"""Parity at the two 7B-shaped single-layer workloads, every module against
the float64 oracle.

* Llama-2-7B-shaped layer (hidden 4096, MLP 11008; q/k r = 512, v/o/gate/
  up/down r = 1024; B = 128; bf16 G, fp32 W and moments): ten Adam steps,
  max relative error of W <= 2e-3 on each of the seven modules.  The
  projector is a fixed bf16-exact orthonormal matrix on both sides (the
  refresh is checked on its own below and in the refresh tests).
* Qwen2-7B-shaped GQA layer (hidden 3584, k/v 512 x 3584, MLP 18944; q/o
  r = 896, k/v 256, MLP 1024; B = 128): the first step refreshes every
  projector and steps in the same call (auto_refresh, (t - 1) mod T = 0),
  then a second step.  Each device projector is checked for P^T P = I,
  principal angles up to the spectral gap against the exact top-r subspace,
  and captured energy against the float64 restatement of the library's
  randomized method with the same sketch (tests/gpu_helpers.check_refresh);
  W is then checked against the oracle run with the device's own bf16
  projector (the top-r subspace near r lies in V's flat noise bulk, where no
  two correct methods agree on the individual vectors), refresh off, at
  2e-3.

The oracle recomputes one module at a time; gradients are drawn one step at a
time (the whole layer's ten steps would not fit the host comfortably).
"""

import numpy as np
import pytest

from oracle import moara_ref as o
import synth

from gpu_helpers import rel_err, check_refresh
from oracle import rsi_ref as R

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

LR = 1e-3


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2609_15037_gb300 as pkg
    return pkg


def _grad(md, i, t, wl):
    return synth.to_bf16_exact(synth.lowrank_grad(md.m, md.n, wl["signal_rank"], wl["sigma0"],
                                                  wl["noise"], t, seed=0, module=i,
                                                  noise_rel=wl["noise_rel"]))


def _dev(G):
    return torch.tensor(G, dtype=torch.float32).to(torch.bfloat16).cuda()


def test_llama2_7b_layer_ten_steps(M):
    wl = synth.workload("llama7b_layer")
    mods, B = wl["modules"], wl["block_size"]
    steps = 10
    g = M.MoaraGroup(block_size=B, adam_eps=wl["adam_eps"], scale=0.25, precision=M.MOARA_PREC_BF16_TC)
    hp_o = o.Hparams(block_size=B, adam_eps=wl["adam_eps"], scale=0.25)
    states = []
    for i, md in enumerate(mods):
        W0 = synth.init_weight(md.m, md.n, seed=0, module=i)
        P = synth.to_bf16_exact(synth.random_orthonormal(md.m, md.r, seed=0, module=i))
        mid = g.add(md.m, md.n, md.r, "bf16", W0=W0)
        g.load_projector(mid, P)
        states.append(o.init_state(W0, md.r, B, P=P))
    M.moara_profile_enable(g.ctx, True)
    for t in range(1, steps + 1):
        Gs = [_grad(md, i, t, wl) for i, md in enumerate(mods)]
        g.step([_dev(G) for G in Gs], t, LR)
        for i in range(len(mods)):
            states[i] = o.step(states[i], Gs[i], t, LR, hp_o, refresh=False)
    torch.cuda.synchronize()
    prof = M.moara_profile_read(g.ctx)
    assert g.status() == 0
    assert prof["tc_project"][1] == steps and prof["tc_backproject"][1] == steps
    for i, md in enumerate(mods):
        W = g.modules[i].W.double().cpu().numpy()
        assert rel_err(W, states[i].W) <= 2e-3, md.name
    g.close()


def test_qwen2_7b_layer_refresh_and_step(M):
    wl = synth.workload("qwen2_7b_layer")
    mods, B = wl["modules"], wl["block_size"]
    g = M.MoaraGroup(block_size=B, adam_eps=wl["adam_eps"], scale=0.25, precision=M.MOARA_PREC_BF16_TC)
    hp_o = o.Hparams(block_size=B, adam_eps=wl["adam_eps"], scale=0.25)
    W0s = []
    for i, md in enumerate(mods):
        W0 = synth.init_weight(md.m, md.n, seed=0, module=i)
        g.add(md.m, md.n, md.r, "bf16", W0=W0)
        W0s.append(W0)
    G1 = [_grad(md, i, 1, wl) for i, md in enumerate(mods)]
    g.step([_dev(G) for G in G1], 1, LR, auto_refresh=True)
    torch.cuda.synchronize()
    assert g.status() == 0
    Pb = []
    hp = g.hp
    for i, md in enumerate(mods):
        P = g.modules[i].P.double().cpu().numpy()
        V = o.decompose(G1[i], B)[1]
        res = check_refresh(P, V, md.r, hp.oversample, hp.power_iters, R.sketch_key(hp.seed, g.ids[i], 0))
        print(f"{md.name} {md.m}x{md.n} r={md.r}: deficit {res['deficit']:.2e} "
              f"(float64 method {res['deficit_rsi']:.2e}), k_gap {res['k_gap']}, |P^T P - I| {res['orth']:.1e}")
        Pb.append(g.modules[i].P_bf16.view(torch.bfloat16).double().cpu().numpy())
    # the oracle fed the device's bf16 projector, refresh off
    G2 = [_grad(md, i, 2, wl) for i, md in enumerate(mods)]
    g.step([_dev(G) for G in G2], 2, LR)
    torch.cuda.synchronize()
    assert g.status() == 0
    for i, md in enumerate(mods):
        st = o.run(o.init_state(W0s[i], md.r, B, P=Pb[i]), [G1[i], G2[i]], LR, hp_o, auto_refresh=False)
        W = g.modules[i].W.double().cpu().numpy()
        assert rel_err(W, st.W) <= 2e-3, md.name
    g.close()
