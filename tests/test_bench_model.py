"""CPU checks of the bench's byte and flop model: the algorithmic bytes and
flops of one full-model step of the 224-matrix Llama-2-7B module-aware
workload (G 2mn, W 8mn, direction moments 16rn, P 2mr, magnitude moments
16mk per module; flops 4mrn), the per-kernel bytes of the tensor-core step,
and the binding roof of each product kernel at the measured peaks."""

import importlib.util
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    sys.path.insert(0, ROOT)
    spec = importlib.util.spec_from_file_location("bench_model", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _sums(mods, B):
    smn = sum(md.m * md.n for md in mods)
    srn = sum(md.r * md.n for md in mods)
    smr = sum(md.m * md.r for md in mods)
    smk = sum(md.m * (-(-md.n // B)) for md in mods)
    smrn = sum(md.m * md.r * md.n for md in mods)
    return smn, srn, smr, smk, smrn


def test_full_model_bytes_and_flops(bench):
    import synth
    wl = synth.workload("llama2_7b_full_module_aware")
    mods, B = wl["modules"], wl["block_size"]
    smn, srn, smr, smk, smrn = _sums(mods, B)
    # per layer: 4 x 4096^2 + 3 x 4096 x 11008 entries
    assert smn == 32 * (4 * 4096 * 4096 + 3 * 4096 * 11008)
    tb, tf, _ = bench._algorithmic(mods, B)
    assert tb == 10 * smn + 16 * srn + 2 * smr + 16 * smk
    assert tf == 4 * smrn
    assert tb / 1e9 == pytest.approx(90.63, abs=0.01)
    assert tf / 1e12 == pytest.approx(30.24, abs=0.01)
    kb = bench._kernel_bytes(mods, B, True)
    assert kb["tc_backproject"] == 8 * smn + 2 * srn + 2 * smr + 4 * smk
    assert kb["tc_project"] == 2 * smn + 2 * smr + 18 * srn
    # bf16 states halve W and the moments
    tb2, _, _ = bench._algorithmic(mods, B, 2)
    assert tb2 == 6 * smn + 8 * srn + 2 * smr + 16 * smk


def test_smaller_side_rule_bytes(bench):
    """Under the smaller-side rule gate/up (11008 x 4096) carry m x r moments
    and an n x r projector; the others are unchanged."""
    import synth
    wl = synth.workload("llama2_7b_full_module_aware")
    mods, B = wl["modules"], wl["block_size"]
    left, _, _ = bench._algorithmic(mods, B)
    right, _, _ = bench._algorithmic(mods, B, 4, "smaller")
    tall = [md for md in mods if md.m > md.n]
    assert len(tall) == 64 and all(md.name.split(".")[1] in ("gate", "up") for md in tall)
    delta = sum(16 * md.r * (md.m - md.n) + 2 * md.r * (md.n - md.m) for md in tall)
    assert right - left == delta
