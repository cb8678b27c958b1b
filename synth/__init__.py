"""Seeded synthetic inputs shared by the tests, the bench and the smoke check.

This package holds workload shapes and random-input recipes only; it contains
none of the optimizer's arithmetic (no decomposition, projection, Adam or
refresh).  Both the oracle side and the CUDA side receive byte-identical
inputs from here.
"""

from .workloads import (Module, layer_modules, model_modules, WORKLOADS,
                        workload)
from .generators import (lowrank_factors, lowrank_grad, grads_for_steps,
                         init_weight, random_orthonormal, signed_permutation,
                         to_bf16_exact, lowrank_grad_torch)

__all__ = [
    "Module", "layer_modules", "model_modules", "WORKLOADS", "workload",
    "lowrank_factors", "lowrank_grad", "grads_for_steps", "init_weight",
    "random_orthonormal", "signed_permutation", "to_bf16_exact",
    "lowrank_grad_torch",
]
