"""Workload shapes: the target weights of one decoder layer or a whole model.

Shapes follow PyTorch ``nn.Linear`` (out, in): q/k/v/o are (q_out, hidden)
etc.; gate/up are (mlp, hidden) and down is (hidden, mlp).  The rank tables are
the literal per-module ranks of each workload (not computed here).
"""

from __future__ import annotations

from dataclasses import dataclass

MODULE_TYPES = ("q", "k", "v", "o", "gate", "up", "down")


@dataclass(frozen=True)
class Module:
    name: str       # e.g. "layer3.down"
    mtype: str      # one of MODULE_TYPES
    m: int          # rows (out features)
    n: int          # cols (in features)
    r: int          # projection rank


def _shapes(hidden, mlp, q_out, kv_out):
    return {
        "q": (q_out, hidden), "k": (kv_out, hidden), "v": (kv_out, hidden),
        "o": (hidden, q_out), "gate": (mlp, hidden), "up": (mlp, hidden),
        "down": (hidden, mlp),
    }


def layer_modules(hidden, mlp, ranks, q_out=None, kv_out=None, prefix="layer0"):
    """The seven target matrices of one decoder layer with their ranks."""
    q_out = hidden if q_out is None else q_out
    kv_out = hidden if kv_out is None else kv_out
    shp = _shapes(hidden, mlp, q_out, kv_out)
    return [Module(f"{prefix}.{t}", t, shp[t][0], shp[t][1], int(ranks[t]))
            for t in MODULE_TYPES]


def model_modules(layers, hidden, mlp, ranks, q_out=None, kv_out=None):
    out = []
    for layer in range(layers):
        out += layer_modules(hidden, mlp, ranks, q_out, kv_out, f"layer{layer}")
    return out


def _uniform(r):
    return {t: r for t in MODULE_TYPES}


# Module-aware table at r_base = 1024 (q/k donors at r/2, down receiver at 2r).
RANKS_7B_MODULE_AWARE = {"q": 512, "k": 512, "v": 1024, "o": 1024,
                         "gate": 1024, "up": 1024, "down": 2048}
RANKS_7B_LAYER = {"q": 512, "k": 512, "v": 1024, "o": 1024,
                  "gate": 1024, "up": 1024, "down": 1024}
RANKS_300M = {"q": 128, "k": 128, "v": 256, "o": 256,
              "gate": 256, "up": 256, "down": 256}
RANKS_QWEN2_7B = {"q": 896, "k": 256, "v": 256, "o": 896,
                  "gate": 1024, "up": 1024, "down": 1024}


def _wl(**kw):
    return kw


# Each workload: modules, block size, gradient dtype, signal recipe.
WORKLOADS = {
    # Single 256x256 fp32 module, rank-8 signal (sigma_i = 10 * 0.7^i) plus
    # N(0, 0.01^2) noise; r = 32, B = 64; Adam eps 1e-8, lr 1e-3, 10 steps;
    # P from the SVD of the first G, never refreshed.
    "single_fp32_256": _wl(
        modules=[Module("single", "q", 256, 256, 32)], block_size=64,
        grad_dtype="f32", signal_rank=8, sigma0=10.0, noise=0.01,
        noise_rel=False, adam_eps=1e-8, lr=1e-3, steps=10),
    # One Llama-style 300M-shaped layer: hidden 1024, 16 heads x 64, MLP 2816.
    "llama300m_layer": _wl(
        modules=layer_modules(1024, 2816, RANKS_300M), block_size=64,
        grad_dtype="bf16", signal_rank=32, sigma0=10.0, noise=0.01,
        noise_rel=True, adam_eps=1e-6, lr=1e-3, steps=10),
    # One Llama-2-7B-shaped layer: hidden 4096, 32 heads x 128, MLP 11008.
    "llama7b_layer": _wl(
        modules=layer_modules(4096, 11008, RANKS_7B_LAYER), block_size=128,
        grad_dtype="bf16", signal_rank=32, sigma0=10.0, noise=0.01,
        noise_rel=True, adam_eps=1e-6, lr=1e-3, steps=10),
    # One Qwen2-7B-shaped GQA layer: hidden 3584, 28 q / 4 kv heads x 128,
    # MLP 18944.
    "qwen2_7b_layer": _wl(
        modules=layer_modules(3584, 18944, RANKS_QWEN2_7B, q_out=3584,
                              kv_out=512), block_size=128,
        grad_dtype="bf16", signal_rank=32, sigma0=10.0, noise=0.01,
        noise_rel=True, adam_eps=1e-6, lr=1e-3, steps=10),
    # Full models: 32-layer Llama-2-7B (224 matrices) and 30-layer
    # DeepSeek-LLM-7B (210 matrices), uniform rank 1024 or module-aware.
    "llama2_7b_full_module_aware": _wl(
        modules=model_modules(32, 4096, 11008, RANKS_7B_MODULE_AWARE),
        block_size=128, grad_dtype="bf16", signal_rank=32, sigma0=10.0,
        noise=0.01, noise_rel=True, adam_eps=1e-6, lr=1e-3, steps=10),
    "llama2_7b_full_uniform": _wl(
        modules=model_modules(32, 4096, 11008, _uniform(1024)),
        block_size=128, grad_dtype="bf16", signal_rank=32, sigma0=10.0,
        noise=0.01, noise_rel=True, adam_eps=1e-6, lr=1e-3, steps=10),
    "deepseek_llm_7b_full_module_aware": _wl(
        modules=model_modules(30, 4096, 11008, RANKS_7B_MODULE_AWARE),
        block_size=128, grad_dtype="bf16", signal_rank=32, sigma0=10.0,
        noise=0.01, noise_rel=True, adam_eps=1e-6, lr=1e-3, steps=10),
    "deepseek_llm_7b_full_uniform": _wl(
        modules=model_modules(30, 4096, 11008, _uniform(1024)),
        block_size=128, grad_dtype="bf16", signal_rank=32, sigma0=10.0,
        noise=0.01, noise_rel=True, adam_eps=1e-6, lr=1e-3, steps=10),
}


def workload(name):
    return WORKLOADS[name]
