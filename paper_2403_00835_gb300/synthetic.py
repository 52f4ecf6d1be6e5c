"""Seeded synthetic inputs: model shapes, random-init weights and prompts.

This module holds no arithmetic of the decoding method.  It is the one module
that both the CUDA path's users (tests, bench) and the oracle are fed from, so
that both sides see identical inputs.

Workload recipe (stand-ins for the paper's trained models and datasets, which
are not available): LLaMA-style decoders with the shapes of LLaMA-2-7B and
Deepseek-coder-7B (Sec. 4.1), every weight matrix and the embedding drawn
i.i.d. N(0, 0.02^2), every RMSNorm gain = 1, and prompts of tokens drawn
uniformly over the vocabulary.
"""
from __future__ import annotations

from dataclasses import dataclass, replace

import numpy as np


@dataclass(frozen=True)
class ModelConfig:
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rms_eps: float
    rope_theta: float
    dtype: str  # "f32" or "bf16"

    @property
    def n_params(self) -> int:
        d, F, V = self.d_model, self.ffn, self.vocab
        dq, dkv = self.n_heads * self.head_dim, self.n_kv_heads * self.head_dim
        per_layer = d * dq + 2 * d * dkv + dq * d + 3 * d * F + 2 * d
        return self.n_layers * per_layer + 2 * V * d + d

    def with_dtype(self, dtype: str) -> "ModelConfig":
        return replace(self, dtype=dtype, name=f"{self.name.split('-')[0]}-{dtype}")


# Tiny fp32 decoder: 2 layers, d 256, 4 heads x 64, SwiGLU 688, vocab 2048.
TINY = ModelConfig("tiny-f32", 2, 256, 4, 4, 64, 688, 2048, 1e-6, 1e4, "f32")
# Same shapes in bf16: exercises the tensor-core path with ragged tiles
# (688 = 5 x 128 + 48 rows, 688 = 10 x 64 + 48 reduction columns).
TINY_BF16 = replace(TINY, name="tiny-bf16", dtype="bf16")
# LLaMA-2-7B shapes.
LLAMA7B = ModelConfig("llama2-7b", 32, 4096, 32, 32, 128, 11008, 32000, 1e-5, 1e4, "bf16")
# Deepseek-coder-7B shapes (vocab 32256, RoPE theta 1e5).
CODER7B = ModelConfig("coder-7b", 32, 4096, 32, 32, 128, 11008, 32256, 1e-6, 1e5, "bf16")

CONFIGS = {c.name: c for c in (TINY, TINY_BF16, LLAMA7B, CODER7B)}

LAYER_KEYS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")


def _torch_dtype(cfg: ModelConfig):
    import torch
    return torch.float32 if cfg.dtype == "f32" else torch.bfloat16


def make_weights(cfg: ModelConfig, seed: int = 0, device: str = "cpu", std: float = 0.02) -> dict:
    """Random-init weights: matrices [out, in] ~ N(0, std^2), gains = 1.

    Values come from torch's generator on ``device`` seeded with ``seed``;
    a given (seed, device type) always gives the same weights.  Generation
    order: tok_emb, then per layer wq, wk, wv, wo, w_gate, w_up, w_down, then
    lm_head."""
    import torch
    dt = _torch_dtype(cfg)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    d, F, V = cfg.d_model, cfg.ffn, cfg.vocab
    dq, dkv = cfg.n_heads * cfg.head_dim, cfg.n_kv_heads * cfg.head_dim

    def mat(rows, cols):
        w = torch.empty((rows, cols), dtype=dt, device=device)
        # draw in fp32 row blocks to bound the temporary
        step = max(1, (1 << 26) // cols)
        for r0 in range(0, rows, step):
            r1 = min(rows, r0 + step)
            blk = torch.randn((r1 - r0, cols), generator=gen, device=device, dtype=torch.float32)
            w[r0:r1].copy_(blk.mul_(std))
        return w

    def ones(n):
        return torch.ones(n, dtype=dt, device=device)

    w = {"tok_emb": mat(V, d)}
    for k in LAYER_KEYS:
        w[k] = []
    for _ in range(cfg.n_layers):
        w["attn_norm"].append(ones(d))
        w["wq"].append(mat(dq, d))
        w["wk"].append(mat(dkv, d))
        w["wv"].append(mat(dkv, d))
        w["wo"].append(mat(d, dq))
        w["mlp_norm"].append(ones(d))
        w["w_gate"].append(mat(F, d))
        w["w_up"].append(mat(F, d))
        w["w_down"].append(mat(d, F))
    w["final_norm"] = ones(d)
    w["lm_head"] = mat(V, d)
    return w


def weights_to(w: dict, device: str) -> dict:
    """Copy of a weight dict on another device (same values)."""
    out = {}
    for k, v in w.items():
        out[k] = [t.to(device) for t in v] if isinstance(v, list) else v.to(device)
    return out


def make_prompts(vocab: int, lens, seed: int = 1) -> list[list[int]]:
    """Prompts of uniform-random tokens; ``lens`` is a list of lengths."""
    rng = np.random.default_rng(seed)
    return [rng.integers(0, vocab, size=int(n)).astype(np.int64).tolist() for n in lens]


def ragged_lens(batch: int, lo: int, hi: int, seed: int = 1) -> list[int]:
    """Prompt lengths uniform in [lo, hi] (inclusive)."""
    rng = np.random.default_rng(seed + 1000)
    return rng.integers(lo, hi + 1, size=batch).astype(np.int64).tolist()


def make_guesses(vocab: int, batch: int, n: int, seed: int = 2) -> list[list[int]]:
    """Explicit guess blocks [batch][n] for single-step tests."""
    rng = np.random.default_rng(seed)
    return rng.integers(0, vocab, size=(batch, n)).astype(np.int64).tolist()


def oracle_arch_kwargs(cfg: ModelConfig) -> dict:
    return dict(n_layers=cfg.n_layers, d_model=cfg.d_model, n_heads=cfg.n_heads,
                n_kv_heads=cfg.n_kv_heads, head_dim=cfg.head_dim, ffn=cfg.ffn,
                vocab=cfg.vocab, rms_eps=cfg.rms_eps, rope_theta=cfg.rope_theta)
