"""Seeded synthetic inputs for the RoI mask op: layer-set shapes and value recipes.

This module holds no arithmetic of the method itself.  It is shared by the tests,
the benchmark and the smoke check so that the CUDA library and the CPU oracle are
fed the same tensors.

The paper trains masks on Qwen2.5 models (Sec. 5.1); the weights are not
available here, so every tensor is a seeded random stand-in with the shape of the
corresponding linear layer (nn.Linear layout [out_features, in_features], groups
of M along in_features) and these value distributions:
  * W      ~ N(0, 0.02^2), stored as bfloat16 (frozen weights, Appendix A.4)
  * logits "logw": log(max(|W|, 2^-126)) + N(0, 0.1^2)   (magnitude-initialised)
           "normal": N(0, 1)
  * dWm    ~ N(0, (1e-3)^2), bfloat16 (the upstream gradient of the masked weight)
  * X      ~ N(0, 1), bfloat16 [T, in_features] (a layer's normalised input
           activations, for the masked-linear product; seed 7000 + tensor seed)
Seed of tensor (layer l, projection p in q,k,v,o,gate,up,down = 0..6):
1000 + 16 * l + p.
"""
from __future__ import annotations

from dataclasses import dataclass

PROJS = ("q", "k", "v", "o", "gate", "up", "down")


@dataclass(frozen=True)
class LayerSet:
    name: str
    layers: int
    hidden: int
    kv: int
    inter: int

    def shape(self, proj: str) -> tuple[int, int]:
        h, kv, i = self.hidden, self.kv, self.inter
        return {"q": (h, h), "k": (kv, h), "v": (kv, h), "o": (h, h),
                "gate": (i, h), "up": (i, h), "down": (h, i)}[proj]

    def tensors(self):
        """[(layer, proj_index, rows, cols)] in forward order."""
        out = []
        for layer in range(self.layers):
            for p, proj in enumerate(PROJS):
                r, c = self.shape(proj)
                out.append((layer, p, r, c))
        return out

    @property
    def elements(self) -> int:
        return sum(r * c for _, _, r, c in self.tensors())


LAYER_SETS = {
    "qwen2.5-0.5b": LayerSet("qwen2.5-0.5b", 24, 896, 128, 4864),
    "qwen2.5-1.5b": LayerSet("qwen2.5-1.5b", 28, 1536, 256, 8960),
    "qwen2.5-3b": LayerSet("qwen2.5-3b", 36, 2048, 256, 11008),
    "qwen2.5-7b": LayerSet("qwen2.5-7b", 28, 3584, 512, 18944),
}


@dataclass(frozen=True)
class Config:
    """One benchmark / parity configuration."""
    name: str
    layer_set: str | None          # None: the single tiny layer
    nm: tuple                      # ((N, M), ...)
    taus: tuple
    logits: str                    # "logw" or "normal"
    rows: int = 0
    cols: int = 0


CONFIGS = {
    "tiny": Config("tiny", None, ((2, 4),), (1.0,), "logw", rows=128, cols=256),
    "qwen2.5-0.5b": Config("qwen2.5-0.5b", "qwen2.5-0.5b", ((2, 4),), (1.0, 0.1), "logw"),
    "qwen2.5-1.5b": Config("qwen2.5-1.5b", "qwen2.5-1.5b", ((4, 8),), (0.5,), "normal"),
    "qwen2.5-3b": Config("qwen2.5-3b", "qwen2.5-3b", ((8, 16), (16, 32)), (0.2,), "logw"),
    "qwen2.5-7b": Config("qwen2.5-7b", "qwen2.5-7b", ((2, 4), (4, 8)), (1.0,), "normal"),
}


def tensor_seed(layer: int, proj: int) -> int:
    return 1000 + 16 * layer + proj


def make_inputs(rows: int, cols: int, logits: str, seed: int, device="cpu"):
    """(W bf16, logits fp32, dWm bf16) for one tensor, from one seeded generator."""
    import torch
    g = torch.Generator(device=device).manual_seed(int(seed))
    W = (torch.randn(rows, cols, generator=g, device=device) * 0.02).to(torch.bfloat16)
    noise = torch.randn(rows, cols, generator=g, device=device)
    if logits == "logw":
        phi = torch.log(W.float().abs().clamp_min(2.0 ** -126)) + 0.1 * noise
    elif logits == "normal":
        phi = noise
    else:
        raise ValueError(logits)
    dWm = (torch.randn(rows, cols, generator=g, device=device) * 1e-3).to(torch.bfloat16)
    return W, phi.contiguous(), dWm


def make_tokens(T: int, cols: int, seed: int, device="cpu"):
    """X bf16 [T, cols] ~ N(0, 1): the input tokens of one linear layer."""
    import torch
    g = torch.Generator(device=device).manual_seed(7000 + int(seed))
    return torch.randn(T, cols, generator=g, device=device).to(torch.bfloat16).contiguous()


def bf16_bits(t):
    """A bfloat16 torch tensor's raw bit patterns as a numpy uint16 array."""
    import numpy as np
    import torch
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
