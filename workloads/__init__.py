"""Seeded synthetic workloads for the UniF-MoE layer forward pass.

This module only draws random numbers and arranges them into the tensors a
UniF-MoE layer consumes (Sec. III-A: one shared expert plus K residual
experts, each an FFN of width H split into B aligned blocks; Eq. 17 augmented
router). It contains none of the method's arithmetic: no routing, no scores,
no expert evaluation. Both the CPU oracle and the CUDA path read their inputs
from here, and nothing else is shared between them.

Datasets and pretrained weights from the paper's experiments (DomainBed
images through DeiT-S/16, GLUE text through BERT-large; Sec. IV-A) are not
available, so these generators stand in for them with the same shapes:
197-token ViT sequences at evaluation batch 64, 128-token BERT sequences at
batch 32, FFN widths of ViT-S/ViT-B/BERT-base, experts sparsely upcycled from
one base FFN (a copy plus a small Gaussian perturbation).

Layouts (row-major, the `torch.nn.Linear` weight layout for the experts):
  w_router [d][K+1]      column 0 = W_shr, columns 1..K = W_g  (Eq. 17)
  w_up     [K+1][H][d]   expert 0 = shared; row h is the key K_e[:, h]
  w_down   [K+1][d][H]   column h is the value V_e[h, :]
  x        [T][d]
  mask     [T] uint8 (1 = real token, 0 = padding) or None
  router_bias [K+1] float32 or None (the paper has none; only the
              load-imbalance workload uses one, to skew expert popularity)
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional

import torch

__all__ = ["LayerSpec", "Workload", "CONFIGS", "make_weights", "make_tokens", "make_workload", "spec"]

NAN = float("nan")


@dataclass(frozen=True)
class LayerSpec:
    """Shape and routing thresholds of one UniF-MoE layer."""
    name: str
    index: int            # seed namespace: seeds are index*1000 + {0 weights, 1 x, 2 mask}
    tokens: int           # T (token slots, padding included)
    d_model: int          # d
    d_ff: int             # H
    n_experts: int        # K residual experts (the shared expert is extra)
    n_blocks: int         # B
    dtype: str            # "f32" or "bf16"
    tau: float = NAN      # NaN = paper default (B-1)/B^2
    alpha_fixed: float = NAN
    beta_fixed: float = NAN
    topk_fixed: int = 0
    prefix_blocks: int = 0
    seq_len: int = 0      # >0: tokens are batch x seq_len with random valid lengths
    min_len: int = 0
    zipf_s: float = 0.0   # >0: router bias -s*ln(j) on residual expert j (1-based)
    clusters: int = 0     # >0: x is a Gaussian mixture with this many clusters

    @property
    def block_width(self) -> int:
        return self.d_ff // self.n_blocks

    def with_(self, **kw) -> "LayerSpec":
        d = dict(self.__dict__)
        d.update(kw)
        return LayerSpec(**d)


# The five workloads the layer is exercised on. Shapes follow the paper's
# backbones (DeiT-S/16 d=384 H=1536 with 197 tokens and eval batch 64;
# BERT max length 128, batch 32) and its block/expert settings (K=6..16,
# B=8..16; Sec. IV-A and the appendix).
CONFIGS = {
    "tiny_f32": LayerSpec("tiny_f32", 0, 256, 64, 256, 4, 4, "f32"),
    "vit_s": LayerSpec("vit_s", 1, 64 * 197, 384, 1536, 8, 8, "bf16"),
    "bert_base": LayerSpec("bert_base", 2, 32 * 128, 768, 3072, 8, 8, "bf16",
                           seq_len=128, min_len=16),
    "vit_b": LayerSpec("vit_b", 3, 64 * 197, 768, 3072, 16, 16, "bf16"),
    "stress": LayerSpec("stress", 4, 65536, 1024, 4096, 32, 16, "bf16",
                        zipf_s=1.2, clusters=4),
}


def spec(name: str, **overrides) -> LayerSpec:
    s = CONFIGS[name]
    return s.with_(**overrides) if overrides else s


@dataclass
class Workload:
    spec: LayerSpec
    w_router: torch.Tensor
    w_up: torch.Tensor
    w_down: torch.Tensor
    router_bias: Optional[torch.Tensor]
    x: torch.Tensor
    mask: Optional[torch.Tensor] = field(default=None)

    @property
    def torch_dtype(self) -> torch.dtype:
        return torch.float32 if self.spec.dtype == "f32" else torch.bfloat16


def _gen(seed: int) -> torch.Generator:
    g = torch.Generator(device="cpu")
    g.manual_seed(seed)
    return g


def make_weights(s: LayerSpec, seed: Optional[int] = None):
    """Upcycled experts: a base FFN (W1 ~ N(0, 1/sqrt(d)), W2 ~ N(0, 1/sqrt(H)),
    the numbers being standard deviations) copied into K+1 experts, each plus
    an independent N(0, 0.05 * std) perturbation; router columns N(0, 0.02).
    Returns (w_router, w_up, w_down, router_bias) in the layer dtype
    (router_bias is float32 or None)."""
    g = _gen(s.index * 1000 if seed is None else seed)
    d, H, K = s.d_model, s.d_ff, s.n_experts
    std1, std2 = 1.0 / math.sqrt(d), 1.0 / math.sqrt(H)
    base_up = torch.randn(H, d, generator=g) * std1
    base_down = torch.randn(d, H, generator=g) * std2
    w_up = base_up.unsqueeze(0) + torch.randn(K + 1, H, d, generator=g) * (0.05 * std1)
    w_down = base_down.unsqueeze(0) + torch.randn(K + 1, d, H, generator=g) * (0.05 * std2)
    w_router = torch.randn(d, K + 1, generator=g) * 0.02
    bias = None
    if s.zipf_s > 0:
        bias = torch.zeros(K + 1, dtype=torch.float32)
        j = torch.arange(1, K + 1, dtype=torch.float64)
        bias[1:] = (-s.zipf_s * torch.log(j)).to(torch.float32)
    dt = torch.float32 if s.dtype == "f32" else torch.bfloat16
    return w_router.to(dt), w_up.to(dt), w_down.to(dt), bias


def make_tokens(s: LayerSpec, w_router: torch.Tensor, T: Optional[int] = None,
                seed: Optional[int] = None):
    """Tokens x ~ N(0, 1) (already layer-normalised activations), plus the
    padding mask for variable-length text batches (valid lengths uniform in
    [min_len, seq_len]; padded rows are filled with NaN so that any use of
    them shows). The load-imbalance workload draws x from a mixture of
    `clusters` Gaussians whose means sit at {-8, -2, 2, 8}/|W_shr| along the
    unit shared-router direction (so the shared logit spans its range) plus
    4/|W_j| along one residual-expert direction j per cluster."""
    T = s.tokens if T is None else T
    g = _gen(s.index * 1000 + 1 if seed is None else seed)
    x = torch.randn(T, s.d_model, generator=g)
    if s.clusters > 0:
        wr = w_router.to(torch.float32)
        w_shr = wr[:, 0]
        shift = torch.tensor([-8.0, -2.0, 2.0, 8.0])[: s.clusters]
        K = s.n_experts
        experts = [1 + (c * max(1, K // s.clusters)) % K for c in range(s.clusters)]
        cid = torch.randint(0, s.clusters, (T,), generator=g)
        means = torch.zeros(s.clusters, s.d_model)
        for c in range(s.clusters):
            wj = wr[:, experts[c]]
            means[c] = (shift[c] / w_shr.norm() ** 2) * w_shr + (4.0 / wj.norm() ** 2) * wj
        x = x + means[cid]
    mask = None
    if s.seq_len > 0:
        gm = _gen(s.index * 1000 + 2 if seed is None else seed + 1)
        nseq = T // s.seq_len
        lens = torch.randint(s.min_len, s.seq_len + 1, (nseq,), generator=gm)
        pos = torch.arange(s.seq_len).unsqueeze(0)
        mask = (pos < lens.unsqueeze(1)).reshape(-1).to(torch.uint8)
        if mask.numel() < T:
            mask = torch.cat([mask, torch.ones(T - mask.numel(), dtype=torch.uint8)])
        x[mask == 0] = float("nan")
    dt = torch.float32 if s.dtype == "f32" else torch.bfloat16
    return x.to(dt), mask


def make_workload(s: LayerSpec, T: Optional[int] = None) -> Workload:
    w_router, w_up, w_down, bias = make_weights(s)
    x, mask = make_tokens(s, w_router, T)
    return Workload(s, w_router, w_up, w_down, bias, x, mask)
