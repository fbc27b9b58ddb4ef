"""Seeded synthetic inputs for the pruned-pool decode MoE layer.

This module only draws random tensors with the shapes and value distributions
of the workloads; it holds none of the layer's arithmetic, so both the CUDA path
and the CPU oracle can be fed from it.  All draws use a torch generator seeded
explicitly (on the CPU, or on a CUDA device for the multi-GB cases) so a run is
reproducible on one machine.

Distributions (Qwen-class decode layer):
  * expert weights W_gu [E, 2I, H], W_down [E, H, I]: bf16 ~ N(0, 0.02)
  * router weight Wr [E, H]: fp32 ~ N(0, 0.02)
  * hidden states x [B, H]: bf16 ~ N(0, 1)
  * retained set K': importance ~ U[0, 1) per expert, keep the m' largest
    (ties to the lowest id) -- a stand-in for the calibration-based ranking
    of Sec. 2.3 / Sec. 3.1, which needs a trained model.
  * popularity skew: per-layer Zipf(s) rank bias, realised through one extra
    exactly-representable router term (x[:, H-1] = 1, Wr[:, H-1] = bias).
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

WEIGHT_STD = 0.02
ROUTER_STD = 0.02


@dataclass(frozen=True)
class LayerShape:
    hidden: int        # H
    num_experts: int   # E
    inter: int         # I
    top_k: int         # k

    @property
    def expert_bytes(self) -> int:
        """bf16 bytes of one expert: [2I, H] gate/up plus [H, I] down."""
        return 2 * (2 * self.inter * self.hidden + self.hidden * self.inter)


TINY = LayerShape(hidden=256, num_experts=16, inter=128, top_k=2)
QWEN = LayerShape(hidden=2048, num_experts=128, inter=768, top_k=8)
# Qwen3.6-shaped layer: 256 experts, top-8 (Sec. 2.1).  The expert size is
# derived, not printed: a 60 GiB bf16 pool over 40 layers of 256 experts is
# about 3.1 M parameters per expert, i.e. I = 512 at H = 2048.
QWEN36 = LayerShape(hidden=2048, num_experts=256, inter=512, top_k=8)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def expert_weights(shape: LayerShape, seed: int, device="cpu"):
    """(W_gu bf16 [E, 2I, H], W_down bf16 [E, H, I]) ~ N(0, 0.02)."""
    g = _gen(seed, device)
    E, H, I = shape.num_experts, shape.hidden, shape.inter
    w_gu = torch.empty((E, 2 * I, H), dtype=torch.bfloat16, device=device)
    w_d = torch.empty((E, H, I), dtype=torch.bfloat16, device=device)
    # draw expert by expert to bound the fp32 temporaries
    for e in range(E):
        w_gu[e] = (torch.randn((2 * I, H), generator=g, device=device) * WEIGHT_STD).to(torch.bfloat16)
        w_d[e] = (torch.randn((H, I), generator=g, device=device) * WEIGHT_STD).to(torch.bfloat16)
    return w_gu, w_d


def router_weight(shape: LayerShape, seed: int, device="cpu") -> torch.Tensor:
    """fp32 [E, H] ~ N(0, 0.02)."""
    g = _gen(seed, device)
    return torch.randn((shape.num_experts, shape.hidden), generator=g, device=device) * ROUTER_STD


def hidden_states(batch: int, shape: LayerShape, seed: int, device="cpu") -> torch.Tensor:
    """bf16 [B, H] ~ N(0, 1)."""
    g = _gen(seed, device)
    return torch.randn((batch, shape.hidden), generator=g, device=device).to(torch.bfloat16)


def shared_expert(hidden: int, inter_shared: int, seed: int, device="cpu"):
    """Shared expert of one layer: (gate row fp32 [H] ~ N(0, 0.05), gate/up bf16
    [2Is, H] and down bf16 [H, Is] ~ N(0, 0.02))."""
    one = LayerShape(hidden=hidden, num_experts=1, inter=inter_shared, top_k=1)
    gu, dn = expert_weights(one, seed, device=device)
    g = _gen(seed + 17, device)
    w_sg = (torch.randn((hidden,), generator=g, device=device) * 0.05).to(torch.float32)
    return w_sg, gu[0].contiguous(), dn[0].contiguous()


def retained_set(num_experts: int, n_retained: int, seed: int, shuffle: bool = False) -> torch.Tensor:
    """int32 ids of the m' experts with the largest U[0,1) importance score.

    Sorted ascending unless `shuffle` (order is irrelevant to the layer).
    """
    g = _gen(seed, "cpu")
    score = torch.rand((num_experts,), generator=g, dtype=torch.float64)
    # stable sort on -score keeps the lowest id first among equal scores
    order = torch.sort(-score, stable=True).indices[:n_retained]
    ids = torch.sort(order).values.to(torch.int32)
    if shuffle:
        ids = ids[torch.randperm(n_retained, generator=g)]
    return ids.contiguous()


def zipf_rank_bias(num_experts: int, s: float, seed: int) -> torch.Tensor:
    """fp32 [E]: bias_e = -s * ln(rank_e), rank a seeded permutation of 1..E.

    Adding it to the logits skews routing toward low-rank experts like a
    Zipf(s) popularity law (the pmf's normaliser cancels in top-k and softmax).
    """
    g = _gen(seed, "cpu")
    rank = torch.randperm(num_experts, generator=g).to(torch.float64) + 1.0
    return (-s * torch.log(rank)).to(torch.float32)


def apply_popularity_bias(hidden: torch.Tensor, router_w: torch.Tensor, bias: torch.Tensor):
    """Realise a per-expert logit bias with the existing inputs: x[:, H-1] = 1 and
    Wr[:, H-1] = bias, so the bias enters the router dot product as one exact term."""
    hidden = hidden.clone()
    router_w = router_w.clone()
    hidden[:, -1] = 1.0
    router_w[:, -1] = bias.to(router_w.device, router_w.dtype)
    return hidden, router_w


def bf16_bits(t: torch.Tensor):
    """numpy uint16 view of a bf16 tensor's bit patterns (host copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view("uint16")
