"""One masked decoder layer (the secure forward pass of Sec. 4.1, one layer).

Every linear layer is an outsourced Pi_Sec-Linear call (``protocol.SecureLinear``):
the fused QKV projection, the attention output projection, the fused gate+up
projection and the down projection (the four per-layer calls of Sec. 4.1).
The non-linear parts stay on the trusted side in plain fp32 on the device, as
the paper keeps them on the client (attention is local, Sec. 3.2 "Local
attention computation"): RMSNorm, causal grouped-query attention with a
softmax, SiLU(gate) * up, and the residual adds.  Rotary position embeddings
are not described by the paper and are left out.

Weights are seeded random N(0, 0.02) (the paper's checkpoints are not
available); RMSNorm weights are 1.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import protocol as PR
from . import workloads as wl


@dataclass(frozen=True)
class LayerShape:
    hidden: int = 8192
    n_heads: int = 64
    n_kv: int = 8
    head_dim: int = 128
    ffn: int = 28672
    eps: float = 1e-5

    @property
    def qkv(self) -> int:
        return (self.n_heads + 2 * self.n_kv) * self.head_dim


def rmsnorm(x: torch.Tensor, eps: float) -> torch.Tensor:
    return x * torch.rsqrt(x.pow(2).mean(dim=-1, keepdim=True) + eps)


def attention(qkv: torch.Tensor, s: LayerShape) -> torch.Tensor:
    """Causal grouped-query attention in fp32; qkv is l x (H + 2 KV) * d."""
    l = qkv.shape[0]
    q = qkv[:, : s.n_heads * s.head_dim].view(l, s.n_heads, s.head_dim).transpose(0, 1)
    k = qkv[:, s.n_heads * s.head_dim: (s.n_heads + s.n_kv) * s.head_dim].view(l, s.n_kv, s.head_dim)
    v = qkv[:, (s.n_heads + s.n_kv) * s.head_dim:].view(l, s.n_kv, s.head_dim)
    rep = s.n_heads // s.n_kv
    k = k.transpose(0, 1).repeat_interleave(rep, dim=0)
    v = v.transpose(0, 1).repeat_interleave(rep, dim=0)
    scores = torch.matmul(q, k.transpose(1, 2)) * (1.0 / float(s.head_dim) ** 0.5)
    mask = torch.ones(l, l, dtype=torch.bool, device=qkv.device).triu(1)
    scores = scores.masked_fill(mask, float("-inf"))
    out = torch.matmul(torch.softmax(scores, dim=-1), v)            # H x l x d
    return out.transpose(0, 1).reshape(l, s.n_heads * s.head_dim)


class LayerWeights:
    """Seeded float weights of one layer (token-major convention: W is out x in)."""

    def __init__(self, s: LayerShape, seed: int = 11, device="cuda"):
        self.s = s
        self.Wqkv = torch.from_numpy(wl.weights(s.qkv, s.hidden, seed=seed)).to(device)
        self.Wo = torch.from_numpy(wl.weights(s.hidden, s.n_heads * s.head_dim, seed=seed + 1)).to(device)
        self.Wgu = torch.from_numpy(wl.weights(2 * s.ffn, s.hidden, seed=seed + 2)).to(device)
        self.Wdown = torch.from_numpy(wl.weights(s.hidden, s.ffn, seed=seed + 3)).to(device)


def reference_forward(w: LayerWeights, x: torch.Tensor) -> torch.Tensor:
    """The same layer with plain fp32 matrix products (no masking, no quantisation)."""
    s = w.s
    h = rmsnorm(x, s.eps)
    a = attention(h @ w.Wqkv.T, s)
    x = x + a @ w.Wo.T
    gu = rmsnorm(x, s.eps) @ w.Wgu.T
    x = x + (torch.nn.functional.silu(gu[:, : s.ffn]) * gu[:, s.ffn:]) @ w.Wdown.T
    return x


class SecureDecoderLayer:
    """Init W of the four linear layers at construction; forward() runs one pass."""

    def __init__(self, proto: PR.Protocol, w: LayerWeights, layer_id: int = 0):
        s = w.s
        self.s, self.proto = s, proto
        chains = {}

        def chain(n):
            n_pad = PR.pad_width(n)
            if n_pad not in chains:
                chains[n_pad] = PR.Chains(proto, n_pad)
            return chains[n_pad]

        base = 16 * layer_id
        self.qkv = PR.SecureLinear(proto, w.Wqkv, base + 1, chain(s.hidden))
        self.o = PR.SecureLinear(proto, w.Wo, base + 2, chain(s.n_heads * s.head_dim))
        self.gu = PR.SecureLinear(proto, w.Wgu, base + 3, chain(s.hidden))
        self.down = PR.SecureLinear(proto, w.Wdown, base + 4, chain(s.ffn))
        self.chains = chains
        self._pass = 0

    def linears(self):
        return [self.qkv, self.o, self.gu, self.down]

    def init_x(self, l: int):
        """Init X of all four calls of one pass (independent of the activations)."""
        self._pass += 1
        return [lin.init_x(l, 1_000_000 * (i + 1) + self._pass) for i, lin in enumerate(self.linears())]

    def forward(self, x: torch.Tensor, masks=None) -> torch.Tensor:
        s = self.s
        masks = masks if masks is not None else self.init_x(x.shape[0])
        h = rmsnorm(x, s.eps)
        a = attention(self.qkv.forward(h.contiguous(), masks[0]), s)
        x = x + self.o.forward(a.contiguous(), masks[1])
        gu = self.gu.forward(rmsnorm(x, s.eps).contiguous(), masks[2])
        act = torch.nn.functional.silu(gu[:, : s.ffn]) * gu[:, s.ffn:]
        return x + self.down.forward(act.contiguous(), masks[3])
