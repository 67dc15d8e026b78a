"""One masked decoder layer (the secure forward pass of Sec. 4.1, one layer).

Every linear layer is an outsourced Pi_Sec-Linear call (``protocol.SecureLinear``):
the fused QKV projection, the attention output projection, the fused gate+up
projection and the down projection (the four per-layer calls of Sec. 4.1).
The non-linear parts stay on the trusted side in plain fp32 on the device, as
the paper keeps them on the client (attention is local, Sec. 3.2 "Local
attention computation"): RMSNorm and SiLU(gate) * up (one-pass kernels of this
library), causal grouped-query attention with a softmax (torch's fused
scaled-dot-product attention in fp32, causal), and the residual adds.  Rotary position embeddings are not described by
the paper and are left out.

Weights are seeded random N(0, 0.02) (the paper's checkpoints are not
available); RMSNorm weights are 1.

A pass can run with preallocated buffers (``alloc``) and a device pass
counter, so that the whole layer is captured once as a CUDA graph whose every
replay draws fresh masks.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch
import torch.nn.functional as F

from . import mosaic as M
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


def rmsnorm(x: torch.Tensor, eps: float, out: torch.Tensor | None = None) -> torch.Tensor:
    """x / sqrt(mean(x^2) + eps) per row, one pass (mosaic_rmsnorm)."""
    y = torch.empty_like(x) if out is None else out
    M.mosaic_rmsnorm(x, x.stride(0), x.shape[0], x.shape[1], eps, y, y.stride(0))
    return y


def swiglu(gu: torch.Tensor, ffn: int, out: torch.Tensor | None = None) -> torch.Tensor:
    """SiLU(gate) * up with gate = columns [0, ffn), up = [ffn, 2 ffn), one pass (mosaic_swiglu)."""
    act = torch.empty(gu.shape[0], ffn, dtype=gu.dtype, device=gu.device) if out is None else out
    M.mosaic_swiglu(gu, gu.stride(0), gu.shape[0], ffn, act, act.stride(0))
    return act


def attention(qkv: torch.Tensor, s: LayerShape) -> torch.Tensor:
    """Causal grouped-query attention in fp32; qkv is l x (H + 2 KV) * d,
    the output l x H d (token-major)."""
    l = qkv.shape[0]
    H, KV, d = s.n_heads, s.n_kv, s.head_dim
    q = qkv[:, : H * d].view(l, H, d).transpose(0, 1)
    k = qkv[:, H * d: (H + KV) * d].view(l, KV, d).transpose(0, 1).repeat_interleave(H // KV, dim=0)
    v = qkv[:, (H + KV) * d:].view(l, KV, d).transpose(0, 1).repeat_interleave(H // KV, dim=0)
    out = F.scaled_dot_product_attention(q.unsqueeze(0), k.unsqueeze(0), v.unsqueeze(0), is_causal=True)
    return out[0].transpose(0, 1).reshape(l, H * d)


class LayerWeights:
    """Seeded float weights of one layer (token-major convention: W is out x in)."""

    def __init__(self, s: LayerShape, seed: int = 11, device="cuda"):
        self.s = s
        self.Wqkv = torch.from_numpy(wl.weights(s.qkv, s.hidden, seed=seed)).to(device)
        self.Wo = torch.from_numpy(wl.weights(s.hidden, s.n_heads * s.head_dim, seed=seed + 1)).to(device)
        self.Wgu = torch.from_numpy(wl.weights(2 * s.ffn, s.hidden, seed=seed + 2)).to(device)
        self.Wdown = torch.from_numpy(wl.weights(s.hidden, s.ffn, seed=seed + 3)).to(device)


def _no_mark(name: str) -> None:
    return None


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
        self.bufs = None

    def linears(self):
        return [self.qkv, self.o, self.gu, self.down]

    def alloc(self, l: int) -> None:
        """Preallocates every per-pass buffer of the four calls for l tokens,
        the Init X workspaces of the four calls (their draws stay there until
        the compositions run, see forward_pass) and the stream of the draws."""
        dev = self.proto.device
        Sr = self.proto.sum_r
        self.initx_ws = [torch.empty(max(lin.init_x_workspace_bytes(l), 256), dtype=torch.uint8, device=dev)
                         for lin in self.linears()]
        self.draw_stream = torch.cuda.Stream(device=dev)
        self.bufs = []
        for lin in self.linears():
            planes = lin.use_planes and l > M.STREAMW_MAX_M
            self.bufs.append(dict(
                Xp=torch.empty(l, lin.n_pad, dtype=torch.int32, device=dev),
                s_x=torch.empty(l, dtype=torch.float32, device=dev),
                Xpl=torch.empty(4, l, lin.n_pad, dtype=torch.int16, device=dev) if planes else None,
                Z=torch.empty(l, lin.m + Sr, dtype=torch.int32, device=dev),
                Y=torch.empty(l, lin.m, dtype=torch.float32, device=dev)))

    def init_x(self, l: int, pass_base: int | None = None, pass_dev=None, out=None):
        """Init X of all four calls of one pass (independent of the activations).
        Call i draws pass pass_base + 1_000_000 i (+ *pass_dev on the device);
        without pass_base a host counter advances per call."""
        if pass_base is None:
            self._pass += 1
            pass_base = self._pass
        outs = out if out is not None else [None] * 4
        return [lin.init_x(l, 1_000_000 * (i + 1) + pass_base, pass_dev=pass_dev, out=outs[i])
                for i, lin in enumerate(self.linears())]

    def _linear(self, i: int, x: torch.Tensor, mp, mark, compose=None) -> torch.Tensor:
        lin = self.linears()[i]
        b = self.bufs[i] if self.bufs is not None else {}
        if compose is not None:
            mark("init_x")
            compose(i)
        mark("encode")
        Xp, s_x, Xpl = lin.mask_input(x, mp, b.get("Xp"), b.get("s_x"), b.get("Xpl"))
        mark("server")
        Z = lin.server(Xp, Xpl, b.get("Z"))
        mark("unmask")
        Y = lin.unmask(Z, mp, s_x, b.get("Y"))
        mark("glue")
        return Y

    def forward(self, x: torch.Tensor, masks=None, mark=None, compose=None) -> torch.Tensor:
        """One pass over l tokens (x: l x hidden fp32).  `mark(part)`, if given,
        is called where each part of the pass begins (init_x, encode, server,
        unmask, glue), e.g. to record CUDA events.  With `compose`, call i's
        Init X composition runs (compose(i)) right before its encode."""
        s = self.s
        mark = mark or _no_mark
        if masks is None:
            mark("init_x")
            masks = self.init_x(x.shape[0])
        mark("glue")
        h = rmsnorm(x, s.eps)
        a = attention(self._linear(0, h, masks[0], mark, compose), s)
        x = x + self._linear(1, a, masks[1], mark, compose)
        gu = self._linear(2, rmsnorm(x, s.eps), masks[2], mark, compose)
        act = swiglu(gu, s.ffn)
        return x + self._linear(3, act, masks[3], mark, compose)

    def forward_pass(self, x: torch.Tensor, pass_base: int, masks, pass_dev=None, mark=None,
                     after=None) -> torch.Tensor:
        """Init X and the layer of one pass, with the Init X draws (ALU-bound
        ChaCha20 in blocks of 128 threads and 9 KB of shared memory) on a side
        stream: call 0's draws at the start of the pass, the other three
        calls' draws once call 0's composition is done, beside its encode,
        server product, unmask and the attention.  Call 0's composition
        (product and gathers, which need the SM's shared memory) runs first,
        before the layer waits for `after`; the others on the main stream
        right before their call's encode.  Call 1's composition waits for all
        three draws, so no draw runs beside an Init X gather.  Same pass ids
        and results as init_x + forward (call i draws pass pass_base +
        1_000_000 (i + 1), plus *pass_dev); `masks` are the four calls'
        preallocated U_x / K buffers; `after`, a stream that the layer (not
        the draws) waits for first, e.g. the copy of x.  Needs alloc."""
        l = x.shape[0]
        main = torch.cuda.current_stream()
        side = self.draw_stream
        side.wait_stream(main)
        lins = self.linears()
        pids = [1_000_000 * (i + 1) + pass_base for i in range(4)]

        def draw(i):
            lins[i].init_x(l, pids[i], pass_dev=pass_dev, out=masks[i], phase=M.INITX_DRAWS, ws=self.initx_ws[i])

        first, rest = torch.cuda.Event(), torch.cuda.Event()
        with torch.cuda.stream(side):
            draw(0)
            first.record(side)
        # Call 0's composition does not depend on x either: it runs before
        # the layer waits for `after`.
        (mark or _no_mark)("init_x")
        main.wait_event(first)
        lins[0].init_x(l, pids[0], pass_dev=pass_dev, out=masks[0], phase=M.INITX_COMPOSE, ws=self.initx_ws[0])
        side.wait_stream(main)
        with torch.cuda.stream(side):
            for j in (1, 2, 3):
                draw(j)
            rest.record(side)
        if after is not None:
            main.wait_stream(after)

        def compose(i):
            if i == 0:
                return
            main.wait_event(rest)
            lins[i].init_x(l, pids[i], pass_dev=pass_dev, out=masks[i], phase=M.INITX_COMPOSE,
                           ws=self.initx_ws[i])

        return self.forward(x, masks, mark=mark, compose=compose)
