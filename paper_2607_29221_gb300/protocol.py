"""Host-side sequencing of the secure linear layer on one GPU.

Allocates device buffers with torch and calls the C ABI in the order of the
protocol boxes (Pi_Sec-Linear, Sec. 4; Pi_Sec-Approx-MatMul, Sec. 3.2).  No
arithmetic happens here: every step is a library call.

  chains = Chains(proto, n_pad)                   # public M_i, N_i products
  layer  = SecureLinear(proto, W, matrix_id, chains, bias)   # Init W
  mp     = layer.init_x(l, pass_id)               # Init X (independent of X)
  Y_tm   = layer.forward(X_tm, mp)                # encode+mask, server, unmask+decode

Token-major layouts throughout: X_tm is l x n, Y_tm is l x m.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import mosaic as M


def _u32(*shape, device="cuda"):
    return torch.empty(*shape, dtype=torch.int32, device=device)


class Protocol:
    """Parameters, key, GEMM variant and a growable workspace."""

    def __init__(self, key_words, params: M.mosaic_params | None = None,
                 variant: int = M.GEMM_AUTO, device="cuda"):
        self.params = params if params is not None else M.default_params()
        self.key = M.make_key(key_words)
        self.variant = variant
        self.device = device
        self._ws = torch.empty(0, dtype=torch.uint8, device=device)

    @property
    def d(self):
        return int(self.params.d)

    @property
    def ranks(self):
        return [int(self.params.r[i]) for i in range(self.d)]

    @property
    def sum_r(self):
        return sum(self.ranks)

    def workspace(self, nbytes: int) -> torch.Tensor:
        if self._ws.numel() < nbytes:
            self._ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=self.device)
        return self._ws

    def sparse_words(self, rows: int) -> int:
        return sum(int(self.params.t[i]) for i in range(1, self.d)) * rows


def pad_width(n: int) -> int:
    p = 32
    while p < n:
        p <<= 1
    return p


class Chains:
    """P (Sr x n_pad), C (n_pad x Sr), C^T for one input width (Init W steps 1-3, 5)."""

    def __init__(self, proto: Protocol, n_pad: int, chain_id: int | None = None):
        self.n_pad = n_pad
        self.chain_id = n_pad if chain_id is None else chain_id
        Sr = proto.sum_r
        self.P = _u32(Sr, n_pad, device=proto.device)
        self.C = _u32(n_pad, Sr, device=proto.device)
        self.CT = _u32(Sr, n_pad, device=proto.device)
        ws = proto.workspace(M.mosaic_workspace_bytes(M.OP_MASK_CHAINS, 0, n_pad, 0, proto.params))
        M.mosaic_mask_chains(proto.params, proto.key, self.chain_id, n_pad, self.P, self.C, self.CT, ws)


@dataclass
class PassMask:
    """Init X output for one pass: U_x^T (l x n_pad) and K^T (l x m)."""
    pass_id: int
    l: int
    Ux: torch.Tensor
    K: torch.Tensor


class SecureLinear:
    """One outsourced linear layer Y = W X + b (Pi_Sec-Linear)."""

    def __init__(self, proto: Protocol, W: torch.Tensor, matrix_id: int, chains: Chains,
                 bias: torch.Tensor | None = None, planes: bool | None = None):
        assert W.dtype == torch.float32 and W.is_cuda and W.dim() == 2
        self.proto = proto
        self.m, self.n = W.shape
        self.n_pad = chains.n_pad
        assert pad_width(self.n) == self.n_pad
        self.matrix_id = matrix_id
        self.chains = chains
        self.bias = bias
        p, dev = proto.params, proto.device
        m, n_pad, Sr = self.m, self.n_pad, proto.sum_r
        self.qmax = M.mosaic_qmax(n_pad, int(p.qbits))
        self.use_planes = (proto.variant in (M.GEMM_TC, M.GEMM_AUTO)) if planes is None else planes
        self.sign_words = _u32(n_pad // 32, device=dev)
        self.s_w = torch.empty(m, dtype=torch.float32, device=dev)
        self.L = _u32(m, proto.ranks[-1], device=dev)
        sw = max(proto.sparse_words(m), 1)
        self.S_idx = _u32(sw, device=dev)
        self.S_val = _u32(sw, device=dev)
        self.Wp = _u32(m + Sr, n_pad, device=dev)
        self.Wp_planes = (torch.empty(4, m + Sr, n_pad, dtype=torch.int16, device=dev)
                          if self.use_planes else None)
        self.J = _u32(m, Sr, device=dev)
        ws = proto.workspace(M.mosaic_workspace_bytes(M.OP_MASK_WEIGHT, m, n_pad, 0, p))
        W = W.contiguous()
        M.mosaic_mask_weight(p, proto.key, matrix_id, W, W.stride(0), m, self.n, n_pad, chains.P,
                             chains.CT, self.sign_words, self.s_w, self.L, self.S_idx, self.S_val,
                             self.Wp, self.Wp_planes, self.J, proto.variant, ws)
        # Stationary tensor-core operands of every pass: [C; J] and L as digit planes.
        self.cj_planes = self.L_planes = None
        if self.use_planes:
            self.cj_planes = torch.empty(M.mosaic_workspace_bytes(M.OP_ACTIVATION_PLANES, m, n_pad, 0, p) // 2,
                                         dtype=torch.int16, device=dev)
            M.mosaic_prepare_activation(p, m, n_pad, chains.C, self.J, self.cj_planes)
            self.L_planes = torch.empty(M.mosaic_workspace_bytes(M.OP_UNMASK_PLANES, m, 0, 0, p) // 2,
                                        dtype=torch.int16, device=dev)
            M.mosaic_prepare_unmask(p, m, self.L, self.L_planes)

    # Init X ---------------------------------------------------------------
    def init_x_workspace_bytes(self, l: int) -> int:
        return M.mosaic_workspace_bytes(M.OP_MASK_ACTIVATION, self.m, self.n_pad, l, self.proto.params)

    def init_x(self, l: int, pass_id: int, pass_dev=None, out: PassMask | None = None,
               phase: int = M.INITX_ALL, ws=None) -> PassMask:
        """Init X for one pass.  pass_dev (a device int64 word, optional) is
        added to pass_id on the device, so that a captured CUDA graph draws a
        fresh pass on every replay; `out` reuses preallocated U_x / K buffers.
        `phase` INITX_DRAWS / INITX_COMPOSE runs one part (the second call
        with the same arguments and the same `ws`, left untouched between)."""
        p, dev = self.proto.params, self.proto.device
        Ux = _u32(l, self.n_pad, device=dev) if out is None else out.Ux
        K = _u32(l, self.m, device=dev) if out is None else out.K
        if ws is None:
            ws = self.proto.workspace(self.init_x_workspace_bytes(l))
        if phase == M.INITX_ALL:
            M.mosaic_mask_activation_ex(p, self.proto.key, pass_id, pass_dev, self.m, self.n_pad, l,
                                        self.chains.C, self.J, self.cj_planes, Ux, K, self.proto.variant, ws)
        else:
            M.mosaic_mask_activation_phase(p, self.proto.key, pass_id, pass_dev, self.m, self.n_pad, l,
                                           self.chains.C, self.J, self.cj_planes, Ux, K, self.proto.variant, ws,
                                           phase)
        return PassMask(pass_id, l, Ux, K) if out is None else out

    # Online ---------------------------------------------------------------
    def mask_input(self, X_tm: torch.Tensor, mp: PassMask, Xp=None, s_x=None, Xplanes=None):
        """Client: X' = encode(R X) + U_x (token-major), optionally its digit planes."""
        l = X_tm.shape[0]
        dev = self.proto.device
        Xp = _u32(l, self.n_pad, device=dev) if Xp is None else Xp
        s_x = torch.empty(l, dtype=torch.float32, device=dev) if s_x is None else s_x
        planes = self.use_planes and l > M.STREAMW_MAX_M
        if planes and Xplanes is None:
            Xplanes = torch.empty(4, l, self.n_pad, dtype=torch.int16, device=dev)
        M.mosaic_encode(X_tm, X_tm.stride(0), l, self.n, self.n_pad, self.qmax, 1, self.sign_words,
                        mp.Ux, self.n_pad, Xp, self.n_pad, s_x, Xplanes if planes else None)
        return Xp, s_x, Xplanes

    def server(self, Xp, Xplanes, Z=None):
        """Untrusted accelerator: Z = X'_tm [W'; P]^T = [Y' | Q_1 .. Q_d] (token-major).

        Up to STREAMW_MAX_M tokens the product streams the uint32 W' (4 bytes an
        element: CUDA cores up to SKINNY_MAX_M tokens, tensor cores with an
        on-chip digit split above); more tokens run on the tensor cores from the
        digit planes of W' and X'."""
        l = Xp.shape[0]
        N = self.m + self.proto.sum_r
        Z = _u32(l, N, device=self.proto.device) if Z is None else Z
        if self.use_planes and l > M.STREAMW_MAX_M:
            M.mosaic_ring_gemm_planes(Xplanes, self.n_pad, l * self.n_pad, self.Wp_planes,
                                      self.n_pad, N * self.n_pad, Z, N, l, N, self.n_pad,
                                      M.GEMM_TC)
        else:
            ws = self.proto.workspace(M.mosaic_workspace_bytes(M.OP_RING_GEMM, l, N, self.n_pad))
            M.mosaic_ring_gemm(Xp, self.n_pad, self.Wp, self.n_pad, Z, N, l, N, self.n_pad,
                               self.proto.variant, ws)
        return Z

    def unmask(self, Z, mp: PassMask, s_x, Y=None, Yhat=None):
        l = Z.shape[0]
        p = self.proto.params
        Y = torch.empty(l, self.m, dtype=torch.float32, device=self.proto.device) if Y is None else Y
        ws = self.proto.workspace(M.mosaic_workspace_bytes(M.OP_UNMASK, self.m, 0, l, p))
        if self.L_planes is not None:
            M.mosaic_unmask_planes(p, l, self.m, Z, Z.stride(0), mp.K, self.L, self.L_planes, self.S_idx,
                                   self.S_val, self.s_w, s_x, self.bias, Y, Yhat, self.m, self.proto.variant, ws)
        else:
            M.mosaic_unmask(p, l, self.m, Z, Z.stride(0), mp.K, self.L, self.S_idx, self.S_val,
                            self.s_w, s_x, self.bias, Y, Yhat, self.m, self.proto.variant, ws)
        return Y

    # Integrity (Init W step 4, Online step 4) ---------------------------
    def freivalds_setup(self, k: int = 4):
        """Draws k check vectors a (k x m) and keeps Ychk = a W' (k x n_pad)."""
        dev = self.proto.device
        self.check_k = k
        self.check_a = _u32(k, self.m, device=dev)
        self.check_Y = _u32(k, self.n_pad, device=dev)
        M.mosaic_freivalds_setup(self.proto.params, self.proto.key, self.matrix_id, k, self.Wp,
                                 self.n_pad, self.m, self.n_pad, self.check_a, self.check_Y)

    def freivalds_check(self, Z, Xp, bad=None, n_bad=None):
        """Per-token check a^T Y' == Ychk X' on the device; returns (bad, n_bad)
        device tensors (bad[j] = failing vectors of token j, n_bad = failing
        tokens).  Read n_bad after a synchronise; nonzero means: abort."""
        l = Z.shape[0]
        dev = self.proto.device
        bad = _u32(l, device=dev) if bad is None else bad
        if n_bad is None:
            n_bad = torch.zeros(1, dtype=torch.int32, device=dev)
        ws = self.proto.workspace(M.mosaic_workspace_bytes(M.OP_FREIVALDS_CHECK, self.check_k, 0, l))
        M.mosaic_freivalds_check(self.check_k, self.check_a, self.check_Y, self.m, self.n_pad, l, Z,
                                 Z.stride(0), Xp, Xp.stride(0), bad, n_bad, ws)
        return bad, n_bad

    def forward(self, X_tm: torch.Tensor, mp: PassMask, Yhat=None):
        Xp, s_x, Xplanes = self.mask_input(X_tm, mp)
        Z = self.server(Xp, Xplanes)
        return self.unmask(Z, mp, s_x, Yhat=Yhat)
