"""Row sharding of one secure linear call (the paper's model-matrix sharding,
Sec. 5.2 "Model sharding"): the rows of W' with their L, S, J rows, s_w and
bias split across devices, X' and the public-chain answer Q computed once.
Running the shards one after the other on one device, the concatenated Y'
and decoded Y equal the unsharded call's, bit for bit."""
import numpy as np
import pytest

from paper_2607_29221_gb300 import workloads as wl

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

KEY = wl.mask_key()


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_29221_gb300 import build
    build.build()
    yield


@pytest.mark.parametrize("l", [3, 64])
def test_row_shards_concatenate_to_the_full_call(l):
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    p = M.default_params(d=3, r=[96, 64, 40], t=[0, 8, 4])
    proto = PR.Protocol(KEY, p, variant=M.GEMM_AUTO)
    m, n = 300, 256
    ch = PR.Chains(proto, PR.pad_width(n))
    W = torch.from_numpy(wl.weights(m, n, std=1.0)).cuda()
    b = torch.from_numpy(wl.bias(m)).cuda()
    layer = PR.SecureLinear(proto, W, 8, ch, bias=b)
    mp = layer.init_x(l, 21)
    Xp, s_x, Xpl = layer.mask_input(torch.from_numpy(wl.activations(l, n)).cuda(), mp)
    Z = layer.server(Xp, Xpl)
    Yhat = torch.empty(l, m, dtype=torch.int32, device="cuda")
    Y = layer.unmask(Z, mp, s_x, Yhat=Yhat)
    Sr, n_pad = proto.sum_r, layer.n_pad
    t = [8, 4]
    Q = Z[:, m:].contiguous()
    for lo, hi in [(0, 100), (100, 220), (220, 300)]:
        ms = hi - lo
        Wp_s = torch.cat([layer.Wp[lo:hi], layer.Wp[m:]]).contiguous()      # [W'_shard; P]
        Z_s = torch.empty(l, ms + Sr, dtype=torch.int32, device="cuda")
        ws = proto.workspace(M.mosaic_workspace_bytes(M.OP_RING_GEMM, l, ms + Sr, n_pad))
        M.mosaic_ring_gemm(Xp, n_pad, Wp_s, n_pad, Z_s, ms + Sr, l, ms + Sr, n_pad, M.GEMM_AUTO, ws)
        assert torch.equal(Z_s[:, :ms], Z[:, lo:hi]) and torch.equal(Z_s[:, ms:], Q)
        off, idx, val = 0, [], []
        for ti in t:
            idx.append(layer.S_idx[off + lo * ti: off + hi * ti])
            val.append(layer.S_val[off + lo * ti: off + hi * ti])
            off += m * ti
        S_idx, S_val = torch.cat(idx).contiguous(), torch.cat(val).contiguous()
        K_s = mp.K[:, lo:hi].contiguous()
        Y_s = torch.empty(l, ms, dtype=torch.float32, device="cuda")
        Yh_s = torch.empty(l, ms, dtype=torch.int32, device="cuda")
        ws = proto.workspace(M.mosaic_workspace_bytes(M.OP_UNMASK, ms, 0, l, p))
        M.mosaic_unmask(p, l, ms, Z_s, ms + Sr, K_s, layer.L[lo:hi].contiguous(), S_idx, S_val,
                        layer.s_w[lo:hi].contiguous(), s_x, b[lo:hi].contiguous(), Y_s, Yh_s, ms,
                        M.GEMM_AUTO, ws)
        M.mosaic_device_status()
        assert torch.equal(Yh_s, Yhat[:, lo:hi])
        assert torch.equal(Y_s, Y[:, lo:hi])
