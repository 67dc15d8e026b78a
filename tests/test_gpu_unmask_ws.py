"""The unmask's optional workspace parts change where data is staged, never
the result.  With the full workspace the call uses tensor-core digit planes of
Q_d (the product then writes Y' - K - Q_d L^T), tile images of Q_1, Q_2 and
line-offset copies of the S lists; without room for the copies the gathers
convert positions per round; at the minimum size (the l x m scratch only) the
product runs without planes and the gathers stage rows directly; a workspace
that starts off a 256-byte boundary is carved from its first boundary.  Y_hat
and Y are bit-identical across all four, and Y_hat equals Y' - K - L Q_d -
sum_i S_{i+1} Q_i computed by the oracle from the same Z."""
from types import SimpleNamespace

import numpy as np
import pytest

import oracle as O
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
    from paper_2607_29221_gb300 import mosaic as M
    M.lib()
    yield


def _up(n):
    return (n + 255) // 256 * 256


def _host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint32).copy()


@pytest.mark.parametrize("m,l", [(131, 67), (256, 64)])
def test_unmask_workspace_sizes_agree(m, l):
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    r, t = (1536, 1024, 652), (80, 80)
    gp = M.default_params(d=3, r=list(r), t=[0, *t])
    proto = PR.Protocol(KEY, gp, variant=M.GEMM_AUTO)
    n = 300
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, torch.from_numpy(wl.weights(m, n, std=1.0)).cuda(), 4, ch)
    if layer.L_planes is None:
        pytest.skip("no tensor-core planes on this device")
    mp = layer.init_x(l, 11)
    Xp, s_x, Xpl = layer.mask_input(torch.from_numpy(wl.activations(l, n)).cuda(), mp)
    Z = layer.server(Xp, Xpl)
    full = M.mosaic_workspace_bytes(M.OP_UNMASK, m, 0, l, gp)
    lines = sum(_up(4 * m * ti) for ti in t)
    # (bytes, offset): the misaligned buffer starts 4 bytes past an aligned one.
    sizes = {"full": (full, 0), "no_line_copies": (full - lines, 0), "minimum": (_up(4 * l * m), 0),
             "misaligned": (full + 256, 4)}
    got = {}
    for name, (nb, off) in sizes.items():
        ws = torch.empty(nb + off, dtype=torch.uint8, device="cuda")[off:]
        Y = torch.empty(l, m, dtype=torch.float32, device="cuda")
        Yhat = torch.empty(l, m, dtype=torch.int32, device="cuda")
        M.mosaic_unmask_planes(gp, l, m, Z, Z.stride(0), mp.K, layer.L, layer.L_planes, layer.S_idx,
                               layer.S_val, layer.s_w, s_x, layer.bias, Y, Yhat, m, M.GEMM_AUTO, ws)
        M.mosaic_device_status()
        got[name] = (_host(Yhat), _host(Y))
    for name in ("no_line_copies", "minimum", "misaligned"):
        assert np.array_equal(got[name][0], got["full"][0]), name
        assert np.array_equal(got[name][1], got["full"][1]), name
    # Y_hat by the oracle's unmask (feature-major) from the same Z, K, L and S lists.
    Zh = _host(Z)
    off = np.cumsum((0,) + r)
    Q = [np.ascontiguousarray(Zh[:, m + off[i]:m + off[i + 1]].T) for i in range(3)]
    S_idx, S_val = _host(layer.S_idx), _host(layer.S_val)
    S = {2: (S_idx[:m * t[0]].reshape(m, t[0]), S_val[:m * t[0]].reshape(m, t[0])),
         3: (S_idx[m * t[0]:m * (t[0] + t[1])].reshape(m, t[1]), S_val[m * t[0]:m * (t[0] + t[1])].reshape(m, t[1]))}
    ws_o = SimpleNamespace(L=_host(layer.L).reshape(m, r[2]), S=S)
    ps_o = SimpleNamespace(K=np.ascontiguousarray(_host(mp.K).reshape(l, m).T))
    want = O.unmask(SimpleNamespace(d=3), ws_o, ps_o, np.ascontiguousarray(Zh[:, :m].T), Q)
    assert np.array_equal(got["full"][0].reshape(l, m), want.T)
