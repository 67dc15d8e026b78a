"""Freivalds integrity check (Sec. 3.2 box, Init W step 4 and Online step 4;
appendix "Computational integrity") through the C ABI against the oracle:
the check vectors and a^T W' bit-exact, honest answers accepted, a corrupted
entry of Y' flagged on exactly its token."""
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
    yield


def _host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint32)


@pytest.mark.parametrize("m,n,l,k", [(128, 256, 64, 4), (131, 300, 9, 3), (200, 256, 1, 16),
                                     (1000, 512, 300, 8)])
def test_freivalds_matches_oracle_and_detects(m, n, l, k):
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    op = O.Params(d=3, r=(96, 64, 40), t=(8, 4))
    gp = M.default_params(d=3, r=[96, 64, 40], t=[0, 8, 4])
    proto = PR.Protocol(KEY, gp, variant=M.GEMM_AUTO)
    W = wl.weights(m, n, std=1.0)
    X = wl.activations(l, n)
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, torch.from_numpy(W).cuda(), 7, ch)
    layer.freivalds_setup(k)
    mp = layer.init_x(l, 11)
    Xp, s_x, Xpl = layer.mask_input(torch.from_numpy(X).cuda(), mp)
    Z = layer.server(Xp, Xpl)
    ref = O.secure_linear(KEY, op, W, X.T.copy(), matrix_id=7, pass_id=11)
    a, Yc = O.freivalds_setup(KEY, op, ref["ws"], 7, k)
    assert np.array_equal(_host(layer.check_a), a)
    assert np.array_equal(_host(layer.check_Y), Yc)
    bad, n_bad = layer.freivalds_check(Z, Xp)
    M.mosaic_device_status()
    assert _host(n_bad)[0] == 0 and not np.any(_host(bad))
    # an odd error in Y'[j][i] is caught by every vector (a_v[i] != 0)
    j, i = l // 2, m // 3
    Zc = Z.clone()
    Zc[j, i] += 977
    bad, n_bad = layer.freivalds_check(Zc, Xp)
    got = _host(bad)
    want = O.freivalds_check(a, Yc, _host(Zc)[:, :m].T.copy(), ref["X_masked"])
    assert np.array_equal(got, want)
    assert got[j] == np.count_nonzero(a[:, i]) and np.count_nonzero(got) == 1
    assert _host(n_bad)[0] == 1
    # the Q columns of Z are not covered by the check
    if l > 1:
        Zq = Z.clone()
        Zq[0, m] += 1
        bad, n_bad = layer.freivalds_check(Zq, Xp)
        assert _host(n_bad)[0] == 0
