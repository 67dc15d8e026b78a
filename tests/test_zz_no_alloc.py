"""mosaic_unmask_noalloc: the unmask for callers that cannot allocate device
memory (a plugin whose host framework owns all device memory, a runtime with a
fixed memory budget, a serving loop that must not enter the allocator).  Its
scratch is a fixed array inside the library instead of a caller workspace.

Checked through the C ABI against mosaic_unmask (the entry point with a
workspace) on two calls in a row: Y_hat bit-exact, decoded Y within
1e-6 x (|Y_hat s_w s_x| + |b|), the tolerance of the other parity tests.
This file is collected last on purpose."""
import numpy as np
import pytest

from paper_2607_29221_gb300 import workloads as wl

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_29221_gb300 import build
    build.build()
    yield


def _pass(layer, X_tm, pass_id):
    mp = layer.init_x(X_tm.shape[0], pass_id)
    Xp, s_x, Xpl = layer.mask_input(X_tm, mp)
    Z = layer.server(Xp, Xpl)
    return mp, s_x, Z


@pytest.mark.parametrize("variant_name,m,n,l", [("imad", 320, 500, 48), ("tc", 320, 500, 48),
                                                ("tc", 4096, 256, 1024)])
def test_noalloc_unmask_matches_workspace_unmask_twice(variant_name, m, n, l):
    """Small shapes on both product variants, and l * m = 2^22 exactly: the l x m
    scratch fills the whole array and every optional part is skipped."""
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    variant = {"imad": M.GEMM_IMAD, "tc": M.GEMM_TC}[variant_name]
    if variant == M.GEMM_TC and not M.mosaic_gemm_variant_available(M.GEMM_TC):
        pytest.skip("tensor-core variant not available")
    key = wl.mask_key()
    proto = PR.Protocol(key, M.default_params(), variant=variant)
    ch = PR.Chains(proto, PR.pad_width(n))
    W = torch.from_numpy(wl.weights(m, n)).cuda()
    b = torch.from_numpy(wl.bias(m)).cuda()
    layer = PR.SecureLinear(proto, W, 9, ch, bias=b)
    runs = []
    for pass_id, seed in ((101, 1), (102, 7)):
        X = torch.from_numpy(wl.activations(l, n, seed=seed)).cuda()
        mp, s_x, Z = _pass(layer, X, pass_id)
        Yhat_ref = torch.empty(l, m, dtype=torch.int32, device="cuda")
        Y_ref = layer.unmask(Z, mp, s_x, Yhat=Yhat_ref)
        runs.append((mp, s_x, Z, Y_ref, Yhat_ref))
    torch.cuda.synchronize()
    # Two no-alloc calls in a row, the second reusing the scratch the first left behind.
    outs = []
    for mp, s_x, Z, _, _ in runs:
        Y = torch.full((l, m), float("nan"), dtype=torch.float32, device="cuda")
        Yhat = torch.zeros(l, m, dtype=torch.int32, device="cuda")
        M.mosaic_unmask_noalloc(proto.params, l, m, Z, Z.stride(0), mp.K, layer.L, layer.S_idx,
                                layer.S_val, layer.s_w, s_x, b, Y, Yhat, m, variant)
        outs.append((Y, Yhat))
    M.mosaic_device_status()
    for (mp, s_x, Z, Y_ref, Yhat_ref), (Y, Yhat) in zip(runs, outs):
        yh_ref = Yhat_ref.cpu().numpy().view(np.uint32)
        assert np.array_equal(Yhat.cpu().numpy().view(np.uint32), yh_ref)
        mag = (np.abs(yh_ref.view(np.int32).astype(np.float64)
                      * layer.s_w.cpu().numpy().astype(np.float64)[None, :]
                      * s_x.cpu().numpy().astype(np.float64)[:, None])
               + np.abs(b.cpu().numpy().astype(np.float64))[None, :])
        err = np.abs(Y.cpu().numpy().astype(np.float64) - Y_ref.cpu().numpy().astype(np.float64))
        assert np.all(err <= 1e-6 * mag)


def test_noalloc_unmask_refuses_oversized_request():
    from paper_2607_29221_gb300 import mosaic as M
    p = M.default_params()
    fake = 1 << 40      # never dereferenced: the size check comes first
    st = M.lib().mosaic_unmask_noalloc(p, 2049, 2048, fake, 6000, fake, fake, fake, fake, fake,
                                       fake, None, fake, None, 2048, M.GEMM_IMAD, None)
    assert st == 6     # MOSAIC_ERR_WORKSPACE: l * m above 2^22
