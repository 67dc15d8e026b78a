"""A whole masked-linear step (Init X, encode + mask-add, server product,
unmask + decode) captured as one CUDA graph, as the benchmark runs it: replay
k draws pass base + k from the device counter, bit-identical in the server
output Z and the decoded Y to the eager call with that pass id, and
consecutive replays use different masks.  (Y itself differs slightly between
passes: the LWE noise E_x of a pass does not cancel in the unmask.)"""
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
    from paper_2607_29221_gb300 import mosaic as M
    M.lib()
    yield


def _bits(t):
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint32).copy()


@pytest.mark.parametrize("l", [48, 8])
def test_graph_step_matches_eager_passes(l):
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    gp = M.default_params(d=3, r=[96, 64, 40], t=[0, 8, 4])
    proto = PR.Protocol(KEY, gp, variant=M.GEMM_AUTO)
    m, n = 200, 256
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, torch.from_numpy(wl.weights(m, n, std=1.0)).cuda(), 3, ch)
    N = m + proto.sum_r
    X = torch.from_numpy(wl.activations(l, n)).cuda()
    bufs = dict(Xp=torch.empty(l, layer.n_pad, dtype=torch.int32, device="cuda"),
                s_x=torch.empty(l, dtype=torch.float32, device="cuda"),
                Xpl=torch.empty(4, l, layer.n_pad, dtype=torch.int16, device="cuda"),
                Z=torch.empty(l, N, dtype=torch.int32, device="cuda"),
                Y=torch.empty(l, m, dtype=torch.float32, device="cuda"))

    def step(mp):
        layer.mask_input(X, mp, bufs["Xp"], bufs["s_x"], bufs["Xpl"])
        layer.server(bufs["Xp"], bufs["Xpl"], bufs["Z"])
        layer.unmask(bufs["Z"], mp, bufs["s_x"], bufs["Y"])

    base = 5000
    eager = []
    for k in range(2):
        step(layer.init_x(l, base + k))
        eager.append((_bits(bufs["Z"]), _bits(bufs["Y"])))
    ctr = torch.zeros(1, dtype=torch.int64, device="cuda")
    gm = layer.init_x(l, base)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        step(layer.init_x(l, base, pass_dev=ctr, out=gm))
        M.mosaic_advance_pass(ctr, 1, stream=side)
    torch.cuda.synchronize()
    assert int(ctr.item()) == 0
    for k in range(2):
        g.replay()
        Z, Y = _bits(bufs["Z"]), _bits(bufs["Y"])
        assert np.array_equal(Z, eager[k][0]), k
        assert np.array_equal(Y, eager[k][1]), k
    assert int(ctr.item()) == 2
    assert not np.array_equal(eager[0][0], eager[1][0])   # fresh masks per pass
    M.mosaic_device_status()


def test_kernel_timing_records_eager_launches_only():
    """Per-kernel timing: an eager step with timing on records every launch
    of the library (Init X draws, product and gathers, the server product, the
    unmask) under the entry point that made it, as many as the launch counter
    saw, with the outputs unchanged; a launch captured into a CUDA graph is
    not recorded."""
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    gp = M.default_params(d=3, r=[96, 64, 40], t=[0, 8, 4])
    proto = PR.Protocol(KEY, gp, variant=M.GEMM_TC)
    m, n, l = 256, 256, 64
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, torch.from_numpy(wl.weights(m, n, std=1.0)).cuda(), 3, ch)
    X = torch.from_numpy(wl.activations(l, n)).cuda()
    Y0 = layer.forward(X, layer.init_x(l, 77)).clone()
    mp = layer.init_x(l, 78)
    Xp = torch.empty(l, layer.n_pad, dtype=torch.int32, device="cuda")
    s_x = torch.empty(l, dtype=torch.float32, device="cuda")
    Xpl = torch.empty(4, l, layer.n_pad, dtype=torch.int16, device="cuda")
    Z = torch.empty(l, m + proto.sum_r, dtype=torch.int32, device="cuda")
    layer.mask_input(X, mp, Xp, s_x, Xpl)
    torch.cuda.synchronize()
    M.mosaic_kernel_times(reset=True)
    M.mosaic_kernel_timing(True)
    try:
        n0 = M.mosaic_kernel_launches()
        Y1 = layer.forward(X, layer.init_x(l, 77))
        torch.cuda.synchronize()
        launched = M.mosaic_kernel_launches() - n0
        kt = M.mosaic_kernel_times(reset=True)
        side = torch.cuda.Stream()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=side):
            layer.server(Xp, Xpl, Z)
        torch.cuda.synchronize()
        captured = M.mosaic_kernel_times(reset=True)
    finally:
        M.mosaic_kernel_timing(False)
    assert torch.equal(Y0, Y1)
    assert sum(v[0] for v in kt.values()) == launched
    for key in ("init_x:initx_draw", "init_x:ring_gemm_tc", "unmask:ring_gemm_tc"):
        assert key in kt and kt[key][0] >= 1 and kt[key][1] > 0.0, (key, kt)
    for role in ("init_x:", "unmask:"):
        assert any(k.startswith(role) and "gather" in k for k in kt), kt
    assert any(k.startswith("encode:") for k in kt) and any(k.startswith("ring_gemm:") for k in kt), kt
    assert captured == {}
    g.replay()
    torch.cuda.synchronize()
    del g


def test_int_mix_rate_is_measured_and_validated():
    """mosaic_int_mix_rate: a positive rate of the ChaCha20 mix within the
    bounds one GB300-class part allows, and a refusal of a scratch buffer
    that is too small."""
    from paper_2607_29221_gb300 import mosaic as M
    scratch = torch.empty(8 * 256 * 256, dtype=torch.int32, device="cuda")
    rate = M.mosaic_int_mix_rate(scratch)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    # between 16 and 256 32-bit ops per clock per SM at 0.5 to 3 GHz
    assert sms * 16 * 0.5e9 < rate < sms * 256 * 3.0e9, rate
    with pytest.raises(M.MosaicError):
        M.mosaic_int_mix_rate(torch.empty(16, dtype=torch.int32, device="cuda"))


def test_smem_read_rate_is_measured_and_validated():
    """mosaic_smem_read_rate: a positive shared-memory read rate no higher than
    a few lines per clock per SM, and a refusal of a scratch buffer that is
    too small."""
    from paper_2607_29221_gb300 import mosaic as M
    scratch = torch.empty(8 * 256 * 256, dtype=torch.int32, device="cuda")
    rate = M.mosaic_smem_read_rate(scratch)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert sms * 16 * 0.5e9 < rate < sms * 512 * 3.0e9, rate
    with pytest.raises(M.MosaicError):
        M.mosaic_smem_read_rate(torch.empty(16, dtype=torch.int32, device="cuda"))
