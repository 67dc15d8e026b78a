"""One masked decoder layer (four secure linear calls + fp32 RMSNorm, causal GQA
attention, SwiGLU, residuals; Sec. 4.1 and Sec. 3.2 "Local attention
computation") against a float reference written here in fp64 numpy -- RMSNorm,
causal grouped-query softmax attention, SiLU(gate) * up, residuals and plain
matrix products, sharing no code with the product's layer.

* The fp32 glue alone agrees with the fp64 reference to fp32 rounding.
* The masked layer's update (output minus the residual input) is within the
  quantisation and protocol noise of the four linear calls (Sec. 4.2-4.3:
  INT16-rot-sigma): small, and growing with sigma.
* The layer captured as one CUDA graph with a device pass counter replays
  bit-identically to eager passes with the same pass ids."""
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


# ---------------------------------------------------------------------------
# fp64 reference of the layer (test-side, independent of decoder.py)
# ---------------------------------------------------------------------------
def ref_rmsnorm(x, eps):
    return x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + eps)


def ref_attention(qkv, H, KV, d):
    """Causal GQA: query head h reads key/value head h // (H / KV)."""
    l = qkv.shape[0]
    out = np.zeros((l, H * d))
    future = np.triu(np.ones((l, l), dtype=bool), 1)
    for h in range(H):
        g = h // (H // KV)
        q = qkv[:, h * d:(h + 1) * d]
        k = qkv[:, (H + g) * d:(H + g + 1) * d]
        v = qkv[:, (H + KV + g) * d:(H + KV + g + 1) * d]
        s = q @ k.T / np.sqrt(d)
        s[future] = -np.inf
        s = np.exp(s - s.max(axis=1, keepdims=True))
        out[:, h * d:(h + 1) * d] = (s / s.sum(axis=1, keepdims=True)) @ v
    return out


def ref_layer(W, x, H, KV, d, ffn, eps):
    Wqkv, Wo, Wgu, Wdown = (w.astype(np.float64) for w in W)
    x = x.astype(np.float64)
    a = ref_attention(ref_rmsnorm(x, eps) @ Wqkv.T, H, KV, d)
    x = x + a @ Wo.T
    gu = ref_rmsnorm(x, eps) @ Wgu.T
    g, u = gu[:, :ffn], gu[:, ffn:]
    return x + (g / (1.0 + np.exp(-g)) * u) @ Wdown.T


def _np(t):
    return t.detach().cpu().numpy()


def _rel(a, b):
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


SHAPES = {
    "small": dict(hidden=512, n_heads=8, n_kv=2, head_dim=64, ffn=1536),
    "gqa8": dict(hidden=2048, n_heads=16, n_kv=2, head_dim=128, ffn=5632),
}


@pytest.mark.parametrize("name,l", [("small", 96), ("gqa8", 200)])
def test_fp32_glue_matches_fp64_reference(name, l):
    from paper_2607_29221_gb300 import decoder as D
    s = D.LayerShape(**SHAPES[name])
    x = wl.activations(l, s.hidden, seed=31)
    qkv = wl.activations(l, s.qkv, seed=32)
    got_n = _np(D.rmsnorm(torch.from_numpy(x).cuda(), s.eps))
    assert _rel(got_n, ref_rmsnorm(x.astype(np.float64), s.eps)) < 1e-6
    gu = wl.activations(l, 2 * s.ffn, seed=33) * 4.0
    got_s = _np(D.swiglu(torch.from_numpy(gu).cuda(), s.ffn))
    g, u = gu[:, :s.ffn].astype(np.float64), gu[:, s.ffn:].astype(np.float64)
    assert _rel(got_s, g / (1.0 + np.exp(-g)) * u) < 1e-6
    got_a = _np(D.attention(torch.from_numpy(qkv).cuda(), s))
    ref_a = ref_attention(qkv.astype(np.float64), s.n_heads, s.n_kv, s.head_dim)
    assert np.max(np.abs(got_a - ref_a)) < 1e-5 * np.max(np.abs(ref_a)) + 1e-6
    # token 0 attends to itself only: its output is its own value row
    g = s.n_heads // s.n_kv
    for h in (0, s.n_heads - 1):
        v0 = qkv[0, (s.n_heads + s.n_kv + h // g) * s.head_dim:(s.n_heads + s.n_kv + h // g + 1) * s.head_dim]
        assert np.allclose(got_a[0, h * s.head_dim:(h + 1) * s.head_dim], v0, rtol=1e-6, atol=1e-6)


@pytest.mark.parametrize("rows,n,ld", [(3, 37, 41), (5, 4096, 4100), (1, 1, 1)])
def test_glue_kernels_on_ragged_rows(rows, n, ld):
    """RMSNorm and SwiGLU on widths that are not multiples of 4 and padded
    leading dimensions (the scalar paths), against fp64; the padding is untouched."""
    from paper_2607_29221_gb300 import decoder as D
    x = wl.activations(rows, ld, seed=34)
    xt = torch.from_numpy(x).cuda()
    y = torch.full((rows, ld), 7.0, dtype=torch.float32, device="cuda")
    M = __import__("paper_2607_29221_gb300.mosaic", fromlist=["x"])
    M.mosaic_rmsnorm(xt, ld, rows, n, 1e-5, y, ld)
    xv = x[:, :n].astype(np.float64)
    want = xv / np.sqrt(np.mean(xv * xv, axis=1, keepdims=True) + 1e-5)
    got = _np(y)
    assert _rel(got[:, :n], want) < 1e-6 and np.all(got[:, n:] == 7.0)
    gu = wl.activations(rows, 2 * n + 3, seed=35)
    out = torch.full((rows, n + 2), 5.0, dtype=torch.float32, device="cuda")
    M.mosaic_swiglu(torch.from_numpy(gu).cuda(), 2 * n + 3, rows, n, out, n + 2)
    g, u = gu[:, :n].astype(np.float64), gu[:, n:2 * n].astype(np.float64)
    got = _np(out)
    assert _rel(got[:, :n], g / (1.0 + np.exp(-g)) * u) < 1e-6 and np.all(got[:, n:] == 5.0)


@pytest.mark.parametrize("name,l", [("small", 96), ("gqa8", 160)])
def test_masked_layer_close_to_float_layer(name, l):
    from paper_2607_29221_gb300 import decoder as D
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    s = D.LayerShape(**SHAPES[name])
    w = D.LayerWeights(s, seed=21)
    x = wl.activations(l, s.hidden)
    ref = ref_layer([_np(w.Wqkv), _np(w.Wo), _np(w.Wgu), _np(w.Wdown)], x, s.n_heads, s.n_kv,
                    s.head_dim, s.ffn, s.eps)
    errs = []
    for sigma in (0.0, 0.5, 2.0):
        proto = PR.Protocol(wl.mask_key(), M.default_params(sigma=sigma), variant=M.GEMM_AUTO)
        layer = D.SecureDecoderLayer(proto, w)
        y = _np(layer.forward(torch.from_numpy(x).cuda()))
        M.mosaic_device_status()
        assert np.all(np.isfinite(y))
        errs.append(_rel(y - x, ref - x))      # relative error of the layer's update
        del layer
    # sigma = 0 leaves the quantisation error: a rotated row's absmax is about 4
    # standard deviations, so rounding to q_max levels adds a relative RMS error of
    # about (4 / q_max) / sqrt(12) = 1.15 / q_max per operand; bound the layer's
    # update by 2.5 / q_max of its narrowest window.
    from paper_2607_29221_gb300 import protocol as PR
    qmin = min(M.mosaic_qmax(PR.pad_width(n)) for n in (s.hidden, s.ffn))
    assert errs[0] < 2.5 / qmin, (errs, qmin)
    assert errs[1] < 2e-2, errs
    assert errs[0] <= errs[1] <= errs[2], errs


def test_layer_graph_replays_match_eager_passes():
    from paper_2607_29221_gb300 import decoder as D
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    s = D.LayerShape(**SHAPES["small"])
    l = 64
    proto = PR.Protocol(wl.mask_key(), M.default_params(), variant=M.GEMM_AUTO)
    layer = D.SecureDecoderLayer(proto, D.LayerWeights(s, seed=23))
    layer.alloc(l)
    x = torch.from_numpy(wl.activations(l, s.hidden, seed=5)).cuda()
    base = 300
    eager = []
    for k in range(2):
        y = layer.forward(x, layer.init_x(l, base + k))
        torch.cuda.synchronize()
        eager.append(_np(y).copy())
    ctr = torch.zeros(1, dtype=torch.int64, device="cuda")
    gm = layer.init_x(l, base)
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        y_g = layer.forward(x, layer.init_x(l, base, pass_dev=ctr, out=gm))
        M.mosaic_advance_pass(ctr, 1, stream=side)
    torch.cuda.synchronize()
    for k in range(2):
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(_np(y_g), eager[k]), k
    assert not np.array_equal(eager[0], eager[1])
    M.mosaic_device_status()


@pytest.mark.parametrize("l", [64, 24])
def test_overlapped_pass_matches_init_x_then_forward(l):
    """forward_pass (the four calls' Init X draws on a side stream from the
    start of the pass, each composition right before its call's encode) gives
    the decoded output of init_x + forward with the same pass ids, bit for bit:
    eager, and captured as one CUDA graph whose replays advance a device pass
    counter.  l = 24 runs the streaming tensor-core server product."""
    from paper_2607_29221_gb300 import decoder as D
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    s = D.LayerShape(**SHAPES["small"])
    proto = PR.Protocol(wl.mask_key(), M.default_params(), variant=M.GEMM_AUTO)
    layer = D.SecureDecoderLayer(proto, D.LayerWeights(s, seed=29))
    layer.alloc(l)
    x = torch.from_numpy(wl.activations(l, s.hidden, seed=6)).cuda()
    base = 700
    want = []
    for k in range(3):
        want.append(_np(layer.forward(x, layer.init_x(l, base + k))).copy())
    masks = layer.init_x(l, 1)
    got = _np(layer.forward_pass(x, base, masks)).copy()
    assert np.array_equal(got, want[0])
    ctr = torch.zeros(1, dtype=torch.int64, device="cuda")
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=side):
        y_g = layer.forward_pass(x, base, masks, pass_dev=ctr)
        M.mosaic_advance_pass(ctr, 1, stream=side)
    torch.cuda.synchronize()
    for k in range(3):
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(_np(y_g), want[k]), k
    M.mosaic_device_status()
