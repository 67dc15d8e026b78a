"""One masked decoder layer (four secure linear calls + fp32 RMSNorm, causal GQA
attention, SwiGLU, residuals) against the same layer computed with plain fp32
matrix products: the error is the quantisation and protocol noise of the
linear calls only (Sec. 4.2-4.3: INT16-rot-sigma), small, and growing with sigma."""
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


def _rel(a, b):
    return float(torch.linalg.vector_norm(a - b) / torch.linalg.vector_norm(b))


def test_masked_layer_close_to_float_layer():
    from paper_2607_29221_gb300 import decoder as D
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    s = D.LayerShape(hidden=512, n_heads=8, n_kv=2, head_dim=64, ffn=1536)
    w = D.LayerWeights(s, seed=21)
    x = torch.from_numpy(wl.activations(96, s.hidden)).cuda()
    ref = D.reference_forward(w, x)
    errs = []
    for sigma in (0.0, 0.5, 2.0):
        proto = PR.Protocol(wl.mask_key(), M.default_params(sigma=sigma), variant=M.GEMM_AUTO)
        layer = D.SecureDecoderLayer(proto, w)
        y = layer.forward(x)
        M.mosaic_device_status()
        assert torch.isfinite(y).all()
        errs.append(_rel(y - x, ref - x))
    # relative error of the layer's update (residual removed)
    assert errs[0] < 2e-3, errs
    assert errs[1] < 2e-2, errs
    assert errs[0] <= errs[1] <= errs[2], errs
