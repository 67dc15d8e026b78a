"""Edge cases of every entry point on the device: empty batches (l = 0, zero
rows, M = 0, N = 0) succeed and touch nothing, an empty contraction (K = 0)
writes the zero matrix, and the largest contraction the library accepts
(K = 2^20) stays bit-exact against the oracle's naive Z_{2^32} triple loop
on every product variant, with both random and all-(-128)-digit operands
(the latter put the largest possible sums into every shift group)."""
import numpy as np
import pytest

import oracle as O
from paper_2607_29221_gb300 import workloads as wl

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

KEY = wl.mask_key()
SENT = 0x5A5A5A5A


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_29221_gb300 import build
    build.build()
    from paper_2607_29221_gb300 import mosaic as M
    M.lib()
    yield


def _M():
    from paper_2607_29221_gb300 import mosaic as M
    return M


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint32)


def sentinel(*shape, dtype=torch.int32):
    return torch.full(shape, SENT, dtype=dtype, device="cuda")


def untouched(t):
    torch.cuda.synchronize()
    return bool((t == SENT).all())


def _variants():
    M = _M()
    return [v for v in (M.GEMM_AUTO, M.GEMM_TC, M.GEMM_MMA_S8, M.GEMM_IMAD)
            if v in (M.GEMM_AUTO, M.GEMM_IMAD) or M.mosaic_gemm_variant_available(v)]


def _gemm(A, B, C, Mm, N, K, variant):
    M = _M()
    ws = torch.empty(max(256, M.mosaic_workspace_bytes(M.OP_RING_GEMM, Mm, N, K)), dtype=torch.uint8,
                     device="cuda")
    M.mosaic_ring_gemm(A, max(K, 1), B, max(K, 1), C, N, Mm, N, K, variant, ws)


def test_empty_batches_touch_nothing():
    M = _M()
    p = M.default_params(d=3, r=[96, 64, 40], t=[0, 6, 5])
    key = M.make_key(KEY)
    m, n_pad = 64, 128
    Sr = 96 + 64 + 40
    buf = sentinel(4096)
    f_buf = sentinel(4096, dtype=torch.float32)
    ctr = torch.zeros(1, dtype=torch.int64, device="cuda")
    # samplers and rotations with no rows
    M.mosaic_prg_uniform(key, 1, 0, 20, 0, 7, buf)
    M.mosaic_prg_gaussian(key, 2, 0, 20, 0.5, 0, buf)
    M.mosaic_prg_sparse(key, 3, 0, 20, 0, 64, 6, buf, buf)
    M.mosaic_hadamard(f_buf, n_pad, f_buf, 0, 100, n_pad)
    M.mosaic_encode(f_buf, n_pad, 0, 100, n_pad, M.mosaic_qmax(n_pad), 1, buf, buf, n_pad, buf, n_pad, f_buf)
    M.mosaic_digit_split(buf, 8, 0, 8, buf)
    # products with an empty side, on every variant
    for v in _variants():
        _gemm(buf, buf, buf, 0, 5, 8, v)
        _gemm(buf, buf, buf, 5, 0, 8, v)
    # the protocol steps with no tokens
    M.mosaic_mask_activation(p, key, 9, m, n_pad, 0, buf, buf, buf, buf, M.GEMM_AUTO, None)
    M.mosaic_mask_activation_ex(p, key, 9, ctr, m, n_pad, 0, buf, buf, None, buf, buf, M.GEMM_AUTO, None)
    M.mosaic_unmask(p, 0, m, buf, m + Sr, buf, buf, buf, buf, f_buf, f_buf, None, f_buf, buf, m,
                    M.GEMM_AUTO, None)
    M.mosaic_unmask_planes(p, 0, m, buf, m + Sr, buf, buf, buf, buf, buf, f_buf, f_buf, None, f_buf, buf,
                           m, M.GEMM_AUTO, None)
    M.mosaic_unmask_noalloc(p, 0, m, buf, m + Sr, buf, buf, buf, buf, f_buf, f_buf, None, f_buf, buf, m,
                            M.GEMM_AUTO)
    M.mosaic_freivalds_check(4, buf, buf, m, n_pad, 0, buf, m, buf, n_pad, buf, buf, None)
    M.mosaic_advance_pass(ctr, 0)
    M.mosaic_device_status()
    assert untouched(buf) and untouched(f_buf)
    assert int(ctr.item()) == 0


@pytest.mark.parametrize("Mm,N", [(3, 5), (130, 257)])
def test_empty_contraction_writes_zeros(Mm, N):
    for v in _variants():
        A = sentinel(Mm, 4)
        B = sentinel(N, 4)
        C = sentinel(Mm, N)
        _gemm(A, B, C, Mm, N, 0, v)
        assert not host(C).any(), v


def _max_k_case(Mm, N, K, adversarial):
    if adversarial:
        A = np.full((Mm, K), 0x7F7F7F80, np.uint32)    # every signed digit -128
        B = np.full((N, K), 0x7F7F7F80, np.uint32)
    else:
        A = wl.uniform_u32(71, Mm, K)
        B = wl.uniform_u32(72, N, K)
    return A, B


@pytest.mark.parametrize("adversarial", [False, True])
@pytest.mark.parametrize("Mm,N", [(3, 40), (20, 24)])
def test_largest_contraction_is_exact(Mm, N, adversarial):
    K = 1 << 20
    A, B = _max_k_case(Mm, N, K, adversarial)
    ref = O.matmul(A, B.T.copy())
    dA, dB = dev(A), dev(B)
    for v in _variants():
        C = sentinel(Mm, N)
        _gemm(dA, dB, C, Mm, N, K, v)
        assert np.array_equal(host(C), ref), v
    _M().mosaic_device_status()


def test_bounded_wait_expiry_is_reported_and_the_context_survives():
    """A bounded device wait on a barrier that nothing completes runs out after
    2 ms; the next device status reports the timeout (and clears it), and the
    context keeps working (a product afterwards is still exact)."""
    M = _M()
    M.mosaic_device_status()
    M.mosaic_selftest_wait(2000)
    with pytest.raises(M.MosaicError) as ei:
        M.mosaic_device_status()
    assert ei.value.status == 7
    M.mosaic_device_status()          # cleared
    A = wl.uniform_u32(81, 5, 33)
    B = wl.uniform_u32(82, 7, 33)
    C = sentinel(5, 7)
    _gemm(dev(A), dev(B), C, 5, 7, 33, M.GEMM_AUTO)
    assert np.array_equal(host(C), O.matmul(A, B.T.copy()))
    M.mosaic_device_status()
