"""Tensor-core ring product (tcgen05 kind::f16 on exact bf16 digit planes)
against the oracle's naive Z_{2^32} triple loop: bit-exact on random,
ragged and adversarial operands.  All digits -128 (a = 0x7F7F7F80) make every
digit product +2^14, so shift group 3 reaches exactly 2^24 at the end of each
256-wide K chunk: the edge of exact fp32 accumulation."""
import numpy as np
import pytest

import oracle as O
from paper_2607_29221_gb300 import workloads as wl

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ALL_M128 = 0x7F7F7F80      # every signed digit is -128
ALL_P127 = 0x7F7F7F7F      # every signed digit is +127


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_29221_gb300 import build
    build.build()
    from paper_2607_29221_gb300 import mosaic as M
    if not M.mosaic_gemm_variant_available(M.GEMM_TC):
        pytest.skip("tensor-core variant not available on this device")
    yield


def _M():
    from paper_2607_29221_gb300 import mosaic as M
    return M


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint32)


def planes_of(a_dev, rows, K, ldp):
    M = _M()
    p = torch.zeros(4, rows, ldp, dtype=torch.int16, device="cuda")
    if rows and K:
        src = torch.zeros(rows, ldp, dtype=torch.int32, device="cuda")
        src[:, :K] = a_dev
        M.mosaic_digit_split(src, ldp, rows, ldp, p)
    return p


def tc_gemm(A, B):
    M = _M()
    Mm, K = A.shape
    N = B.shape[0]
    ldp = max(8, (K + 7) // 8 * 8)
    Ap = planes_of(dev(A), Mm, K, ldp)
    Bp = planes_of(dev(B), N, K, ldp)
    C = torch.full((Mm, N + 4), -1, dtype=torch.int32, device="cuda")
    M.mosaic_ring_gemm_planes(Ap, ldp, Mm * ldp, Bp, ldp, N * ldp, C, N + 4, Mm, N, K, M.GEMM_TC)
    M.mosaic_device_status()
    got = host(C)
    assert np.all(got[:, N:] == 0xFFFFFFFF)
    return got[:, :N]


def ref(A, B):
    return O.matmul(A, B.T.copy())


@pytest.mark.parametrize("Mm,N,K", [(128, 128, 32), (128, 128, 256), (130, 257, 33), (1, 1, 8),
                                    (300, 129, 1000), (257, 384, 652), (64, 200, 7),
                                    (512, 640, 4096), (129, 1000, 2049)])
def test_tc_random(Mm, N, K):
    A = wl.uniform_u32(11, Mm, K)
    B = wl.uniform_u32(12, N, K)
    assert np.array_equal(tc_gemm(A, B), ref(A, B))


@pytest.mark.parametrize("K", [256, 512, 1024, 768 + 32, 2048])
@pytest.mark.parametrize("va,vb", [(ALL_M128, ALL_M128), (ALL_P127, ALL_M128), (ALL_P127, ALL_P127)])
def test_tc_adversarial_digits(K, va, vb):
    A = np.full((128, K), va, np.uint32)
    B = np.full((128, K), vb, np.uint32)
    assert np.array_equal(tc_gemm(A, B), ref(A, B))


def test_tc_mixed_magnitudes():
    """Large partial sums followed by small products (rounding would drop the small ones)."""
    K = 512
    A = np.full((256, K), ALL_M128, np.uint32)
    B = np.full((128, K), ALL_M128, np.uint32)
    rng = np.random.Generator(np.random.PCG64(5))
    A[:, 200:] = rng.integers(0, 2**32, (256, K - 200), dtype=np.uint64).astype(np.uint32)
    B[::2, 255] = 0x80808081          # digit 0 = +1, others 0
    A[::3, 255] = 0x80808081
    assert np.array_equal(tc_gemm(A, B), ref(A, B))


def test_tc_through_uint32_entry():
    M = _M()
    A = wl.uniform_u32(21, 200, 96)
    B = wl.uniform_u32(22, 300, 96)
    p = M.default_params()
    ws = torch.empty(M.mosaic_workspace_bytes(M.OP_RING_GEMM, 200, 300, 96, p), dtype=torch.uint8,
                     device="cuda")
    C = torch.empty(200, 300, dtype=torch.int32, device="cuda")
    M.mosaic_ring_gemm(dev(A), 96, dev(B), 96, C, 300, 200, 300, 96, M.GEMM_TC, ws)
    M.mosaic_device_status()
    assert np.array_equal(host(C), ref(A, B))


def test_tc_protocol_layer_matches_oracle():
    """The single 64x256x128 layer with the server product on tensor cores."""
    import test_gpu_parity as T
    g, r, op, m, l = T._run_layer(3, (1536, 1024, 652), (80, 80), m=128, n=256, l=64,
                                  variant=_M().GEMM_TC)
    T._check_layer(g, r, op, m, l)


# --------------------------------------------------------------------------
# Few tokens (M <= 16): the TC variant streams uint32 B through TMA instead of
# splitting it into planes; same ring product, checked the same way.
# --------------------------------------------------------------------------
def ring_gemm_u32(A, B, pad_a=0, pad_b=0, variant=None):
    M = _M()
    variant = M.GEMM_TC if variant is None else variant
    Mm, K = A.shape
    N = B.shape[0]
    lda = (K + 3) // 4 * 4 + pad_a
    ldb = (K + 3) // 4 * 4 + pad_b
    Ad = torch.zeros(Mm, lda, dtype=torch.int32, device="cuda")
    Bd = torch.zeros(N, ldb, dtype=torch.int32, device="cuda")
    Ad[:, :K] = dev(A)
    Bd[:, :K] = dev(B)
    C = torch.full((Mm, N + 4), -1, dtype=torch.int32, device="cuda")
    nb = M.mosaic_workspace_bytes(M.OP_RING_GEMM, Mm, N, K)
    ws = torch.empty(max(nb, 16), dtype=torch.uint8, device="cuda")
    M.mosaic_ring_gemm(Ad, lda, Bd, ldb, C, N + 4, Mm, N, K, variant, ws)
    M.mosaic_device_status()
    got = host(C)
    assert np.all(got[:, N:] == 0xFFFFFFFF)
    return got[:, :N]


@pytest.mark.parametrize("Mm", [1, 2, 3, 4, 5, 8, 9, 16])
@pytest.mark.parametrize("N,K", [(1, 1), (61, 128), (59, 129), (300, 652), (1000, 4100), (121, 8192)])
def test_few_tokens_random(Mm, N, K):
    A = wl.uniform_u32(31 + Mm, Mm, K)
    B = wl.uniform_u32(37, N, K)
    assert np.array_equal(ring_gemm_u32(A, B), ref(A, B))


@pytest.mark.parametrize("val", [0xFFFFFFFF, 0x80000000, ALL_M128, ALL_P127])
def test_few_tokens_constant(val):
    """Constant operands: every row of C is K * val^2 mod 2^32 exactly."""
    Mm, N, K = 7, 190, 1000
    A = np.full((Mm, K), val, dtype=np.uint32)
    B = np.full((N, K), val, dtype=np.uint32)
    want = np.uint32((K * val * val) % (1 << 32))
    assert np.all(ring_gemm_u32(A, B) == want)


def test_few_tokens_unaligned_rows():
    """Row strides that are not multiples of 4 words: AUTO takes the CUDA-core
    product, TC refuses them as misaligned."""
    M = _M()
    A = wl.uniform_u32(41, 3, 130)
    B = wl.uniform_u32(42, 77, 130)
    assert np.array_equal(ring_gemm_u32(A, B, pad_a=1, pad_b=3, variant=M.GEMM_AUTO), ref(A, B))
    with pytest.raises(M.MosaicError, match="misaligned"):
        ring_gemm_u32(A, B, pad_a=1, pad_b=3, variant=M.GEMM_TC)


def test_few_tokens_edges():
    """17 tokens leave the streaming kernel; K = 0 gives zeros."""
    A = wl.uniform_u32(43, 17, 300)
    B = wl.uniform_u32(44, 65, 300)
    assert np.array_equal(ring_gemm_u32(A, B), ref(A, B))
    M = _M()
    C = torch.full((2, 8), -1, dtype=torch.int32, device="cuda")
    Z = torch.zeros(2, 4, dtype=torch.int32, device="cuda")
    M.mosaic_ring_gemm(Z, 4, Z, 4, C, 8, 2, 2, 0, M.GEMM_TC)
    got = host(C)
    assert np.all(got[:, :2] == 0) and np.all(got[:, 2:] == 0xFFFFFFFF)


# --------------------------------------------------------------------------
# 17..64 tokens: the TC variant streams uint32 B by TMA, splits it into fp16
# digits in tensor memory on the chip and runs 4 MMAs per 16 K (one per digit
# of B, N = (4 - i) x token tile); stream-K over (128-row tile, 256-K chunk)
# units, partial tiles added with red.add.
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Mm", [17, 24, 32, 33, 48, 49, 64])
@pytest.mark.parametrize("N,K", [(1, 1), (61, 128), (129, 33), (300, 652), (1000, 4100), (121, 8192),
                                 (257, 257)])
def test_streamw_tokens_random(Mm, N, K):
    A = wl.uniform_u32(131 + Mm, Mm, K)
    B = wl.uniform_u32(137, N, K)
    assert np.array_equal(ring_gemm_u32(A, B), ref(A, B))


@pytest.mark.parametrize("Mm", [20, 40, 64])
@pytest.mark.parametrize("va,vb", [(ALL_M128, ALL_M128), (ALL_P127, ALL_M128), (0xFFFFFFFF, 0x80000000),
                                   (0xFFFFFFFF, 0xFFFFFFFF)])
def test_streamw_tokens_adversarial(Mm, va, vb):
    """Constant digits over K = 3000: shift group 3 reaches 2^24 at every drain
    with all digits -128; every entry is K va vb mod 2^32."""
    Mm, N, K = Mm, 300, 3000
    A = np.full((Mm, K), va, np.uint32)
    B = np.full((N, K), vb, np.uint32)
    want = np.uint32((K * va * vb) % (1 << 32))
    assert np.all(ring_gemm_u32(A, B) == want)


def test_streamw_tokens_many_tiles_and_units():
    """More (tile, chunk) units than SMs with a ragged last tile and K chunk:
    CTAs start and end inside tiles."""
    A = wl.uniform_u32(141, 40, 5000)
    B = wl.uniform_u32(142, 20000 + 77, 5000)
    assert np.array_equal(ring_gemm_u32(A, B), ref(A, B))


@pytest.mark.parametrize("N", [5000, 9984])
def test_tc_whole_waves_then_stream_k(N):
    """160 (312) tiles on 152 SMs with 8 K chunks: the first one (two) waves of
    tiles run whole, one tile per CTA per wave, and the last 8 tiles' chunks
    are shared by all CTAs."""
    A = wl.uniform_u32(51, 512, 2048)
    B = wl.uniform_u32(52, N, 2048)
    assert np.array_equal(tc_gemm(A, B), ref(A, B))



# --------------------------------------------------------------------------
# Legacy mma.sync s8 variant (int8 digit planes, int32 accumulators)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("Mm,N,K", [(1, 1, 1), (64, 64, 64), (65, 130, 33), (300, 129, 1000), (128, 257, 2049),
                                    (17, 999, 4096)])
def test_mma_s8_random(Mm, N, K):
    M = _M()
    if not M.mosaic_gemm_variant_available(M.GEMM_MMA_S8):
        pytest.skip("mma.sync s8 variant not available")
    A = wl.uniform_u32(61, Mm, K)
    B = wl.uniform_u32(62, N, K)
    assert np.array_equal(ring_gemm_u32(A, B, variant=M.GEMM_MMA_S8), ref(A, B))


@pytest.mark.parametrize("va,vb", [(ALL_M128, ALL_M128), (ALL_P127, ALL_M128), (0xFFFFFFFF, 0x80000000)])
def test_mma_s8_adversarial(va, vb):
    """Constant digits over K = 5000: the int32 group sums wrap mod 2^32."""
    M = _M()
    if not M.mosaic_gemm_variant_available(M.GEMM_MMA_S8):
        pytest.skip("mma.sync s8 variant not available")
    Mm, N, K = 70, 90, 5000
    A = np.full((Mm, K), va, np.uint32)
    B = np.full((N, K), vb, np.uint32)
    want = np.uint32((K * va * vb) % (1 << 32))
    assert np.all(ring_gemm_u32(A, B, variant=M.GEMM_MMA_S8) == want)
