"""Parity of the CUDA path (through the C ABI) with the CPU oracle on the
same seeded inputs: bit-exact for every ring, integer and sampled output and
for the fp32 rotation (same stage order); decoded floats within
1e-6 x (|Y_hat s_w s_x| + |b|) of the oracle's fp64 decode."""
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


def M_():
    from paper_2607_29221_gb300 import mosaic as M
    return M


def dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a).cuda()


def host_u32(t):
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint32)


def host_f32(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def ckey():
    return M_().make_key(KEY)


# --------------------------------------------------------------------------
# Samplers
# --------------------------------------------------------------------------
@pytest.mark.parametrize("rows,cols,ld,rounds", [(1, 1, 1, 20), (3, 17, 20, 20), (65, 652, 652, 20),
                                                 (1024, 1536, 1536, 20), (7, 33, 40, 8),
                                                 (9, 31, 31, 12)])
def test_prg_uniform(rows, cols, ld, rounds):
    M = M_()
    tg, sid = O.tag(O.KIND_L), 0x123456789
    out = torch.full((rows, ld), -1, dtype=torch.int32, device="cuda")
    M.mosaic_prg_uniform(ckey(), tg, sid, rounds, rows, cols, out, ld)
    got = host_u32(out)
    assert np.array_equal(got[:, :cols], O.sample_uniform(KEY, tg, sid, rows, cols, rounds))
    assert np.all(got[:, cols:] == 0xFFFFFFFF)


@pytest.mark.parametrize("sigma", [0.5, 1.0, 2.0, 0.0, 8.0])
@pytest.mark.parametrize("count", [1, 7, 12345, 1 << 20])
def test_prg_gaussian(sigma, count):
    M = M_()
    out = torch.full((count + 3,), 7, dtype=torch.int32, device="cuda")
    M.mosaic_prg_gaussian(ckey(), O.tag(O.KIND_EW), 42, 20, sigma, count, out)
    got = host_u32(out)
    assert np.array_equal(got[:count], O.sample_gaussian(KEY, O.tag(O.KIND_EW), 42, count, sigma))
    assert np.all(got[count:] == 7)


@pytest.mark.parametrize("rows,r,t", [(1, 4, 2), (100, 1536, 80), (2049, 1024, 80), (33, 652, 1),
                                      (5, 64, 32)])
def test_prg_sparse(rows, r, t):
    M = M_()
    idx = torch.zeros(rows, t, dtype=torch.int32, device="cuda")
    val = torch.zeros(rows, t, dtype=torch.int32, device="cuda")
    fail = torch.zeros(1, dtype=torch.int32, device="cuda")
    M.mosaic_prg_sparse(ckey(), O.tag(O.KIND_T, 2), 9, 20, rows, r, t, idx, val, fail)
    wi, wv = O.sample_sparse(KEY, O.tag(O.KIND_T, 2), 9, rows, r, t)
    assert np.array_equal(host_u32(idx), wi)
    assert np.array_equal(host_u32(val), wv)
    assert host_u32(fail)[0] == 0


# --------------------------------------------------------------------------
# Rotation and encoding
# --------------------------------------------------------------------------
NPADS = [32, 64, 128, 256, 512, 1024, 2048, 4096, 8192, 16384, 32768, 65536]


@pytest.mark.parametrize("n_pad", NPADS)
def test_hadamard_bit_exact(n_pad):
    M = M_()
    rows = 5 if n_pad >= 8192 else 19
    # (n_pad // 2 - 3 leaves the upper half of a 65536 row empty)
    for n in sorted({n_pad, max(1, n_pad - 3), n_pad // 2 + 1, max(1, n_pad // 2 - 3)}):
        x = wl.activations(rows, n, seed=n)
        words = O.sample_signs(KEY, 11, n_pad)
        y = torch.empty(rows, n_pad, dtype=torch.float32, device="cuda")
        M.mosaic_hadamard(dev(x), n, y, rows, n, n_pad, dev(words))
        want = O.fwht_rows(x, n_pad, words)
        assert np.array_equal(host_f32(y).view(np.uint32), want.view(np.uint32)), n
    # D = I and a row stride larger than n
    x = wl.activations(3, n_pad + 8, seed=5)
    y = torch.empty(3, n_pad, dtype=torch.float32, device="cuda")
    M.mosaic_hadamard(dev(x), n_pad + 8, y, 3, n_pad, n_pad, None)
    assert np.array_equal(host_f32(y), O.fwht_rows(x[:, :n_pad], n_pad, None))


@pytest.mark.parametrize("n_pad", [32, 256, 1024, 4096, 16384, 32768, 65536])
def test_encode_bit_exact(n_pad):
    M = M_()
    rows = 6 if n_pad >= 16384 else 23
    n = n_pad - 5 if n_pad > 64 else n_pad
    x = wl.spike_activations(rows, n, seed=3)
    x[1, :] = 0.0                  # zero row: scale 0, code 0
    x[2, 7] = np.inf               # non-finite row: scale NaN, code 0
    words = O.sample_signs(KEY, 12, n_pad)
    mask = wl.uniform_u32(9, rows, n_pad)
    qmax = O.qmax_for(n_pad)
    for rotate in (1, 0):
        out = torch.empty(rows, n_pad, dtype=torch.int32, device="cuda")
        sc = torch.empty(rows, dtype=torch.float32, device="cuda")
        planes = torch.empty(4, rows, n_pad, dtype=torch.int16, device="cuda")
        M.mosaic_encode(dev(x), n, rows, n, n_pad, qmax, rotate, dev(words), dev(mask), n_pad, out,
                        n_pad, sc, planes)
        if rotate:
            v = O.fwht_rows(x, n_pad, words)
        else:
            v = np.zeros((rows, n_pad), np.float32); v[:, :n] = x
        code, scale = O.encode_rows(v, qmax)
        got = host_u32(out)
        assert np.array_equal(got, code + mask)
        gs = host_f32(sc)
        assert np.array_equal(np.isnan(gs), np.isnan(scale))
        assert np.array_equal(gs[~np.isnan(gs)], scale[~np.isnan(scale)])
        assert np.isnan(gs[2]) and gs[1] == 0
        # planes are the signed digits of out, exactly representable in bf16
        pl = host_f32(planes.view(torch.bfloat16).float()).astype(np.int64)
        rebuilt = sum(pl[i] << (8 * i) for i in range(4)) % (1 << 32)
        assert np.array_equal(rebuilt.astype(np.uint32), got)
        assert pl.min() >= -128 and pl.max() <= 127


def test_digit_split_identity():
    M = M_()
    a = wl.uniform_u32(4, 37, 64)
    a[0, :8] = [0, 0x7F7F7F7F, 0x80808080, 0xFFFFFFFF, 1, 0x80000000, 0x7FFFFFFF, 0x01010101]
    planes = torch.empty(4, 37, 64, dtype=torch.int16, device="cuda")
    M.mosaic_digit_split(dev(a), 64, 37, 64, planes)
    pl = host_f32(planes.view(torch.bfloat16).float()).astype(np.int64)
    assert pl.min() >= -128 and pl.max() <= 127
    rebuilt = sum(pl[i] << (8 * i) for i in range(4)) % (1 << 32)
    assert np.array_equal(rebuilt.astype(np.uint32), a)
    # 0x80808080 + 0x80808080 = 0x01010100 (mod 2^32) -> digits (0-128, 1-128, 1-128, 1-128)
    assert list(pl[:, 0, 2]) == [-128, -127, -127, -127]


# --------------------------------------------------------------------------
# Ring product
# --------------------------------------------------------------------------
GEMM_SHAPES = [(1, 1, 1), (5, 3, 7), (130, 257, 33), (128, 128, 16), (300, 129, 1000), (64, 200, 0),
               (257, 384, 652)]


@pytest.mark.parametrize("Mm,N,K", GEMM_SHAPES)
def test_ring_gemm_imad(Mm, N, K):
    M = M_()
    A = wl.uniform_u32(1, Mm, max(K, 1))[:, :K].copy()
    B = wl.uniform_u32(2, N, max(K, 1))[:, :K].copy()
    if K:
        A[0, :] = 0xFFFFFFFF; B[0, :] = 0xFFFFFFFF
    C = torch.full((Mm, N + 3), -1, dtype=torch.int32, device="cuda")
    M.mosaic_ring_gemm(dev(A) if K else torch.zeros(Mm, 1, dtype=torch.int32, device="cuda"),
                       max(K, 1), dev(B) if K else torch.zeros(N, 1, dtype=torch.int32, device="cuda"),
                       max(K, 1), C, N + 3, Mm, N, K, M.GEMM_IMAD)
    got = host_u32(C)
    want = O.matmul(A, B.T.copy()) if K else np.zeros((Mm, N), np.uint32)
    assert np.array_equal(got[:, :N], want)
    assert np.all(got[:, N:] == 0xFFFFFFFF)


# --------------------------------------------------------------------------
# Masks, server, unmask
# --------------------------------------------------------------------------
def _params(d, r, t, sigma=0.5, act_nested=True):
    M = M_()
    tt = [0] + list(t)
    return (M.default_params(d=d, r=list(r) + [0] * (3 - len(r)), t=tt + [0] * (3 - len(tt)),
                             sigma=sigma, act_nested=int(act_nested)),
            O.Params(d=d, r=tuple(r), t=tuple(t), sigma=sigma, act_nested=act_nested))


def _run_layer(d, r, t, m, n, l, sigma=0.5, w_std=1.0, bias=True, variant=None, act_nested=True):
    from paper_2607_29221_gb300 import protocol as PR
    M = M_()
    gp, op = _params(d, r, t, sigma, act_nested)
    variant = M.GEMM_IMAD if variant is None else variant
    proto = PR.Protocol(KEY, gp, variant=variant)
    n_pad = PR.pad_width(n)
    W = wl.weights(m, n, std=w_std)
    X_tm = wl.activations(l, n)
    b = wl.bias(m) if bias else None
    ch = PR.Chains(proto, n_pad)
    layer = PR.SecureLinear(proto, dev(W), 5, ch, bias=dev(b) if bias else None)
    mp = layer.init_x(l, 77)
    Xp, s_x, Xpl = layer.mask_input(dev(X_tm), mp)
    Z = layer.server(Xp, Xpl)
    Yhat = torch.empty(l, m, dtype=torch.int32, device="cuda")
    Y = layer.unmask(Z, mp, s_x, Yhat=Yhat)
    g = dict(P=host_u32(ch.P), C=host_u32(ch.C), CT=host_u32(ch.CT), Wp=host_u32(layer.Wp),
             J=host_u32(layer.J), L=host_u32(layer.L), S_idx=host_u32(layer.S_idx),
             S_val=host_u32(layer.S_val), s_w=host_f32(layer.s_w), signs=host_u32(layer.sign_words),
             Ux=host_u32(mp.Ux), K=host_u32(mp.K), Xp=host_u32(Xp), s_x=host_f32(s_x),
             Z=host_u32(Z), Yhat=host_u32(Yhat), Y=host_f32(Y))
    ref = O.secure_linear(KEY, op, W, X_tm.T.copy(), matrix_id=5, pass_id=77, b=b)
    ref["bias"] = b
    return g, ref, op, m, l


def _check_layer(g, ref, op, m, l):
    P = np.vstack(ref["P"]); C = np.hstack(ref["C"])
    assert np.array_equal(g["P"], P)
    assert np.array_equal(g["C"], C)
    assert np.array_equal(g["CT"], C.T)
    ws, ps = ref["ws"], ref["ps"]
    assert np.array_equal(g["signs"], ws.sign_words)
    assert np.array_equal(g["s_w"], ws.s_w)
    assert np.array_equal(g["L"], ws.L)
    off = 0
    for i in range(1, op.d):
        t = op.t[i - 1]
        assert np.array_equal(g["S_idx"][off:off + m * t].reshape(m, t), ws.S[i + 1][0])
        assert np.array_equal(g["S_val"][off:off + m * t].reshape(m, t), ws.S[i + 1][1])
        off += m * t
    assert np.array_equal(g["Wp"][:m], ws.W_masked)
    assert np.array_equal(g["Wp"][m:], P)
    if op.act_nested:
        assert np.array_equal(g["J"], np.hstack(ws.J))
    else:   # only J_1 is written
        assert np.array_equal(g["J"][:, :op.r[0]], ws.J[0])
    assert np.array_equal(g["Ux"], ps.U_x.T)
    assert np.array_equal(g["K"], ps.K.T)
    assert np.array_equal(g["Xp"], ref["X_masked"].T)
    assert np.array_equal(g["s_x"], ref["s_x"])
    Zref = np.hstack([ref["Y_masked"].T] + [q.T for q in ref["Q"]])
    assert np.array_equal(g["Z"], Zref)
    assert np.array_equal(g["Yhat"], ref["Y_hat"].T)
    Yref = ref["Y"].T
    mag = np.abs(ref["Y_hat"].T.view(np.int32).astype(np.float64) * ws.s_w[None, :].astype(np.float64)
                 * ref["s_x"][:, None].astype(np.float64))
    if ref["bias"] is not None:
        mag = mag + np.abs(ref["bias"].astype(np.float64))[None, :]
    assert np.all(np.abs(g["Y"].astype(np.float64) - Yref) <= 1e-6 * mag)


def _variants():
    M = M_()
    out = [M.GEMM_IMAD]
    if M.mosaic_gemm_variant_available(M.GEMM_TC):
        out.append(M.GEMM_TC)
    if M.mosaic_gemm_variant_available(M.GEMM_MMA_S8):
        out.append(M.GEMM_MMA_S8)
    return out


@pytest.mark.parametrize("d,r,t", [(1, (96,), ()), (2, (96, 64), (6,)), (3, (96, 64, 40), (6, 5))])
def test_layer_small_ranks(d, r, t):
    for variant in _variants():
        g, ref, op, m, l = _run_layer(d, r, t, m=40, n=100, l=21, variant=variant)
        _check_layer(g, ref, op, m, l)


def test_layer_ranks_not_multiple_of_eight():
    """r_d = 37 and m, l ragged: every product has a ragged K tail."""
    for variant in _variants():
        g, ref, op, m, l = _run_layer(3, (100, 70, 37), (9, 7), m=131, n=300, l=67, variant=variant)
        _check_layer(g, ref, op, m, l)


@pytest.mark.parametrize("l", [1, 2, 5, 16, 17])
def test_layer_few_tokens(l):
    """Decode-size token counts: up to 16 tokens the server and the per-pass
    client products stream their uint32 operands (aligned ranks here)."""
    for variant in _variants():
        g, ref, op, m, l = _run_layer(3, (96, 64, 40), (6, 5), m=200, n=256, l=l, variant=variant)
        _check_layer(g, ref, op, m, l)


def test_layer_one_token_example_params():
    """One token through the 64x256x128 shape with Example 3.1 parameters."""
    g, ref, op, m, l = _run_layer(3, (1536, 1024, 652), (80, 80), m=128, n=256, l=1,
                                  variant=M_().GEMM_AUTO)
    _check_layer(g, ref, op, m, l)


@pytest.mark.parametrize("r,t", [((98, 70, 37), (8, 4)), ((96, 64, 40), (16, 12)),
                                 ((1536, 1024, 652), (80, 80)), ((1568, 1544, 96), (12, 20)),
                                 ((1600, 1560, 96), (12, 20))])
def test_layer_tiled_gather_shapes(r, t):
    """Hamming weights that are multiples of 4 take the tiled gather: ragged
    row tiles (m = 131, l = 67), segments that are not multiples of 32, a
    segment offset that is not 16-byte aligned (r_1 = 98), the longest
    segment it stages (1536 words, from prepared tile images for Init X and
    per-call images of Q for the unmask) and longer ones (1544-1600) that fall
    back to the row-staged gather."""
    for variant in _variants():
        g, ref, op, m, l = _run_layer(3, r, t, m=131, n=300, l=67, variant=variant)
        _check_layer(g, ref, op, m, l)


@pytest.mark.parametrize("l", [40, 3])
def test_unmask_clamps_out_of_range_positions(l):
    """Caller-supplied S positions at or beyond r_i are read as r_i - 1 (no
    read leaves the staged segment): the unmask with positions 2^32 - 1 gives
    the same Y_hat as with positions r_i - 1 (tiled gather at 40 tokens, the
    few-rows gather at 3)."""
    from paper_2607_29221_gb300 import protocol as PR
    M = M_()
    gp, op = _params(3, (96, 64, 40), (8, 4))
    proto = PR.Protocol(KEY, gp, variant=M.GEMM_AUTO)
    m, n = 70, 128
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, dev(wl.weights(m, n, std=1.0)), 9, ch)
    mp = layer.init_x(l, 3)
    Xp, s_x, Xpl = layer.mask_input(dev(wl.activations(l, n)), mp)
    Z = layer.server(Xp, Xpl)
    rng = np.random.default_rng(5)
    base = layer.S_idx.clone()
    levels = ((96, 8), (64, 4))
    hits = [torch.from_numpy(rng.random(m * ti) < 0.2).cuda() for _, ti in levels]
    outs = []
    for fill in ("huge", "last"):
        idx = base.clone()
        off = 0
        for (ri, ti), hit in zip(levels, hits):
            blk = idx[off:off + m * ti]
            blk[hit] = -1 if fill == "huge" else ri - 1
            off += m * ti
        layer.S_idx = idx
        Yhat = torch.empty(l, m, dtype=torch.int32, device="cuda")
        layer.unmask(Z, mp, s_x, Yhat=Yhat)
        M.mosaic_device_status()
        outs.append(host_u32(Yhat))
    layer.S_idx = base
    assert np.array_equal(outs[0], outs[1])


@pytest.mark.parametrize("d,r,t,l", [(3, (96, 64, 40), (6, 5), 21), (3, (96, 64, 40), (8, 4), 3),
                                     (2, (100, 70), (9,), 67), (3, (1536, 1024, 652), (80, 80), 64)])
def test_layer_lwe_only_activation_mask(d, r, t, l):
    """act_nested = 0 (Sec. 5.2: the recursive LPN part of the activation mask
    omitted, U_x = C_1 R + E_x, K = J_1 R at rank r_1): every ring output
    bit-exact, on the tensor-core, streaming (l <= 16) and CUDA-core paths."""
    for variant in _variants():
        g, ref, op, m, l_ = _run_layer(d, r, t, m=131 if r[0] < 1000 else 128,
                                       n=300 if r[0] < 1000 else 256, l=l, variant=variant,
                                       act_nested=False)
        _check_layer(g, ref, op, m, l_)


@pytest.mark.parametrize("l", [5, 64, 300])
def test_cached_planes_match_uncached(l):
    """mosaic_mask_activation_planes / mosaic_unmask_planes (stationary operands
    split once) give exactly what the plain entry points give."""
    from paper_2607_29221_gb300 import protocol as PR
    M = M_()
    if not M.mosaic_gemm_variant_available(M.GEMM_TC):
        pytest.skip("tensor-core variant not available")
    gp, _ = _params(3, (1536, 1024, 652), (80, 80))
    proto = PR.Protocol(KEY, gp, variant=M.GEMM_TC)
    m, n = 384, 1000
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, dev(wl.weights(m, n, std=1.0)), 4, ch, bias=dev(wl.bias(m)))
    assert layer.cj_planes is not None
    outs = []
    for cached in (True, False):
        if not cached:
            layer.cj_planes = layer.L_planes = None
        mp = layer.init_x(l, 9)
        Xp, s_x, Xpl = layer.mask_input(dev(wl.activations(l, n)), mp)
        Z = layer.server(Xp, Xpl)
        Yhat = torch.empty(l, m, dtype=torch.int32, device="cuda")
        Y = layer.unmask(Z, mp, s_x, Yhat=Yhat)
        M.mosaic_device_status()
        outs.append((host_u32(mp.Ux), host_u32(mp.K), host_u32(Yhat), host_f32(Y)))
    for a, b in zip(*outs):
        assert np.array_equal(a, b)


def test_layer_rotation_width_65536():
    """n = 36900 rotates at width 65536 (halves, then the last stage apart):
    every ring output bit-exact, one token and five tokens."""
    for l in (1, 5):
        g, ref, op, m, l_ = _run_layer(3, (96, 64, 40), (8, 4), m=40, n=36900, l=l,
                                       variant=M_().GEMM_AUTO)
        _check_layer(g, ref, op, m, l_)


def test_layer_zero_noise_and_no_bias():
    g, ref, op, m, l = _run_layer(3, (96, 64, 40), (6, 5), m=33, n=64, l=9, sigma=0.0, bias=False)
    _check_layer(g, ref, op, m, l)
    assert np.array_equal(ref["Y_hat"], ref["ws"].W_hat @ ref["X_hat"])


def test_layer_single_64x256x128():
    """The small workload (X 64x256, W 256->128, N(0,1)) with Example 3.1 parameters."""
    g, ref, op, m, l = _run_layer(3, (1536, 1024, 652), (80, 80), m=128, n=256, l=64)
    _check_layer(g, ref, op, m, l)


@pytest.mark.slow
def test_layer_attn_proj_7b_full():
    """Attention projection at 7B shape (X 512x4096, W 4096x4096), full oracle."""
    g, ref, op, m, l = _run_layer(3, (1536, 1024, 652), (80, 80), m=4096, n=4096, l=512,
                                  w_std=0.02, variant=_variants()[-1])
    _check_layer(g, ref, op, m, l)


def test_mask_activation_entry_points_and_device_pass_id():
    """mosaic_mask_activation, _planes and _ex give the same U_x, K; with a
    device pass word the pass is pass_id + *pass_dev, and a CUDA graph
    captured around _ex and mosaic_advance_pass draws passes k, k+1, ... on
    its replays."""
    from paper_2607_29221_gb300 import protocol as PR
    M = M_()
    gp, _ = _params(3, (96, 64, 40), (8, 4))
    proto = PR.Protocol(KEY, gp, variant=M.GEMM_AUTO)
    m, n, l = 200, 256, 48
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, dev(wl.weights(m, n, std=1.0)), 6, ch)
    n_pad = layer.n_pad
    ws = proto.workspace(M.mosaic_workspace_bytes(M.OP_MASK_ACTIVATION, m, n_pad, l, gp))

    def bufs():
        return (torch.empty(l, n_pad, dtype=torch.int32, device="cuda"),
                torch.empty(l, m, dtype=torch.int32, device="cuda"))

    want = {}
    for pid in (40, 41, 42):
        U, K = bufs()
        M.mosaic_mask_activation(gp, proto.key, pid, m, n_pad, l, ch.C, layer.J, U, K, proto.variant, ws)
        want[pid] = (host_u32(U), host_u32(K))
    if layer.cj_planes is not None:
        U, K = bufs()
        M.mosaic_mask_activation_planes(gp, proto.key, 40, m, n_pad, l, ch.C, layer.J, layer.cj_planes, U, K,
                                        proto.variant, ws)
        assert np.array_equal(host_u32(U), want[40][0]) and np.array_equal(host_u32(K), want[40][1])
    ctr = torch.tensor([1], dtype=torch.int64, device="cuda")
    U, K = bufs()
    M.mosaic_mask_activation_ex(gp, proto.key, 40, ctr, m, n_pad, l, ch.C, layer.J, layer.cj_planes, U, K,
                                proto.variant, ws)
    assert np.array_equal(host_u32(U), want[41][0]) and np.array_equal(host_u32(K), want[41][1])
    # graph: replay r draws pass 40 + r
    ctr.zero_()
    U, K = bufs()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        M.mosaic_mask_activation_ex(gp, proto.key, 40, ctr, m, n_pad, l, ch.C, layer.J, layer.cj_planes, U, K,
                                    proto.variant, ws)
        M.mosaic_advance_pass(ctr, 1)
    torch.cuda.synchronize()
    assert int(ctr.item()) == 0          # capturing ran nothing
    for r in range(3):
        g.replay()
        torch.cuda.synchronize()
        assert np.array_equal(host_u32(U), want[40 + r][0]) and np.array_equal(host_u32(K), want[40 + r][1])
    assert int(ctr.item()) == 3
    M.mosaic_device_status()


@pytest.mark.parametrize("n_pad", [16384, 32768])
def test_rotation_and_encode_streamed_rows(n_pad):
    """Rows of 16384 and 32768 whose length is a multiple of 32 run on the
    persistent kernel that fetches each block's next row by TMA: more rows than
    SMs (each block loops over several rows), a row stride above the length,
    and a length below n_pad; rotation alone, and encode with and without the
    mask, digit planes and rotation, all bit-exact."""
    M = M_()
    rows = 330 if n_pad == 16384 else 170
    for n, ldx in ((n_pad, n_pad), (n_pad - 4096, n_pad - 4096 + 64)):
        x = wl.spike_activations(rows, ldx, seed=n + 1)
        x[3, :] = 0.0
        x[5, 17] = np.nan
        words = O.sample_signs(KEY, 13, n_pad)
        y = torch.empty(rows, n_pad, dtype=torch.float32, device="cuda")
        M.mosaic_hadamard(dev(x), ldx, y, rows, n, n_pad, dev(words))
        want = O.fwht_rows(x[:, :n], n_pad, words)
        got = host_f32(y)
        # the NaN row: same NaN positions (payload bits may differ), every other value bit-exact
        assert np.array_equal(np.isnan(got), np.isnan(want)), n
        fin = ~np.isnan(want)
        assert np.array_equal(got.view(np.uint32)[fin], want.view(np.uint32)[fin]), n
        qmax = O.qmax_for(n_pad)
        mask = wl.uniform_u32(17, rows, n_pad)
        for rotate, use_mask, use_planes in ((1, True, True), (1, False, False), (0, True, False)):
            out = torch.empty(rows, n_pad, dtype=torch.int32, device="cuda")
            sc = torch.empty(rows, dtype=torch.float32, device="cuda")
            planes = torch.empty(4, rows, n_pad, dtype=torch.int16, device="cuda") if use_planes else None
            M.mosaic_encode(dev(x), ldx, rows, n, n_pad, qmax, rotate, dev(words),
                            dev(mask) if use_mask else None, n_pad, out, n_pad, sc, planes)
            if rotate:
                v = want
            else:
                v = np.zeros((rows, n_pad), np.float32); v[:, :n] = x[:, :n]
            code, scale = O.encode_rows(v, qmax)
            got = host_u32(out)
            assert np.array_equal(got, code + mask if use_mask else code), (n, rotate, use_mask)
            gs = host_f32(sc)
            assert np.array_equal(np.isnan(gs), np.isnan(scale))
            assert np.array_equal(gs[~np.isnan(gs)], scale[~np.isnan(scale)])
            if use_planes:
                pl = host_f32(planes.view(torch.bfloat16).float()).astype(np.int64)
                rebuilt = sum(pl[i] << (8 * i) for i in range(4)) % (1 << 32)
                assert np.array_equal(rebuilt.astype(np.uint32), got)
    M.mosaic_device_status()
