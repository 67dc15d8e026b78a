"""Parity at the full sizes of the paper-shaped workloads, in the launch
configuration the benchmark uses (tensor-core variant, Example 3.1
parameters): the FFN up/down projections at 7B shape, every linear of one
70B decoder layer at 2048 tokens, and the 70B decode sweep (1 to 256 tokens).
The GPU runs each secure linear call in full; the oracle recomputes the public
chains in full and every other output at sampled weight rows and tokens
(``oracle.sampled``), and they must agree bit-exactly; decoded floats within
1e-6 x (|Y_hat s_w s_x| + |b|).  The sampled rows include both sides of
128-row tile edges spread over the whole matrix and the last tile; the sampled
tokens both sides of 128-token tile edges.

Every entry of the server output Z = X' [W'; P]^T is covered as well, by a
host-side Freivalds check over Z_{2^32} (numpy uint32 arithmetic, nothing from
the GPU's arithmetic): for four random vectors a, Z a = X' ([W'; P]^T a) on the
GPU's own X' and [W'; P], which the sampled comparisons pin to the oracle.  A
wrong entry e escapes one vector with probability at most 2^-(32 - v), v the
trailing zero bits of e."""
import numpy as np
import pytest

import oracle as O
from oracle import sampled as OS
from paper_2607_29221_gb300 import workloads as wl

torch = pytest.importorskip("torch")
pytestmark = [pytest.mark.gpu, pytest.mark.slow]

KEY = wl.mask_key()
_CHAINS = {}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_29221_gb300 import build
    build.build()
    yield
    _CHAINS.clear()


def _proto():
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    return PR.Protocol(KEY, M.default_params(), variant=M.GEMM_AUTO)


def _chains(proto, n_pad):
    """GPU chains checked in full against the oracle's, once per width."""
    from paper_2607_29221_gb300 import protocol as PR
    if n_pad not in _CHAINS:
        ch = PR.Chains(proto, n_pad)
        P, C = O.chains(KEY, O.Params(), n_pad)
        Pf, Cf = np.vstack(P), np.hstack(C)
        torch.cuda.synchronize()
        assert np.array_equal(ch.P.cpu().numpy().view(np.uint32), Pf)
        assert np.array_equal(ch.C.cpu().numpy().view(np.uint32), Cf)
        assert np.array_equal(ch.CT.cpu().numpy().view(np.uint32), Cf.T)
        _CHAINS[n_pad] = (ch, P, C)
    return _CHAINS[n_pad]


def _u32(t):
    return t.cpu().numpy().view(np.uint32)


def _sample_rows(m, edges=24):
    """Rows 0, 1, m/3, m/2 + 7, m - 1, both sides of `edges` 128-row tile edges
    spread evenly over the matrix, and the first row of the last tile."""
    cuts = np.unique(np.linspace(1, max(1, (m - 1) // 128), edges).astype(np.int64)) * 128
    rows = [0, 1, m // 3, m // 2 + 7, m - 1, (m - 1) // 128 * 128]
    rows += [c - 1 for c in cuts] + [c for c in cuts]
    return np.unique(np.clip(np.array(rows), 0, m - 1))


def _sample_tokens(l):
    """Tokens 0, l/2, l - 1 and both sides of every 128-token tile edge."""
    toks = [0, l // 2, l - 1] + [c + d for c in range(128, l, 128) for d in (-1, 0)]
    return np.unique(np.clip(np.array(toks), 0, l - 1))


def _freivalds_host(Wp, Xp, Z, seed, k=4):
    """Z a == X' (Wp^T a) over Z_{2^32} for k random a (numpy uint32, wraps)."""
    N = Z.shape[1]
    Wh, Xh, Zh = _u32(Wp[:N]), _u32(Xp), _u32(Z)
    a = np.random.Generator(np.random.PCG64(seed)).integers(0, 1 << 32, size=(N, k), dtype=np.uint32)
    v = np.zeros((Wh.shape[1], k), np.uint32)          # Wp^T a, accumulated row block by row block
    for s0 in range(0, N, 4096):
        blk = Wh[s0:s0 + 4096]
        for i in range(k):
            v[:, i] += (blk * a[s0:s0 + 4096, i:i + 1]).sum(axis=0, dtype=np.uint32)
    assert np.array_equal(Zh @ a, Xh @ v)


def _check_linear(proto, m, n, ls, matrix_id, w_std=0.02, seed_off=0):
    from paper_2607_29221_gb300 import protocol as PR
    p = O.Params()
    n_pad = PR.pad_width(n)
    ch, P, C = _chains(proto, n_pad)
    W = wl.weights(m, n, seed=wl.SEED_W + seed_off, std=w_std)
    b = wl.bias(m, seed=wl.SEED_B + seed_off)
    layer = PR.SecureLinear(proto, torch.from_numpy(W).cuda(), matrix_id, ch, torch.from_numpy(b).cuda())
    rows = _sample_rows(m)
    wr = OS.weight_rows(KEY, p, W[rows], rows, matrix_id, P, C, n_pad)
    rows_t = torch.from_numpy(rows).cuda()
    torch.cuda.synchronize()
    assert np.array_equal(_u32(layer.sign_words), wr.sign_words)
    assert np.array_equal(layer.s_w[rows_t].cpu().numpy(), wr.s_w)
    assert np.array_equal(_u32(layer.Wp[rows_t]), wr.W_masked)
    assert np.array_equal(_u32(layer.L[rows_t]), wr.L)
    assert np.array_equal(_u32(layer.J[rows_t]), np.hstack(wr.J))
    off = 0
    for i in range(1, p.d):
        t = p.t[i - 1]
        Si = layer.S_idx[off:off + m * t].view(m, t)[rows_t]
        Sv = layer.S_val[off:off + m * t].view(m, t)[rows_t]
        assert np.array_equal(_u32(Si), wr.S[i + 1][0]) and np.array_equal(_u32(Sv), wr.S[i + 1][1])
        off += m * t
    for l in ls:
        pass_id = 7000 + 10 * matrix_id + l
        X_tm = wl.activations(l, n, seed=wl.SEED_X + l + seed_off)
        mp = layer.init_x(l, pass_id)
        Xp, s_x, Xpl = layer.mask_input(torch.from_numpy(X_tm).cuda(), mp)
        Z = layer.server(Xp, Xpl)
        Yhat = torch.empty(l, m, dtype=torch.int32, device="cuda")
        Y = layer.unmask(Z, mp, s_x, Yhat=Yhat)
        toks = _sample_tokens(l)
        tc = OS.token_cols(KEY, p, X_tm[toks], toks, pass_id, wr.sign_words, wr.qmax, C, n_pad)
        K = OS.k_entries(p, wr, tc)
        Ym, Q = OS.server_entries(wr, tc, P)
        Yh = OS.unmask_entries(p, wr, K, Ym, Q)
        Yf = O.decode(Yh, wr.s_w, tc.s_x, b[rows])
        tk = torch.from_numpy(toks).cuda()
        torch.cuda.synchronize()
        assert np.array_equal(_u32(mp.Ux[tk]), tc.U_x.T), (m, n, l)
        assert np.array_equal(_u32(mp.K[tk][:, rows_t]), K.T), (m, n, l)
        assert np.array_equal(_u32(Xp[tk]), tc.X_masked.T), (m, n, l)
        assert np.array_equal(s_x[tk].cpu().numpy(), tc.s_x)
        Zs = _u32(Z[tk])
        assert np.array_equal(Zs[:, rows], Ym.T), (m, n, l)
        assert np.array_equal(Zs[:, m:], np.hstack([q.T for q in Q])), (m, n, l)
        assert np.array_equal(_u32(Yhat[tk][:, rows_t]), Yh.T), (m, n, l)
        _freivalds_host(layer.Wp, Xp, Z, seed=l + m)
        mag = np.abs(Yh.T.view(np.int32) * wr.s_w[None, :].astype(np.float64)
                     * tc.s_x[:, None].astype(np.float64)) + np.abs(b[rows].astype(np.float64))[None, :]
        err = np.abs(Y[tk][:, rows_t].cpu().numpy().astype(np.float64) - Yf.T)
        assert np.all(err <= 1e-6 * mag), (m, n, l)
    from paper_2607_29221_gb300 import mosaic as M
    M.mosaic_device_status()
    del layer
    torch.cuda.empty_cache()


def test_ffn_7b_up_and_down():
    proto = _proto()
    wk = wl.WORKLOADS["ffn_7b_2048x4096x14336"]
    for i, lin in enumerate(wk.linears):
        _check_linear(proto, lin.m, lin.n, [wk.l], matrix_id=20 + i, seed_off=i)


@pytest.mark.parametrize("which", ["qkv", "o", "gate_up", "down"])
def test_decoder_70b_prefill_linear(which):
    proto = _proto()
    wk = wl.WORKLOADS["decoder_70b_prefill_2048"]
    lin = next(x for x in wk.linears if x.name == which)
    _check_linear(proto, lin.m, lin.n, [wk.l], matrix_id=30 + [x.name for x in wk.linears].index(which),
                  seed_off=3)


def test_decode_sweep_70b():
    proto = _proto()
    wk = wl.WORKLOADS["decode_70b_sweep"]
    for i, lin in enumerate(wk.linears):
        ls = list(wk.decode_batches) if lin.name == "o" else [1, 256]
        _check_linear(proto, lin.m, lin.n, ls, matrix_id=40 + i, seed_off=5 + i)
