"""Pins of the CPU oracle against facts fixed outside it: an independent ChaCha20
implementation, closed forms of the Hadamard matrix and the discrete Gaussian,
brute-force ring arithmetic, and the algebraic identities of the protocol
(Sec. 3.1 eq. approx-error, Sec. 3.2 unmask derivation, Sec. 4 eq.
had-product-preserved, Thm 3.2, Table tab:lpn-tradeoff)."""
import math

import dataclasses

import numpy as np
import pytest

import oracle as O
from paper_2607_29221_gb300 import workloads as wl

KEY = wl.mask_key()


# --------------------------------------------------------------------------
# PRG
# --------------------------------------------------------------------------
def test_chacha20_matches_independent_implementation():
    """Block function vs the `cryptography` package's ChaCha20 (RFC 8439, 20 rounds)."""
    cg = pytest.importorskip("cryptography.hazmat.primitives.ciphers")
    algorithms = pytest.importorskip("cryptography.hazmat.primitives.ciphers.algorithms")
    key_bytes = KEY.astype("<u4").tobytes()
    for counter, nonce in [(0, (0, 0, 0)), (1, (9, 0x4a, 0)), (12345, (0x105, 7, 0xdeadbeef)),
                           (2**32 - 1, (0xffffffff, 0xffffffff, 0xffffffff))]:
        nonce16 = np.array([counter, *nonce], dtype="<u4").tobytes()
        enc = cg.Cipher(algorithms.ChaCha20(key_bytes, nonce16), mode=None).encryptor()
        ks = np.frombuffer(enc.update(bytes(64)), dtype="<u4")
        got = O.chacha_block(KEY, counter, np.array(nonce, np.uint32))
        assert np.array_equal(got, ks), (counter, nonce)


def test_prg_word_layout_and_streams():
    """Word w is word w mod 16 of block w // 16; (tag, stream id) select the nonce."""
    tg, sid = O.tag(O.KIND_R), 0x1_0000_0002
    w = O.prg_words(KEY, tg, sid, 0, 80)
    nonce = np.array([tg, sid & 0xffffffff, sid >> 32], np.uint32)
    for b in range(5):
        assert np.array_equal(w[16 * b:16 * b + 16], O.chacha_block(KEY, b, nonce))
    assert np.array_equal(O.prg_words(KEY, tg, sid, 37, 20), w[37:57])
    assert not np.array_equal(O.prg_words(KEY, tg, sid + 1, 0, 16), w[:16])
    assert not np.array_equal(O.prg_words(KEY, O.tag(O.KIND_R, 1), sid, 0, 16), w[:16])


def test_uniform_words_are_uniform():
    from scipy import stats
    u = O.sample_uniform(KEY, O.tag(O.KIND_L), 5, 512, 512)
    byt = u.view(np.uint8).ravel()
    counts = np.bincount(byt, minlength=256)
    assert stats.chisquare(counts).pvalue > 1e-4


# --------------------------------------------------------------------------
# Discrete Gaussian
# --------------------------------------------------------------------------
def _gauss_probs(sigma, B):
    w = np.array([math.exp(-k * k / (2 * sigma * sigma)) for k in range(-B, B + 1)])
    return w / w.sum()


@pytest.mark.parametrize("sigma", [0.5, 1.0, 2.0])
def test_gaussian_table_matches_closed_form(sigma):
    t = O.gaussian_table(sigma)
    B = O.gaussian_bound(sigma)
    assert B == math.ceil(12 * sigma) and len(t) == 2 * B + 1
    assert np.all(np.diff(t.astype(object)) >= 0)
    assert int(t[-1]) == 2**64 - 1
    p = _gauss_probs(sigma, B)
    cdf = np.cumsum(p)
    got = t.astype(np.float64) / 2.0**64
    assert np.allclose(got, np.minimum(cdf, 1.0), rtol=1e-12, atol=2.0**-60)


def test_gaussian_sigma_half_frequencies():
    """sigma = 0.5 (Example 3.1): P(0) = 0.78657, P(+-1) = 0.10645, P(+-2) = 2.6387e-4,
    variance 0.21501 (parameter semantics exp(-k^2/2sigma^2), Sec. 3.1)."""
    from scipy import stats
    n = 2_000_000
    s = O.sample_gaussian(KEY, O.tag(O.KIND_EW), 1, n, 0.5).view(np.int32)
    p = _gauss_probs(0.5, 6)
    assert abs(p[6] - 0.78657) < 1e-5 and abs(p[7] - 0.10645) < 1e-5 and abs(p[8] - 2.6387e-4) < 1e-8
    vals, counts = np.unique(s, return_counts=True)
    assert set(vals.tolist()) <= {-3, -2, -1, 0, 1, 2, 3}
    obs = np.array([np.sum(s == k) for k in (-2, -1, 0, 1, 2)], dtype=np.float64)
    obs[0] += np.sum(s <= -3); obs[-1] += np.sum(s >= 3)
    exp = p[4:9].copy(); exp[0] += p[:4].sum(); exp[-1] += p[9:].sum()
    assert stats.chisquare(obs, exp * n).pvalue > 1e-4
    var_exact = float(np.sum(p * np.arange(-6, 7) ** 2))
    assert abs(var_exact - 0.21501) < 1e-5
    se = math.sqrt(np.sum(p * np.arange(-6, 7) ** 4) / n)
    assert abs(np.mean(s.astype(np.float64) ** 2) - var_exact) < 4 * se
    assert abs(np.mean(s)) < 4 * math.sqrt(var_exact / n)


def test_gaussian_zero_sigma_is_zero():
    assert not np.any(O.sample_gaussian(KEY, O.tag(O.KIND_EX), 3, 1000, 0.0))


# --------------------------------------------------------------------------
# Sparse LPN rows
# --------------------------------------------------------------------------
def test_sparse_rows_exact_weight_and_uniform_positions():
    from scipy import stats
    r, t, rows = 1024, 80, 2000
    idx, val = O.sample_sparse(KEY, O.tag(O.KIND_S, 2), 9, rows, r, t)
    assert idx.max() < r
    for j in range(rows):
        assert len(set(idx[j].tolist())) == t
    assert np.all(val != 0)
    counts = np.bincount(idx.ravel(), minlength=r)
    assert stats.chisquare(counts).pvalue > 1e-4
    # Window layout: row j starts at stream word j * 65536.
    w = O.prg_words(KEY, O.tag(O.KIND_S, 2), 9, 3 * 65536, 1)
    assert idx[3, 0] == (int(w[0]) * r) >> 32


# --------------------------------------------------------------------------
# Hadamard rotation
# --------------------------------------------------------------------------
def _sylvester(n):
    H = np.ones((1, 1))
    while H.shape[0] < n:
        H = np.block([[H, H], [H, -H]])
    return H


@pytest.mark.parametrize("n", [2, 8, 64, 256, 1024])
def test_fwht_is_sylvester_hadamard(n):
    """Rows of R = H D on the identity give the explicit Sylvester matrix / sqrt(n)."""
    words = O.sample_signs(KEY, 77, n)
    d = O.signs_to_pm1(words, n)
    H = _sylvester(n)
    eye = np.eye(n)
    got = O.fwht_rows_f64(eye, words)                      # row i = H D e_i = d_i H[:, i]
    assert np.allclose(got, (H * d[None, :]).T / math.sqrt(n), atol=1e-15)
    # Unnormalised transform is exact on integers: H H^T = n I.
    unnorm = O.fwht_rows_f64(H, None) * math.sqrt(n)
    assert np.array_equal(np.rint(unnorm), n * np.eye(n))
    # fp32 path agrees with fp64 to rounding.
    x = wl.activations(4, n)
    y32 = O.fwht_rows(x, n, words).astype(np.float64)
    y64 = O.fwht_rows_f64(x.astype(np.float64), words)
    assert np.allclose(y32, y64, rtol=0, atol=1e-5 * np.abs(x).max() * math.log2(n) + 1e-7)


def test_fwht_orthogonal_norm_and_spike():
    """R^T R = I (Sec. 4), norm preservation, ||R e_1||_inf = 1/sqrt(n) (App. error-post-rot)."""
    n = 4096
    words = O.sample_signs(KEY, 3, n)
    x = wl.activations(8, n).astype(np.float64)
    y = O.fwht_rows_f64(x, words)
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), rtol=1e-12)
    e1 = np.zeros((1, n), np.float32); e1[0, 0] = 1.0
    r = O.fwht_rows(e1, n, words)
    assert np.max(np.abs(r)) == np.float32(1.0 / math.sqrt(n))
    y32 = O.fwht_rows(x.astype(np.float32), n, words)
    assert np.allclose(np.linalg.norm(y32, axis=1), np.linalg.norm(x, axis=1), rtol=1e-6)


def test_rotation_preserves_product_and_spreads_outliers():
    """(W R^T)(R X) = W X (eq. had-product-preserved) and ||R x||_inf ~ ||x||_2 sqrt(log n / n)."""
    n, m, l = 512, 16, 8
    words = O.sample_signs(KEY, 4, n)
    W = wl.weights(m, n).astype(np.float64)
    X = wl.spike_activations(l, n).astype(np.float64)       # l x n, outlier channels
    Wr = O.fwht_rows_f64(W, words)
    Xr = O.fwht_rows_f64(X, words)
    assert np.allclose(Wr @ Xr.T, W @ X.T, rtol=1e-10, atol=1e-10)
    ratio_before = np.abs(X).max(axis=1) / np.linalg.norm(X, axis=1)
    ratio_after = np.abs(Xr).max(axis=1) / np.linalg.norm(Xr, axis=1)
    assert np.all(ratio_before > 0.4)
    assert np.all(ratio_after < 3.0 * math.sqrt(math.log(n) / n))


def test_fwht_zero_padding():
    n, n_pad = 14336, 16384
    words = O.sample_signs(KEY, 5, n_pad)
    x = wl.activations(2, n)
    xp = np.zeros((2, n_pad), np.float32); xp[:, :n] = x
    assert np.array_equal(O.fwht_rows(x, n_pad, words), O.fwht_rows(xp, n_pad, words))


# --------------------------------------------------------------------------
# Quantisation
# --------------------------------------------------------------------------
def test_qmax_window():
    """n_pad q_max^2 <= 2^31 (Sec. 4, kappa = 32), the largest such q."""
    want = {256: 2896, 4096: 724, 8192: 512, 16384: 362, 32768: 256}
    for n_pad, q in want.items():
        assert O.qmax_for(n_pad) == q
        assert n_pad * q * q <= 2**31 < n_pad * (q + 1) ** 2
    assert O.qmax_for(2) == 2**15 - 1


def test_encode_rounding_and_edges():
    v = np.array([[4.0, 2.5, 3.5, -2.5, -0.5, 0.5, 1.5, 0.0],
                  [0.0] * 8,
                  [1.0, np.inf, 0, 0, 0, 0, 0, 0],
                  [-3.0, 1.0, 0, 0, 0, 0, 0, 0]], np.float32)
    code, scale = O.encode_rows(v, 4)
    c = code.view(np.int32)
    assert scale[0] == 1.0
    assert c[0].tolist() == [4, 2, 4, -2, 0, 0, 2, 0]        # ties to even
    assert scale[1] == 0.0 and not c[1].any()
    assert np.isnan(scale[2]) and not c[2].any()
    assert scale[3] == np.float32(0.75) and c[3, 0] == -4
    x = wl.activations(16, 1024)
    code, s = O.encode_rows(x, 724)
    q = code.view(np.int32)
    assert np.abs(q).max() == 724 and np.all(np.abs(q).max(axis=1) == 724)
    assert np.all(np.abs(q * s[:, None] - x) <= s[:, None] * (0.5 + 1e-6))


# --------------------------------------------------------------------------
# Ring arithmetic
# --------------------------------------------------------------------------
def test_ring_matmul_bruteforce():
    rng = np.random.Generator(np.random.PCG64(0))
    for (M, K, N) in [(1, 1, 1), (3, 5, 2), (8, 8, 8), (7, 3, 6)]:
        A = rng.integers(0, 2**32, (M, K), dtype=np.uint64).astype(np.uint32)
        B = rng.integers(0, 2**32, (K, N), dtype=np.uint64).astype(np.uint32)
        A[0, :] = 0xFFFFFFFF; B[:, 0] = 0xFFFFFFFF
        want = (A.astype(object) @ B.astype(object)) % (2**32)
        assert np.array_equal(O.matmul(A, B).astype(object), want)
    one = np.array([[2**32 - 1, 3]], np.uint32)
    two = np.array([[2**32 - 1], [5]], np.uint32)
    assert O.matmul(one, two)[0, 0] == 16


def test_ring_matmul_vs_numpy_wrap():
    A = wl.uniform_u32(1, 67, 300)
    B = wl.uniform_u32(2, 300, 45)
    assert np.array_equal(O.matmul(A, B), A @ B)


def test_sparse_products_vs_dense():
    rng = np.random.Generator(np.random.PCG64(1))
    r, l, rows, t = 96, 10, 20, 7
    idx, val = O.sample_sparse(KEY, O.tag(O.KIND_S, 2), 1, rows, r, t)
    Sd = np.zeros((rows, r), np.uint32)
    for j in range(rows):
        Sd[j, idx[j]] = val[j]
    Q = rng.integers(0, 2**32, (r, l), dtype=np.uint64).astype(np.uint32)
    assert np.array_equal(O.sparse_rows_matmul((idx, val), Q), Sd @ Q)
    idx2, val2 = O.sample_sparse(KEY, O.tag(O.KIND_T, 2), 1, l, r, t)
    Td = np.zeros((r, l), np.uint32)
    for k in range(l):
        Td[idx2[k], k] = val2[k]
    A = rng.integers(0, 2**32, (rows, r), dtype=np.uint64).astype(np.uint32)
    assert np.array_equal(O.matmul_sparse_cols(A, (idx2, val2)), A @ Td)


# --------------------------------------------------------------------------
# Protocol identities
# --------------------------------------------------------------------------
SMALL = O.Params(d=3, r=(96, 64, 40), t=(6, 5))


def _run(p, m=24, n=48, l=10, sigma=None, x_zero=False, seed_off=0):
    if sigma is not None:
        p = dataclasses.replace(p, sigma=sigma)
    W = wl.weights(m, n, seed=wl.SEED_W + seed_off, std=1.0)
    X = wl.activations(l, n, seed=wl.SEED_X + seed_off).T.copy()
    if x_zero:
        X[:] = 0
    return p, O.secure_linear(KEY, p, W, X, matrix_id=3 + seed_off, pass_id=17 + seed_off), W, X


@pytest.mark.parametrize("act_nested", [True, False])
@pytest.mark.parametrize("d", [1, 2, 3])
def test_zero_noise_protocol_is_exact(d, act_nested):
    """sigma = 0: Y_hat = W_hat X_hat exactly (the INT16-rot-sigma=0 case, Sec. 4.3),
    with the nested activation mask and with the LWE-only one of Sec. 5.2."""
    p = O.Params(d=d, r=SMALL.r[:d], t=SMALL.t[: d - 1], sigma=0.0, act_nested=act_nested)
    _, r, _, _ = _run(p)
    assert np.array_equal(r["Y_hat"], r["ws"].W_hat @ r["X_hat"])


@pytest.mark.parametrize("act_nested", [True, False])
@pytest.mark.parametrize("d", [1, 2, 3])
def test_noise_identity(d, act_nested):
    """Y_hat - W_hat X_hat = W_hat E_x + E_w X_hat + E_w E_x (mod 2^32), eq. approx-error
    and the Sec. 3.2 unmask derivation, with the E's re-read from the sampled state."""
    p = O.Params(d=d, r=SMALL.r[:d], t=SMALL.t[: d - 1], sigma=1.0, act_nested=act_nested)
    _, r, _, _ = _run(p, seed_off=d)
    Wh, Xh, Ew, Ex = r["ws"].W_hat, r["X_hat"], r["ws"].E_w, r["ps"].E_x
    assert np.any(Ew) and np.any(Ex)
    lhs = r["Y_hat"] - Wh @ Xh
    rhs = Wh @ Ex + Ew @ Xh + Ew @ Ex
    assert np.array_equal(lhs, rhs)


def test_depth_one_matches_simple_protocol():
    """d = 1 reduces to Sec. 3.1: Y ~ Y' - L M (X + E_x) - (W' N) R (eq. approx-error)."""
    p = O.Params(d=1, r=(96,), t=(), sigma=0.5)
    _, r, _, _ = _run(p)
    ws, ps = r["ws"], r["ps"]
    Mm = r["P"][0]                       # M = M_1 (public)
    Nn = r["C"][0]                       # N = N_1 (public)
    simple = r["Y_masked"] - ws.L @ (Mm @ (r["X_hat"] + ps.E_x)) - (ws.W_masked @ Nn) @ ps.R
    assert np.array_equal(simple, r["Y_hat"])


def _sparse_dense(S, rows, r):
    """(idx, val), rows x t with distinct positions per row -> dense rows x r."""
    idx, val = S
    D = np.zeros((rows, r), np.uint32)
    np.put_along_axis(D, idx.astype(np.int64), val, axis=1)
    return D


def _rank_gf2(A):
    """Rank over GF(2) of the low bits of A (rows as Python integers)."""
    rows = [int("".join("1" if b else "0" for b in row) or "0", 2) for row in (A & 1).astype(bool)]
    rank = 0
    while rows:
        piv = max(rows)
        if piv == 0:
            break
        rows.remove(piv)
        top = piv.bit_length() - 1
        rows = [x ^ piv if (x >> top) & 1 else x for x in rows]
        rank += 1
    return rank


@pytest.mark.parametrize("act_nested", [True, False])
@pytest.mark.parametrize("d", [1, 2, 3])
def test_masks_follow_the_nested_substitution_form(d, act_nested):
    """The masks against the nested form they come from, evaluated inside out from the
    sampled M_i, N_i (not from the oracle's chain products):
      eq. weight-mask, first line: U_w - E_w = (((L M_d + S_d) M_{d-1} + S_{d-1}) ... + S_2) M_1;
      eq. activation-mask:         U_x - E_x = N_1 (T_2 + N_2 (T_3 + ... N_d R))
                                   (N_1 R with the LWE-only activation mask of Sec. 5.2);
      Init X 1c with J_i = (W_hat + E_w) N_1 ... N_i:  K = (W_hat + E_w)(U_x - E_x).
    A dropped LPN term, a term at the wrong level or a missing E fails here even when
    the unmask drops the same term (which the noise identity cannot see)."""
    p = O.Params(d=d, r=SMALL.r[:d], t=SMALL.t[: d - 1], sigma=1.0, act_nested=act_nested)
    m, n, l = 40, 100, 12
    _, r, _, _ = _run(p, m=m, n=n, l=l, seed_off=10 + d)
    ws, ps, n_pad = r["ws"], r["ps"], r["n_pad"]
    rk = p.ranks(n_pad)
    Ms = [O.sample_uniform(KEY, O.tag(O.KIND_M, i), n_pad, rk[i], rk[i - 1]) for i in range(1, d + 1)]
    Ns = [O.sample_uniform(KEY, O.tag(O.KIND_N, i), n_pad, rk[i - 1], rk[i]) for i in range(1, d + 1)]
    acc = ws.L
    for i in range(d, 0, -1):                       # level i: acc <- acc M_i (+ S_i below level 1)
        acc = acc @ Ms[i - 1]
        if i > 1:
            acc = acc + _sparse_dense(ws.S[i], m, rk[i - 1])
    assert np.array_equal(ws.W_masked - ws.W_hat - ws.E_w, acc)
    if act_nested:
        acc = ps.R
        for i in range(d, 0, -1):                   # acc <- N_i (acc + T_{i+1})
            if i < d:
                acc = acc + _sparse_dense(ps.T[i + 1], l, rk[i]).T
            acc = Ns[i - 1] @ acc
    else:
        acc = Ns[0] @ ps.R
    Ux_noiseless = ps.U_x - ps.E_x
    assert np.array_equal(Ux_noiseless, acc)
    assert np.array_equal(ps.K, (ws.W_hat + ws.E_w) @ Ux_noiseless)


def test_weight_mask_rank_mod_2():
    """Rank facts of eq. weight-mask: every term has row space inside that of M_1, so
    rank(U_w - E_w) <= r_1; without the sparse LPN terms it would be <= r_d, and with
    them (d >= 2) it exceeds r_d.  Checked over GF(2) on a 256 x 256 case."""
    for d, r, t in ((3, (96, 64, 40), (6, 5)), (2, (96, 40), (6,)), (1, (96,), ())):
        p = O.Params(d=d, r=r, t=t, sigma=1.0)
        _, res, _, _ = _run(p, m=256, n=256, l=4, seed_off=20 + d)
        ws = res["ws"]
        rank = _rank_gf2(ws.W_masked - ws.W_hat - ws.E_w)
        assert rank <= r[0]
        if d >= 2:
            assert rank > r[-1]


def test_masked_input_is_uniform_when_x_is_zero():
    from scipy import stats
    p = O.Params(d=3, r=(96, 64, 40), t=(6, 5), sigma=0.5)
    _, r, _, _ = _run(p, m=8, n=256, l=64, x_zero=True)
    byt = r["X_masked"].view(np.uint8).ravel()
    assert stats.chisquare(np.bincount(byt, minlength=256)).pvalue > 1e-4


def test_noise_tail_bound_thm_3_2():
    """Fraction of entries with |noise| > c sigma sqrt(||x_k||^2 + ||w_j||^2) is <= 2 exp(-c^2/2)."""
    p = O.Params(d=3, r=SMALL.r, t=SMALL.t, sigma=0.5)
    _, r, _, _ = _run(p, m=64, n=256, l=32)
    noise = (r["Y_hat"] - r["ws"].W_hat @ r["X_hat"]).view(np.int32).astype(np.float64)
    wn = np.sum(r["ws"].W_hat.view(np.int32).astype(np.float64) ** 2, axis=1)
    xn = np.sum(r["X_hat"].view(np.int32).astype(np.float64) ** 2, axis=0)
    scale = p.sigma * np.sqrt(wn[:, None] + xn[None, :])
    for c in (2.0, 3.0, 4.0):
        assert np.mean(np.abs(noise) > c * scale) <= 2 * math.exp(-c * c / 2)


def test_decode_zero_noise_close_to_float_product():
    """sigma = 0: the decoded product differs from fp64 W X by quantisation error only."""
    p = O.Params(d=3, r=SMALL.r, t=SMALL.t, sigma=0.0)
    _, r, W, X = _run(p, m=32, n=256, l=16)
    ref = W.astype(np.float64) @ X.astype(np.float64)
    s_w, s_x, q = r["ws"].s_w.astype(np.float64), r["s_x"].astype(np.float64), r["ws"].qmax
    # |err| <= s_w s_x (0.5 (||x_hat||_1 + ||w_hat||_1) + 0.25 n) + float rounding
    wh = np.abs(r["ws"].W_hat.view(np.int32)).sum(axis=1).astype(np.float64)
    xh = np.abs(r["X_hat"].view(np.int32)).sum(axis=0).astype(np.float64)
    bound = s_w[:, None] * s_x[None, :] * (0.5 * (wh[:, None] + xh[None, :]) + 0.25 * 256)
    assert np.all(np.abs(r["Y"] - ref) <= bound * 1.001 + 1e-6 * np.abs(ref))
    assert np.linalg.norm(r["Y"] - ref) / np.linalg.norm(ref) < 2e-3


def test_client_state_matches_tradeoff_table():
    """Client state of the nested protocol: (m+n)(r_1+..+r_d) + m r_d words
    (Table tab:lpn-tradeoff: 1536(2m+n), 2560(m+n)+1024m, 3212(m+n)+652m) and
    client compute per (m+n) l of r_d + sum t (1536, 1104, 812)."""
    for d, state_c, compute in [(1, None, 1536), (2, None, 1104), (3, None, 812)]:
        p = O.Params(d=d, r=(1536, 1024, 652)[:d], t=(80, 80)[: d - 1])
        m, n_pad = 3, 4
        r = p.ranks(n_pad)
        # C_i = N_1..N_i: n x r_i;  J_i: m x r_i;  L: m x r_d
        words = sum(n_pad * r[i] for i in range(1, d + 1)) + sum(m * r[i] for i in range(1, d + 1)) + m * r[d]
        table = {1: 1536 * (2 * m + n_pad), 2: 2560 * (m + n_pad) + 1024 * m,
                 3: 3212 * (m + n_pad) + 652 * m}[d]
        assert words == table
        assert r[d] + sum(p.t) == compute


def test_oracle_layout_of_init_x():
    """R^T rows are the uniform stream of (R, pass_id); T columns are sparse rows."""
    p = O.Params(d=2, r=(32, 16), t=(3,), sigma=0.5)
    P, C = O.chains(KEY, p, 64)
    ws = O.init_w(KEY, p, wl.weights(8, 64), 1, P, C, 64)
    ps = O.init_x(KEY, p, 5, 2, C, ws.J, 64)
    assert np.array_equal(ps.R.T, O.sample_uniform(KEY, O.tag(O.KIND_R), 2, 5, 16))
    assert np.array_equal(ps.T[2][0], O.sample_sparse(KEY, O.tag(O.KIND_T, 2), 2, 5, 32, 3)[0])


def test_lwe_only_activation_mask_structure():
    """act_nested = False (Sec. 5.2, "Protocol parameterization"): only J_1 is
    kept, no T is drawn and R has r_1 rows; the mask differs from the nested
    one drawn from the same key (the identities above pin its arithmetic)."""
    p = O.Params(d=3, r=(12, 8, 5), t=(3, 2), sigma=0.5, act_nested=False)
    _, r, _, _ = _run(p, m=6, n=16, l=9)
    ws, ps = r["ws"], r["ps"]
    assert len(ws.J) == 1 and ps.T == {} and ps.R.shape == (12, 9)
    _, rn, _, _ = _run(dataclasses.replace(p, act_nested=True), m=6, n=16, l=9)
    assert len(rn["ws"].J) == 3 and rn["ps"].R.shape == (5, 9)
    assert not np.array_equal(rn["ps"].U_x, ps.U_x)
    assert np.array_equal(rn["ws"].J[0], ws.J[0])


# --------------------------------------------------------------------------
# Freivalds integrity check (Init W 4, Online 4; "Computational integrity")
# --------------------------------------------------------------------------
def test_freivalds_accepts_honest_and_flags_corruption():
    """An honest Y' = W' X' passes for every vector (associativity of the ring
    product); an odd error in one entry of column j is caught by every vector
    with a_v[i] != 0 at that row (a_v[i] * e = 0 mod 2^32 needs a_v[i] = 0),
    and an error 2^31 exactly by the vectors whose a_v[i] is odd."""
    p = O.Params(d=3, r=SMALL.r, t=SMALL.t, sigma=0.5)
    _, r, _, _ = _run(p, m=20, n=48, l=9)
    ws = r["ws"]
    a, Yc = O.freivalds_setup(KEY, p, ws, 3, 6)
    assert a.shape == (6, 20) and Yc.shape == (6, 64)
    assert np.array_equal(a, O.sample_uniform(KEY, O.tag(O.KIND_CHECK), 3, 6, 20))
    Yp, Xp = r["Y_masked"], r["X_masked"]
    assert not np.any(O.freivalds_check(a, Yc, Yp, Xp))
    bad = Yp.copy()
    bad[7, 4] = np.uint32((int(bad[7, 4]) + 12345) % 2**32)   # odd error at row 7, token 4
    got = O.freivalds_check(a, Yc, bad, Xp)
    assert got[4] == np.count_nonzero(a[:, 7]) and got[4] == 6
    assert np.count_nonzero(got) == 1
    bad = Yp.copy()
    bad[2, 1] = np.uint32((int(bad[2, 1]) + 2**31) % 2**32)
    got = O.freivalds_check(a, Yc, bad, Xp)
    assert got[1] == int(np.sum(a[:, 2] & 1)) and np.count_nonzero(got) == (1 if got[1] else 0)


def test_freivalds_check_vectors_on_a_bruteforce_case():
    """Tiny case against Python integers: a^T (W' X') and (a^T W') X' mod 2^32."""
    rng = np.random.default_rng(9)
    W = rng.integers(0, 2**32, (3, 4), dtype=np.uint64).astype(np.uint32)
    X = rng.integers(0, 2**32, (4, 2), dtype=np.uint64).astype(np.uint32)
    a = rng.integers(0, 2**32, (2, 3), dtype=np.uint64).astype(np.uint32)
    Y = O.matmul(W, X)
    for v in range(2):
        for j in range(2):
            lhs = sum(int(a[v, i]) * sum(int(W[i, c]) * int(X[c, j]) for c in range(4)) for i in range(3))
            assert (lhs % 2**32) == int(O.matmul(a, Y)[v, j])
            rhs = sum(sum(int(a[v, i]) * int(W[i, c]) for i in range(3)) * int(X[c, j]) for c in range(4))
            assert (rhs % 2**32) == int(O.matmul(O.matmul(a, W), X)[v, j])
