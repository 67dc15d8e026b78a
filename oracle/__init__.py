"""MOSAIC oracle: plain, slow, obviously correct CPU reference of the masked
ring-matmul path.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
benchmark's ``cpu_baseline`` / ``--impl reference`` legs may import this
package.  The product (``paper_2607_29221_gb300``) never imports it, and it
never imports the product.  The two share only the seeded inputs of
``paper_2607_29221_gb300.workloads`` (a module with none of the method's
arithmetic).

Everything here follows the paper's notation and orientation: W is m x n,
X is n x l, Y = W X is m x l (the CUDA path stores the transposes).  The heavy
loops live in ``mosaic_oracle.c``; this file composes them step by step in the
order of the protocol boxes:

* ``chains``      -- public M_i, N_i and their products (Sec. 3.2 box, Init W 1-3, 5)
* ``init_w``      -- Pi_Sec-Linear Init W + Pi_Sec-Approx-MatMul Init W
* ``init_x``      -- Pi_Sec-Approx-MatMul Init X (steps 1a-1c)
* ``mask_input``  -- Pi_Sec-Linear Online step 1 and Approx-MatMul Online step 2
* ``server``      -- Approx-MatMul Online step 3 (Y' = W'X', Q_i = P_i X')
* ``unmask``      -- Approx-MatMul Online step 5
* ``decode``      -- Pi_Sec-Linear Online step 3 (fp64)
* ``freivalds_*`` -- Approx-MatMul Init W step 4 and Online step 4 (integrity check)

Parity status: every function is pinned by ``tests/test_oracle_pins.py``
except the PRG stream layout and the sampler details (which words feed which
element), which are this build's own definitions: "parity unpinned" for those
layout choices -- GPU-vs-oracle agreement is their only check.  The ChaCha20
block itself is pinned to an independent implementation.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass
from decimal import Decimal, localcontext

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mosaic_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libmosaic_oracle.so")

# ---------------------------------------------------------------------------
# Stream tags (this build's PRG layout: kind in the low byte, level i above it)
# ---------------------------------------------------------------------------
KIND_M, KIND_N, KIND_L, KIND_S, KIND_EW, KIND_R, KIND_T, KIND_EX, KIND_SIGN, KIND_CHECK = range(1, 11)


def tag(kind: int, level: int = 0) -> int:
    return kind | (level << 8)


@dataclass(frozen=True)
class Params:
    """Protocol parameters; defaults are Example 3.1 (lambda = 140)."""
    d: int = 3
    r: tuple = (1536, 1024, 652)     # r_1 .. r_d
    t: tuple = (80, 80)              # t_2 .. t_d
    sigma: float = 0.5
    qbits: int = 16
    rounds: int = 20
    act_nested: bool = True          # False: the paper's deployed LWE-only activation mask

    def ranks(self, n_pad: int) -> list:
        """[r_0 = n_pad, r_1, ..., r_d]"""
        return [n_pad] + list(self.r[: self.d])


def build(force: bool = False) -> str:
    """Compile the oracle's C core with gcc (OpenMP if available)."""
    os.makedirs(_BUILD, exist_ok=True)
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    try:
        subprocess.run(base + ["-fopenmp", _SRC, "-o", tmp, "-lm"], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base + [_SRC, "-o", tmp, "-lm"], check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        _declare(_lib)
    return _lib


_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_U32 = ctypes.c_uint32
_U64 = ctypes.c_uint64
_INT = ctypes.c_int


def _declare(L):
    L.orc_chacha_block.argtypes = [_P, _U32, _P, _INT, _P]
    L.orc_prg_words.argtypes = [_P, _U32, _U64, _INT, _U64, _I64, _P]
    L.orc_sample_uniform.argtypes = [_P, _U32, _U64, _INT, _I64, _I64, _P]
    L.orc_sample_gaussian.argtypes = [_P, _U32, _U64, _INT, _P, _INT, _I64, _P]
    L.orc_sample_sparse.argtypes = [_P, _U32, _U64, _INT, _I64, _U32, _INT, _P, _P]
    L.orc_sample_sparse.restype = _INT
    L.orc_sample_gaussian_at.argtypes = [_P, _U32, _U64, _INT, _P, _INT, _I64, _I64, _P]
    L.orc_sample_sparse_row.argtypes = [_P, _U32, _U64, _INT, _I64, _U32, _INT, _P, _P]
    L.orc_sample_sparse_row.restype = _INT
    L.orc_fwht_rows.argtypes = [_P, _I64, _I64, _I64, _I64, _P, _P]
    L.orc_fwht_rows_f64.argtypes = [_P, _I64, _I64, _P, _P]
    L.orc_encode_rows.argtypes = [_P, _I64, _I64, ctypes.c_int32, _P, _P]
    L.orc_ring_matmul.argtypes = [_P, _I64, _P, _I64, _P, _I64, _I64, _I64, _I64]
    L.orc_sparse_rows_matmul.argtypes = [_P, _P, _I64, _INT, _P, _I64, _I64, _P]
    L.orc_matmul_sparse_cols.argtypes = [_P, _I64, _I64, _P, _P, _I64, _INT, _P]
    L.orc_num_threads.restype = _INT


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a: np.ndarray, dtype) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dtype)


def num_threads() -> int:
    return int(lib().orc_num_threads())


# ---------------------------------------------------------------------------
# PRG and samplers
# ---------------------------------------------------------------------------
def chacha_block(key, counter: int, nonce, rounds: int = 20) -> np.ndarray:
    k = _c(key, np.uint32)
    n = _c(nonce, np.uint32)
    out = np.empty(16, np.uint32)
    lib().orc_chacha_block(_ptr(k), counter, _ptr(n), rounds, _ptr(out))
    return out


def prg_words(key, tg: int, stream_id: int, first: int, count: int, rounds: int = 20) -> np.ndarray:
    k = _c(key, np.uint32)
    out = np.empty(count, np.uint32)
    lib().orc_prg_words(_ptr(k), tg, stream_id, rounds, first, count, _ptr(out))
    return out


def sample_uniform(key, tg: int, stream_id: int, rows: int, cols: int, rounds: int = 20) -> np.ndarray:
    k = _c(key, np.uint32)
    out = np.empty((rows, cols), np.uint32)
    lib().orc_sample_uniform(_ptr(k), tg, stream_id, rounds, rows, cols, _ptr(out))
    return out


def gaussian_bound(sigma: float) -> int:
    """Table half-width B = ceil(12 sigma): mass beyond it is below 2^-64."""
    return int(math.ceil(12.0 * float(np.float32(sigma))))


def gaussian_table(sigma: float) -> np.ndarray:
    """table[j] = floor(2^64 * CDF(j - B)) for Pr[k] ~ exp(-k^2/(2 sigma^2))
    on [-B, B] (Sec. 3.1, Thm 3.2 statement), in 60-digit decimal arithmetic;
    the last entry saturates at 2^64 - 1."""
    s = Decimal(float(np.float32(sigma)))
    B = gaussian_bound(sigma)
    with localcontext() as ctx:
        ctx.prec = 60
        w = [(-(Decimal(k) ** 2) / (2 * s * s)).exp() for k in range(-B, B + 1)]
        z = sum(w)
        acc = Decimal(0)
        table = []
        for wk in w:
            acc += wk
            v = int((acc / z * (Decimal(2) ** 64)).to_integral_value(rounding="ROUND_FLOOR"))
            table.append(min(v, 2 ** 64 - 1))
    return np.array(table, dtype=np.uint64)


def sample_gaussian(key, tg: int, stream_id: int, count: int, sigma: float, rounds: int = 20) -> np.ndarray:
    """count discrete-Gaussian ring elements (uint32 two's complement)."""
    out = np.zeros(count, np.uint32)
    if float(sigma) == 0.0 or count == 0:
        return out
    k = _c(key, np.uint32)
    table = gaussian_table(sigma)
    lib().orc_sample_gaussian(_ptr(k), tg, stream_id, rounds, _ptr(table), gaussian_bound(sigma),
                              count, _ptr(out))
    return out


def sample_sparse(key, tg: int, stream_id: int, rows: int, r: int, t: int, rounds: int = 20):
    """rows sparse vectors over [0, r) with exactly t nonzeros: (idx, val), each rows x t."""
    k = _c(key, np.uint32)
    idx = np.zeros((rows, t), np.uint32)
    val = np.zeros((rows, t), np.uint32)
    st = lib().orc_sample_sparse(_ptr(k), tg, stream_id, rounds, rows, r, t, _ptr(idx), _ptr(val))
    if st != 0:
        raise RuntimeError("sparse sampler exhausted a row window")
    return idx, val


def sample_gaussian_at(key, tg: int, stream_id: int, first: int, count: int, sigma: float,
                       rounds: int = 20) -> np.ndarray:
    """Elements [first, first + count) of the Gaussian stream of sample_gaussian."""
    out = np.zeros(count, np.uint32)
    if float(sigma) == 0.0 or count == 0:
        return out
    k = _c(key, np.uint32)
    table = gaussian_table(sigma)
    lib().orc_sample_gaussian_at(_ptr(k), tg, stream_id, rounds, _ptr(table), gaussian_bound(sigma),
                                 first, count, _ptr(out))
    return out


def sample_sparse_row(key, tg: int, stream_id: int, row: int, r: int, t: int, rounds: int = 20):
    """Row `row` of the sparse matrix of sample_sparse: (idx, val), each of length t."""
    k = _c(key, np.uint32)
    idx = np.zeros(t, np.uint32)
    val = np.zeros(t, np.uint32)
    if lib().orc_sample_sparse_row(_ptr(k), tg, stream_id, rounds, row, r, t, _ptr(idx), _ptr(val)) != 0:
        raise RuntimeError("sparse sampler exhausted a row window")
    return idx, val


def sample_signs(key, stream_id: int, n_pad: int, rounds: int = 20) -> np.ndarray:
    """Sign words of d (Pi_Sec-Linear Init W step 1): bit c of the stream is 1 where d_c = -1."""
    return prg_words(key, tag(KIND_SIGN), stream_id, 0, (n_pad + 31) // 32, rounds)


def signs_to_pm1(words: np.ndarray, n_pad: int) -> np.ndarray:
    bits = (words[np.arange(n_pad) // 32] >> (np.arange(n_pad) % 32).astype(np.uint32)) & 1
    return np.where(bits == 1, -1.0, 1.0)


# ---------------------------------------------------------------------------
# Rotation, quantisation, ring products
# ---------------------------------------------------------------------------
def fwht_rows(x: np.ndarray, n_pad: int, sign_words) -> np.ndarray:
    """Rows of x (rows x n, float32) -> rows of H D x (rows x n_pad, float32)."""
    x = _c(x, np.float32)
    rows, n = x.shape
    y = np.empty((rows, n_pad), np.float32)
    sw = _c(sign_words, np.uint32) if sign_words is not None else None
    lib().orc_fwht_rows(_ptr(x), rows, n, n, n_pad, _ptr(sw) if sw is not None else None, _ptr(y))
    return y


def fwht_rows_f64(x: np.ndarray, sign_words) -> np.ndarray:
    x = _c(x, np.float64)
    rows, n_pad = x.shape
    y = np.empty_like(x)
    sw = _c(sign_words, np.uint32) if sign_words is not None else None
    lib().orc_fwht_rows_f64(_ptr(x), rows, n_pad, _ptr(sw) if sw is not None else None, _ptr(y))
    return y


def qmax_for(n_pad: int, qbits: int = 16) -> int:
    """Operand window: the largest q with n_pad q^2 <= 2^31 (Sec. 4 straw-man
    paragraph, kappa = 32), capped at the signed b-bit range 2^(b-1) - 1."""
    return min((1 << (qbits - 1)) - 1, math.isqrt((1 << 31) // n_pad))


def encode_rows(v: np.ndarray, qmax: int):
    """Per-row quantisation -> (codes uint32 rows x n_pad, scales float32 rows)."""
    v = _c(v, np.float32)
    rows, n_pad = v.shape
    code = np.empty((rows, n_pad), np.uint32)
    scale = np.empty(rows, np.float32)
    lib().orc_encode_rows(_ptr(v), rows, n_pad, qmax, _ptr(code), _ptr(scale))
    return code, scale


def matmul(A: np.ndarray, B: np.ndarray) -> np.ndarray:
    """A B over Z_{2^32} by the naive triple loop."""
    A = _c(A, np.uint32)
    B = _c(B, np.uint32)
    M, K = A.shape
    K2, N = B.shape
    assert K == K2
    C = np.empty((M, N), np.uint32)
    lib().orc_ring_matmul(_ptr(A), K, _ptr(B), N, _ptr(C), N, M, N, K)
    return C


def sparse_rows_matmul(S, Q: np.ndarray) -> np.ndarray:
    """S Q with S row-sparse given as (idx, val), each rows x t."""
    idx, val = (_c(a, np.uint32) for a in S)
    Q = _c(Q, np.uint32)
    rows, t = idx.shape
    l = Q.shape[1]
    out = np.empty((rows, l), np.uint32)
    lib().orc_sparse_rows_matmul(_ptr(idx), _ptr(val), rows, t, _ptr(Q), l, l, _ptr(out))
    return out


def matmul_sparse_cols(A: np.ndarray, T) -> np.ndarray:
    """A T with T column-sparse given as (idx, val), each l x t (one row per column of T)."""
    A = _c(A, np.uint32)
    idx, val = (_c(a, np.uint32) for a in T)
    rows = A.shape[0]
    l, t = idx.shape
    out = np.empty((rows, l), np.uint32)
    lib().orc_matmul_sparse_cols(_ptr(A), A.shape[1], rows, _ptr(idx), _ptr(val), l, t, _ptr(out))
    return out


# ---------------------------------------------------------------------------
# Protocol (Sec. 3.2 box Pi_Sec-Approx-MatMul and Sec. 4 box Pi_Sec-Linear)
# ---------------------------------------------------------------------------
def chains(key, p: Params, n_pad: int, stream_id: int | None = None):
    """Public M_i (r_i x r_{i-1}) and N_i (r_{i-1} x r_i), r_0 = n_pad, shared by
    every weight matrix of input width n_pad; returns
    P_i = M_i ... M_1 (r_i x n_pad) and C_i = N_1 ... N_i (n_pad x r_i), i = 1..d."""
    sid = n_pad if stream_id is None else stream_id
    r = p.ranks(n_pad)
    M = [sample_uniform(key, tag(KIND_M, i), sid, r[i], r[i - 1], p.rounds) for i in range(1, p.d + 1)]
    N = [sample_uniform(key, tag(KIND_N, i), sid, r[i - 1], r[i], p.rounds) for i in range(1, p.d + 1)]
    P = [M[0]]
    C = [N[0]]
    for i in range(1, p.d):
        P.append(matmul(M[i], P[-1]))
        C.append(matmul(C[-1], N[i]))
    return P, C


@dataclass
class WeightState:
    """Client- and server-side state of one weight matrix after Init W."""
    W_masked: np.ndarray      # W' = W_hat + U_w           (m x n_pad), stored on G
    W_hat: np.ndarray         # quantised rotated weights  (m x n_pad)
    s_w: np.ndarray           # per-row scales             (m,)
    sign_words: np.ndarray    # d of R = H D               (n_pad/32,)
    L: np.ndarray             # m x r_d
    S: dict                   # i+1 -> (idx, val), m x t_{i+1}, over [0, r_i)
    E_w: np.ndarray           # m x n_pad (kept for the tests' noise identity)
    J: list                   # J_i = (W_hat + E_w) C_i, m x r_i
    n: int
    n_pad: int
    qmax: int


def init_w(key, p: Params, W: np.ndarray, matrix_id: int, P, C, n_pad: int) -> WeightState:
    """Pi_Sec-Linear Init W (rotate W R^T, per-row quantise) followed by
    Pi_Sec-Approx-MatMul Init W (sample L, S_{i+1}, E_w; U_w; W'; J_i)."""
    m, n = W.shape
    r = p.ranks(n_pad)
    d_words = sample_signs(key, matrix_id, n_pad, p.rounds)
    W_rot = fwht_rows(W, n_pad, d_words)                    # W R^T, row by row
    qmax = qmax_for(n_pad, p.qbits)
    W_hat, s_w = encode_rows(W_rot, qmax)
    L = sample_uniform(key, tag(KIND_L), matrix_id, m, r[p.d], p.rounds)
    S = {}
    for i in range(1, p.d):
        S[i + 1] = sample_sparse(key, tag(KIND_S, i + 1), matrix_id, m, r[i], p.t[i - 1], p.rounds)
    E_w = sample_gaussian(key, tag(KIND_EW), matrix_id, m * n_pad, p.sigma, p.rounds).reshape(m, n_pad)
    U_w = matmul(L, P[p.d - 1])
    for i in range(1, p.d):
        U_w = U_w + sparse_rows_matmul(S[i + 1], P[i - 1])
    U_w = U_w + E_w
    W_masked = W_hat + U_w
    WE = W_hat + E_w
    # J_i = (W_hat + E_w) N_1 ... N_i (Init W step 3); without the nested
    # activation mask only J_1 is needed (Sec. 5.2, "Protocol parameterization").
    J = [matmul(WE, C[i - 1]) for i in range(1, (p.d if p.act_nested else 1) + 1)]
    return WeightState(W_masked, W_hat, s_w, d_words, L, S, E_w, J, n, n_pad, qmax)


@dataclass
class PassState:
    """Per-pass masking material of Init X."""
    U_x: np.ndarray           # n_pad x l
    K: np.ndarray             # m x l
    R: np.ndarray             # r_d x l
    T: dict                   # i+1 -> (idx, val), l x t_{i+1}: column k of T_{i+1}
    E_x: np.ndarray           # n_pad x l


def init_x(key, p: Params, l: int, pass_id: int, C, J, n_pad: int) -> PassState:
    """Init X (Sec. 3.2 box, steps 1a-1c).  Layout: R^T is sampled as an
    l x r_d uniform matrix, column k of T_{i+1} is sparse row k, and E_x^T is
    sampled as an l x n_pad Gaussian matrix.

    Without the nested activation mask (Sec. 5.2, "Protocol
    parameterization": the recursive LPN part is omitted for activations),
    R is r_1 x l from the same stream, U_x = N_1 R + E_x and K = J_1 R."""
    r = p.ranks(n_pad)
    if not p.act_nested:
        R = sample_uniform(key, tag(KIND_R), pass_id, l, r[1], p.rounds).T.copy()
        E_x = sample_gaussian(key, tag(KIND_EX), pass_id, l * n_pad, p.sigma,
                              p.rounds).reshape(l, n_pad).T.copy()
        U_x = matmul(C[0], R) + E_x
        K = matmul(J[0], R)
        return PassState(U_x, K, R, {}, E_x)
    R = sample_uniform(key, tag(KIND_R), pass_id, l, r[p.d], p.rounds).T.copy()
    T = {}
    for i in range(1, p.d):
        T[i + 1] = sample_sparse(key, tag(KIND_T, i + 1), pass_id, l, r[i], p.t[i - 1], p.rounds)
    E_x = sample_gaussian(key, tag(KIND_EX), pass_id, l * n_pad, p.sigma, p.rounds).reshape(l, n_pad).T.copy()
    U_x = matmul(C[p.d - 1], R)
    for i in range(1, p.d):
        U_x = U_x + matmul_sparse_cols(C[i - 1], T[i + 1])
    U_x = U_x + E_x
    K = matmul(J[p.d - 1], R)
    for i in range(1, p.d):
        K = K + matmul_sparse_cols(J[i - 1], T[i + 1])
    return PassState(U_x, K, R, T, E_x)


def mask_input(X: np.ndarray, ws: WeightState, U_x: np.ndarray):
    """Pi_Sec-Linear Online step 1 (X~ = R X, per-column quantise) and
    Approx-MatMul Online step 2 (X' = X_hat + U_x).  X is n x l (float32).
    Returns (X_hat, s_x, X') with X_hat, X' n_pad x l."""
    Xt_rot = fwht_rows(X.T, ws.n_pad, ws.sign_words)        # columns of R X, as rows
    Xt_hat, s_x = encode_rows(Xt_rot, ws.qmax)
    X_hat = Xt_hat.T.copy()
    return X_hat, s_x, X_hat + U_x


def server(ws: WeightState, P, X_masked: np.ndarray):
    """Approx-MatMul Online step 3: Y' = W' X' and Q_i = P_i X', i = 1..d."""
    Y_masked = matmul(ws.W_masked, X_masked)
    Q = [matmul(Pi, X_masked) for Pi in P]
    return Y_masked, Q


def unmask(p: Params, ws: WeightState, ps: PassState, Y_masked: np.ndarray, Q) -> np.ndarray:
    """Approx-MatMul Online step 5: Y_hat = Y' - K - L Q_d - sum_i S_{i+1} Q_i."""
    Y = Y_masked - ps.K
    Y = Y - matmul(ws.L, Q[p.d - 1])
    for i in range(1, p.d):
        Y = Y - sparse_rows_matmul(ws.S[i + 1], Q[i - 1])
    return Y


def freivalds_setup(key, p: Params, ws: WeightState, matrix_id: int, k: int):
    """Init W step 4 with the check vectors in Z_{2^32}^m (rows of a, k x m,
    from stream (CHECK, matrix_id)): returns (a, Y_chk = a W')."""
    m = ws.W_masked.shape[0]
    a = sample_uniform(key, tag(KIND_CHECK), matrix_id, k, m, p.rounds)
    return a, matmul(a, ws.W_masked)


def freivalds_check(a: np.ndarray, Y_chk: np.ndarray, Y_masked: np.ndarray, X_masked: np.ndarray):
    """Online step 4 (appendix "Computational integrity"), per column j of Y':
    the number of check vectors v with a_v^T Y'_j != Y_chk,v X'_j (mod 2^32)."""
    lhs = matmul(a, Y_masked)
    rhs = matmul(Y_chk, X_masked)
    return np.sum(lhs != rhs, axis=0).astype(np.uint32)


def decode(Y_hat: np.ndarray, s_w: np.ndarray, s_x: np.ndarray, b=None) -> np.ndarray:
    """Pi_Sec-Linear Online step 3 in fp64: Y = s_w s_x Y_hat (+ b), Y_hat read
    as a signed 32-bit integer."""
    Y = Y_hat.view(np.int32).astype(np.float64) * s_w.astype(np.float64)[:, None]
    Y = Y * s_x.astype(np.float64)[None, :]
    if b is not None:
        Y = Y + np.asarray(b, np.float64)[:, None]
    return Y


def secure_linear(key, p: Params, W: np.ndarray, X: np.ndarray, matrix_id: int, pass_id: int,
                  b=None, chains_=None):
    """One full Pi_Sec-Linear call: returns a dict of every intermediate."""
    m, n = W.shape
    n_pad = 1 << max(0, (n - 1).bit_length())
    P, C = chains_ if chains_ is not None else chains(key, p, n_pad)
    ws = init_w(key, p, W, matrix_id, P, C, n_pad)
    l = X.shape[1]
    ps = init_x(key, p, l, pass_id, C, ws.J, n_pad)
    X_hat, s_x, X_masked = mask_input(X, ws, ps.U_x)
    Y_masked, Q = server(ws, P, X_masked)
    Y_hat = unmask(p, ws, ps, Y_masked, Q)
    Y = decode(Y_hat, ws.s_w, s_x, b)
    return dict(P=P, C=C, ws=ws, ps=ps, X_hat=X_hat, s_x=s_x, X_masked=X_masked,
                Y_masked=Y_masked, Q=Q, Y_hat=Y_hat, Y=Y, n_pad=n_pad)
