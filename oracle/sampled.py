"""Sampled-output oracle for full-size workloads.

TEST INFRASTRUCTURE (part of the oracle package; see its header).  For
weight matrices and batches too large for the naive triple loop, these
functions restate the same protocol steps as ``oracle`` (Sec. 3.2 box
Pi_Sec-Approx-MatMul and Sec. 4 box Pi_Sec-Linear, paper orientation) for a
chosen set of weight rows j and tokens k only; every value they return is the
exact value the full computation would have at those positions.  The public
chains P_i, C_i are computed in full by ``oracle.chains``.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import (KIND_EW, KIND_EX, KIND_L, KIND_R, KIND_S, KIND_T, Params, encode_rows,
               fwht_rows, matmul, matmul_sparse_cols, prg_words, qmax_for, sample_gaussian_at,
               sample_signs, sample_sparse_row, sparse_rows_matmul, tag)


def uniform_rows(key, tg, stream_id, rows, cols, rounds=20) -> np.ndarray:
    """Rows `rows` of the uniform matrix whose element (i, c) is stream word i * cols + c."""
    return np.stack([prg_words(key, tg, stream_id, int(j) * cols, cols, rounds) for j in rows])


@dataclass
class WeightRows:
    rows: np.ndarray          # which output rows j
    sign_words: np.ndarray
    qmax: int
    W_hat: np.ndarray         # len(rows) x n_pad
    s_w: np.ndarray
    L: np.ndarray             # len(rows) x r_d
    S: dict                   # i+1 -> (idx, val), len(rows) x t_{i+1}
    E_w: np.ndarray           # len(rows) x n_pad
    W_masked: np.ndarray      # rows of W'
    J: list                   # J_i rows, len(rows) x r_i


def weight_rows(key, p: Params, W_rows: np.ndarray, rows, matrix_id: int, P, C, n_pad: int) -> WeightRows:
    """Init W (Pi_Sec-Linear steps 1-2, Approx-MatMul steps 1-3) restricted to rows `rows`;
    W_rows holds those rows of W (len(rows) x n, float32)."""
    rows = np.asarray(rows)
    r = p.ranks(n_pad)
    d_words = sample_signs(key, matrix_id, n_pad, p.rounds)
    qmax = qmax_for(n_pad, p.qbits)
    W_hat, s_w = encode_rows(fwht_rows(W_rows, n_pad, d_words), qmax)
    L = uniform_rows(key, tag(KIND_L), matrix_id, rows, r[p.d], p.rounds)
    S = {}
    for i in range(1, p.d):
        pairs = [sample_sparse_row(key, tag(KIND_S, i + 1), matrix_id, int(j), r[i], p.t[i - 1], p.rounds)
                 for j in rows]
        S[i + 1] = (np.stack([a for a, _ in pairs]), np.stack([b for _, b in pairs]))
    E_w = np.stack([sample_gaussian_at(key, tag(KIND_EW), matrix_id, int(j) * n_pad, n_pad, p.sigma,
                                       p.rounds) for j in rows])
    U_w = matmul(L, P[p.d - 1])
    for i in range(1, p.d):
        U_w = U_w + sparse_rows_matmul(S[i + 1], P[i - 1])
    U_w = U_w + E_w
    WE = W_hat + E_w
    J = [matmul(WE, C[i - 1]) for i in range(1, p.d + 1)]
    return WeightRows(rows, d_words, qmax, W_hat, s_w, L, S, E_w, W_hat + U_w, J)


@dataclass
class TokenCols:
    toks: np.ndarray
    R: np.ndarray             # r_d x len(toks)
    T: dict                   # i+1 -> (idx, val), len(toks) x t_{i+1}
    E_x: np.ndarray           # n_pad x len(toks)
    U_x: np.ndarray           # n_pad x len(toks)
    X_hat: np.ndarray         # n_pad x len(toks)
    s_x: np.ndarray
    X_masked: np.ndarray      # n_pad x len(toks)


def token_cols(key, p: Params, X_rows: np.ndarray, toks, pass_id: int, sign_words, qmax: int, C,
               n_pad: int) -> TokenCols:
    """Init X (steps 1a-1b) and the client's masking of X (Online 1-2) for tokens `toks`;
    X_rows holds those tokens' activations (len(toks) x n, float32)."""
    toks = np.asarray(toks)
    r = p.ranks(n_pad)
    R = uniform_rows(key, tag(KIND_R), pass_id, toks, r[p.d], p.rounds).T.copy()
    T = {}
    for i in range(1, p.d):
        pairs = [sample_sparse_row(key, tag(KIND_T, i + 1), pass_id, int(k), r[i], p.t[i - 1], p.rounds)
                 for k in toks]
        T[i + 1] = (np.stack([a for a, _ in pairs]), np.stack([b for _, b in pairs]))
    E_x = np.stack([sample_gaussian_at(key, tag(KIND_EX), pass_id, int(k) * n_pad, n_pad, p.sigma,
                                       p.rounds) for k in toks]).T.copy()
    U_x = matmul(C[p.d - 1], R)
    for i in range(1, p.d):
        U_x = U_x + matmul_sparse_cols(C[i - 1], T[i + 1])
    U_x = U_x + E_x
    Xt_hat, s_x = encode_rows(fwht_rows(X_rows, n_pad, sign_words), qmax)
    X_hat = Xt_hat.T.copy()
    return TokenCols(toks, R, T, E_x, U_x, X_hat, s_x, X_hat + U_x)


def k_entries(p: Params, wr: WeightRows, tc: TokenCols) -> np.ndarray:
    """K = J_d R + sum_i J_i T_{i+1} (Init X step 1c) at rows x toks."""
    K = matmul(wr.J[p.d - 1], tc.R)
    for i in range(1, p.d):
        K = K + matmul_sparse_cols(wr.J[i - 1], tc.T[i + 1])
    return K


def server_rows(wr: WeightRows, tc: TokenCols) -> np.ndarray:
    """Online 3, the weight side: Y' = W' X' at rows x toks."""
    return matmul(wr.W_masked, tc.X_masked)


def server_q(tc: TokenCols, P) -> list:
    """Online 3, the chain side: Q_i = P_i X' at all r_i x toks."""
    return [matmul(Pi, tc.X_masked) for Pi in P]


def server_entries(wr: WeightRows, tc: TokenCols, P):
    """Online 3: Y' = W' X' at rows x toks, and Q_i = P_i X' at all r_i x toks."""
    return server_rows(wr, tc), server_q(tc, P)


def unmask_entries(p: Params, wr: WeightRows, K, Y_masked, Q) -> np.ndarray:
    """Online 5: Y_hat = Y' - K - L Q_d - sum_i S_{i+1} Q_i at rows x toks."""
    Y = Y_masked - K - matmul(wr.L, Q[p.d - 1])
    for i in range(1, p.d):
        Y = Y - sparse_rows_matmul(wr.S[i + 1], Q[i - 1])
    return Y
