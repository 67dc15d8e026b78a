"""The sampled-output oracle (used for full-size parity) agrees exactly with the
full oracle at every sampled position, on a small layer."""
import numpy as np

import oracle as O
from oracle import sampled as OS
from paper_2607_29221_gb300 import workloads as wl

KEY = wl.mask_key()


def test_sampled_matches_full_oracle():
    p = O.Params(d=3, r=(96, 64, 40), t=(6, 5), sigma=1.0)
    m, n, l = 37, 150, 23
    n_pad = 256
    W = wl.weights(m, n, std=1.0)
    X_tm = wl.activations(l, n)
    b = wl.bias(m)
    full = O.secure_linear(KEY, p, W, X_tm.T.copy(), matrix_id=4, pass_id=9, b=b)
    P, C = full["P"], full["C"]
    rows = np.array([0, 5, 36])
    toks = np.array([0, 11, 22])
    wr = OS.weight_rows(KEY, p, W[rows], rows, 4, P, C, n_pad)
    ws = full["ws"]
    assert np.array_equal(wr.W_masked, ws.W_masked[rows])
    assert np.array_equal(wr.s_w, ws.s_w[rows])
    for i in range(3):
        assert np.array_equal(wr.J[i], ws.J[i][rows])
    tc = OS.token_cols(KEY, p, X_tm[toks], toks, 9, wr.sign_words, wr.qmax, C, n_pad)
    assert np.array_equal(tc.U_x, full["ps"].U_x[:, toks])
    assert np.array_equal(tc.X_masked, full["X_masked"][:, toks])
    assert np.array_equal(tc.s_x, full["s_x"][toks])
    K = OS.k_entries(p, wr, tc)
    assert np.array_equal(K, full["ps"].K[np.ix_(rows, toks)])
    Ym, Q = OS.server_entries(wr, tc, P)
    assert np.array_equal(Ym, full["Y_masked"][np.ix_(rows, toks)])
    for i in range(3):
        assert np.array_equal(Q[i], full["Q"][i][:, toks])
    Yh = OS.unmask_entries(p, wr, K, Ym, Q)
    assert np.array_equal(Yh, full["Y_hat"][np.ix_(rows, toks)])
