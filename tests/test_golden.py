"""Values the paper prints (tests/golden/*.json, each with its source passage)
against the library's and the oracle's defaults and the oracle's client state.
Host-only: no GPU call."""
import json
import os

import numpy as np

import oracle as O
from paper_2607_29221_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def test_example_3_1_is_the_default_parameter_set():
    ex = _load("example_3_1.json")
    r = (ex["lwe"]["r_1"],) + tuple(x["r"] for x in ex["lpn"])
    t = tuple(x["t"] for x in ex["lpn"])
    p = O.Params()
    assert (p.d, tuple(p.r), tuple(p.t), p.sigma) == (ex["d"], r, t, ex["lwe"]["sigma"])
    # each LPN level's sample bound N_i is the previous level's secret dimension r_{i-1}
    assert [x["N"] for x in ex["lpn"]] == list(r[:-1])
    from paper_2607_29221_gb300 import build as B
    from paper_2607_29221_gb300 import mosaic as M
    B.build()
    q = M.default_params()
    assert (q.d, list(q.r), list(q.t)[1:], float(q.sigma)) == (ex["d"], list(r), list(t), ex["lwe"]["sigma"])


def test_client_state_of_the_oracle_matches_the_tradeoff_table():
    """Words the oracle keeps on the client per weight matrix -- C_i (n x r_i),
    J_i (m x r_i), L (m x r_d) -- counted from its arrays, against the table's
    a (m + n) + b m; client compute per (m + n) l = r_d + sum t."""
    tab = _load("lpn_tradeoff.json")
    ex = _load("example_3_1.json")
    r_all = (ex["lwe"]["r_1"],) + tuple(x["r"] for x in ex["lpn"])
    t_all = tuple(x["t"] for x in ex["lpn"])
    key = wl.mask_key()
    m, n = 3, 32
    for row in tab["rows"]:
        d = row["d"]
        p = O.Params(d=d, r=r_all[:d], t=t_all[: d - 1])
        P, C = O.chains(key, p, n)
        ws = O.init_w(key, p, wl.weights(m, n, seed=9), 1, P, C, n)
        words = sum(c.size for c in C) + sum(j.size for j in ws.J) + ws.L.size
        assert words == row["state_a"] * (m + n) + row["state_b"] * m, row
        assert p.r[-1] + sum(p.t) == row["compute_per_ml"], row
        assert np.all([c.shape == (n, ri) for c, ri in zip(C, p.r)])
