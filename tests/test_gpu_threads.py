"""First calls from several host threads at once.

The library sets per-kernel shared-memory limits and looks up the driver's
tensor-map encoder lazily, on the first call that needs them.  A fresh
process starts four host threads that pass a barrier and then make their
first calls together (each a whole secure linear call on its own stream: two
through the tensor-core products, two through the streaming few-token
product); every thread's Y_hat must equal the same call made again
afterwards from one thread."""
import os
import subprocess
import sys

import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys, threading
import numpy as np
import torch
sys.path.insert(0, sys.argv[1])
from paper_2607_29221_gb300 import mosaic as M, protocol as PR, workloads as wl
M.lib()
torch.cuda.init()
CASES = [(64, 0), (64, 1), (8, 2), (8, 3)]          # (tokens, case id)
barrier = threading.Barrier(len(CASES))

def run(l, cid, out, wait):
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        m, n = 384, 700
        W = torch.from_numpy(wl.weights(m, n, seed=40 + cid)).cuda()
        X = torch.from_numpy(wl.activations(l, n, seed=50 + cid)).cuda()
        stream.synchronize()
        if wait:
            barrier.wait()
        proto = PR.Protocol(wl.mask_key(), M.default_params(), variant=M.GEMM_AUTO)
        ch = PR.Chains(proto, PR.pad_width(n))
        layer = PR.SecureLinear(proto, W, 60 + cid, ch)
        mp = layer.init_x(l, 70 + cid)
        Yhat = torch.empty(l, m, dtype=torch.int32, device="cuda")
        layer.forward(X, mp, Yhat=Yhat)
        stream.synchronize()
        out[cid] = Yhat.cpu().numpy()

first = {}
errs = []
def guarded(l, cid):
    try:
        run(l, cid, first, True)
    except Exception as e:                      # reported by the parent
        errs.append(repr(e))
ts = [threading.Thread(target=guarded, args=c) for c in CASES]
for t in ts: t.start()
for t in ts: t.join()
assert not errs, errs
M.mosaic_device_status()
again = {}
for l, cid in CASES:
    run(l, cid, again, False)
for l, cid in CASES:
    assert np.array_equal(first[cid], again[cid]), cid
print("threads ok")
"""


def test_first_calls_from_four_threads():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_29221_gb300 import build
    build.build()
    r = subprocess.run([sys.executable, "-c", CHILD, ROOT], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and "threads ok" in r.stdout, r.stdout + r.stderr
