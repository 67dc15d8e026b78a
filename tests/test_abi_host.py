"""The C-ABI library builds, loads and exports every symbol include/mosaic.h
declares; host-only entry points and argument validation work without a GPU
(no compute call is made here)."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle as O
from paper_2607_29221_gb300 import build as B
from paper_2607_29221_gb300 import mosaic as M

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    return M.lib()


def _declared():
    src = open(os.path.join(ROOT, "include", "mosaic.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mosaic_[a-z0-9_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 17
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(M.EXPORTS)


def test_default_params_are_example_3_1(lib):
    p = M.default_params()
    assert (p.kappa, p.d, list(p.r), list(p.t)[1:], p.qbits, p.rounds) == (
        32, 3, [1536, 1024, 652], [80, 80], 16, 20)
    assert abs(p.sigma - 0.5) == 0


def test_status_strings(lib):
    for s in range(8):
        assert lib.mosaic_status_string(s)
    assert lib.mosaic_status_string(99) == b"unknown status"


def test_qmax_matches_oracle(lib):
    for k in range(5, 17):
        assert M.mosaic_qmax(1 << k) == O.qmax_for(1 << k)
    assert M.mosaic_qmax(1 << 16) == 181
    assert M.mosaic_qmax(1000) == 0 and M.mosaic_qmax(1 << 17) == 0 and M.mosaic_qmax(16) == 0


def test_gaussian_table_matches_oracle(lib):
    exact = np.finfo(np.longdouble).nmant >= 112      # binary128 long double (Arm)
    for s in (0.5, 0.7, 1.0, 1.5, 2.0, 8.0):
        a = M.mosaic_gaussian_table(s).astype(object)
        b = O.gaussian_table(s).astype(object)
        assert len(a) == len(b)
        diff = max(abs(x - y) for x, y in zip(a, b))
        assert diff == 0 if exact else diff <= 16, (s, diff)


def test_workspace_sizes(lib):
    p = M.default_params()
    assert M.mosaic_workspace_bytes(M.OP_MASK_WEIGHT, 4096, 4096, 0, p) >= 4096 * 4096 * 4
    assert M.mosaic_workspace_bytes(M.OP_UNMASK, 4096, 0, 512, p) >= 512 * 4096 * 4
    assert M.mosaic_workspace_bytes(M.OP_MASK_ACTIVATION, 4096, 4096, 512, p) >= 512 * 652 * 4
    assert M.mosaic_workspace_bytes(M.OP_RING_GEMM, 8, 8, 8, p) >= 8 * 8 * 8 * 2
    bad = M.default_params(kappa=64)
    assert M.mosaic_workspace_bytes(M.OP_MASK_WEIGHT, 8, 64, 0, bad) == 0


def test_unmask_workspace_holds_the_fast_path(lib):
    """The advertised unmask workspace (Example 3.1, 512 tokens, m = 4096) holds
    every part the fast path carves: the l x m scratch, the digit planes of Q_d
    (4 x l x 656 bf16), the tile images of Q_1 and Q_2 (16 tiles x r_i x 32 words)
    and the line-offset copies of both S lists (m x 80 words each)."""
    p = M.default_params()
    l, m = 512, 4096
    need = (l * m * 4 + 4 * l * 656 * 2 + 16 * 1536 * 32 * 4 + 16 * 1024 * 32 * 4 + 2 * m * 80 * 4)
    assert M.mosaic_workspace_bytes(M.OP_UNMASK, m, 0, l, p) >= need


def _status(fn, *args):
    return getattr(M.lib(), fn)(*args)


def test_validation_without_gpu(lib):
    key = M.make_key(range(8))
    p = M.default_params()
    fake = 1 << 40   # never dereferenced: every call below fails validation first
    # n_pad not a power of two / out of range
    assert _status("mosaic_hadamard", fake, 100, fake, 4, 100, 100, None, None) == 2
    assert _status("mosaic_hadamard", fake, 64, fake, 4, 65, 64, None, None) == 2
    assert _status("mosaic_hadamard", fake, 64, fake + 4, 4, 64, 64, None, None) == 3
    assert _status("mosaic_hadamard", None, 64, fake, 4, 64, 64, None, None) == 1
    # zero rows is a no-op
    assert _status("mosaic_hadamard", None, 64, None, 0, 64, 64, None, None) == 0
    assert _status("mosaic_encode", fake, 64, 4, 64, 64, 0, 1, None, None, 0, fake, 64, fake,
                   None, None) == 1
    assert _status("mosaic_ring_gemm", fake, 4, fake, 4, fake, 4, 4, 4, 8, 3, None, 0, None) == 2
    assert _status("mosaic_ring_gemm", fake, 8, fake, 8, fake, 8, 8, 8, 8, 9, None, 0, None) == 1
    assert _status("mosaic_ring_gemm", None, 8, None, 8, None, 8, 0, 8, 8, 3, None, 0, None) == 0
    assert _status("mosaic_prg_sparse", ctypes.byref(key), 1, 0, 20, 4, 10, 6, fake, fake, None,
                   None) == 1
    assert _status("mosaic_prg_uniform", ctypes.byref(key), 1, 0, 7, 4, 4, fake, 4, None) == 1
    assert _status("mosaic_prg_gaussian", ctypes.byref(key), 1, 0, 20, ctypes.c_float(9.0), 4,
                   fake, None) == 1
    bad = M.default_params(d=4)
    assert _status("mosaic_mask_chains", ctypes.byref(bad), ctypes.byref(key), 0, 64, fake, fake,
                   fake, None, 0, None) == 1
    assert _status("mosaic_mask_chains", ctypes.byref(p), ctypes.byref(key), 0, 64, fake, fake,
                   fake, None, 0, None) == 6
    k64 = M.default_params(kappa=64)
    assert _status("mosaic_unmask", ctypes.byref(k64), 1, 1, fake, 4000, fake, fake, fake, fake,
                   fake, fake, None, fake, None, 1, 3, None, 0, None) == 4


def test_validation_of_newer_entry_points(lib):
    """Argument checks of the check, variant and prepared-operand entry points,
    all decided on the host before any device work."""
    key = M.make_key(range(8))
    p = M.default_params()
    fake = 1 << 40
    # Freivalds: k out of range, empty token batch
    assert _status("mosaic_freivalds_check", 0, fake, fake, 8, 32, 4, fake, 8, fake, 32, fake, fake,
                   None, 0, None) == 1
    assert _status("mosaic_freivalds_check", 4, fake, fake, 8, 32, 0, fake, 8, fake, 32, fake, fake,
                   None, 0, None) == 0
    assert _status("mosaic_freivalds_setup", ctypes.byref(p), ctypes.byref(key), 1, 17, fake, 32, 8, 32,
                   fake, fake, None) == 1
    # act_nested must be 0 or 1
    bad = M.default_params(act_nested=2)
    assert _status("mosaic_mask_activation_ex", ctypes.byref(bad), ctypes.byref(key), 0, None, 8, 32, 4,
                   fake, fake, None, fake, fake, 0, None, 0, None) == 1
    # Init X phases: 1 (draws), 2 (compositions), 3 (both); anything else is refused
    for phase in (0, 4, -1):
        assert _status("mosaic_mask_activation_phase", ctypes.byref(p), ctypes.byref(key), 0, None, 8, 32, 4,
                       fake, fake, None, fake, fake, 0, None, 0, phase, None) == 1
    assert _status("mosaic_mask_activation_phase", ctypes.byref(bad), ctypes.byref(key), 0, None, 8, 32, 4,
                   fake, fake, None, fake, fake, 0, None, 0, 1, None) == 1
    # K above 2^20, rotation widths beyond 65536
    assert _status("mosaic_ring_gemm", fake, 1 << 21, fake, 1 << 21, fake, 8, 8, 8, (1 << 20) + 1, 3,
                   None, 0, None) == 2
    assert _status("mosaic_hadamard", fake, 1 << 17, fake, 1, 1 << 17, 1 << 17, None, None) == 2
    # prepared planes: empty shapes, missing counter
    assert _status("mosaic_prepare_activation", ctypes.byref(p), 0, 64, fake, fake, fake, None) == 2
    assert _status("mosaic_prepare_unmask", ctypes.byref(p), 0, fake, fake, None) == 2
    assert _status("mosaic_advance_pass", None, 1, None) == 1
    assert _status("mosaic_unmask_planes", ctypes.byref(p), 1, 8, fake, 3220, fake, fake, None, fake,
                   fake, fake, fake, None, fake, None, 8, 3, None, 0, None) == 1
    assert _status("mosaic_unmask_planes", ctypes.byref(p), 1, 8, fake, 3220, fake, fake, fake + 2, fake,
                   fake, fake, fake, None, fake, None, 8, 3, None, 0, None) == 3


def test_rate_probes_need_an_output(lib):
    assert _status("mosaic_int_mix_rate", None, 0, None, None) == 1
    assert _status("mosaic_smem_read_rate", None, 0, None, None) == 1


def test_selftest_wait_validates_its_limit(lib):
    assert _status("mosaic_selftest_wait", 0, None) == 1
    assert _status("mosaic_selftest_wait", 1000001, None) == 1


def test_mosaic_mask_dispatch_validation(lib):
    """mosaic_mask: unknown kind or missing io struct is an argument error; each
    kind reaches its role call's own validation (decided on the host)."""
    key = M.make_key(range(8))
    p = M.default_params()
    fake = 1 << 40
    io = M.mosaic_mask_io()
    assert _status("mosaic_mask", 1, ctypes.byref(p), ctypes.byref(key), 0, 0, 64, 0, None, 0, None, 0,
                   None) == 1
    assert _status("mosaic_mask", 9, ctypes.byref(p), ctypes.byref(key), 0, 0, 64, 0, ctypes.byref(io), 0,
                   None, 0, None) == 1
    io.P = io.C = io.CT = fake
    # chains with no workspace: the role call's own MOSAIC_ERR_WORKSPACE
    assert _status("mosaic_mask", M.MASK_CHAINS, ctypes.byref(p), ctypes.byref(key), 0, 0, 64, 0,
                   ctypes.byref(io), 0, None, 0, None) == 6
    # chains with a width that is not a power of two
    assert _status("mosaic_mask", M.MASK_CHAINS, ctypes.byref(p), ctypes.byref(key), 0, 0, 100, 0,
                   ctypes.byref(io), 0, None, 0, None) == 2
    bad = M.default_params(act_nested=2)
    assert _status("mosaic_mask", M.MASK_ACTIVATION, ctypes.byref(bad), ctypes.byref(key), 0, 8, 32, 4,
                   ctypes.byref(io), 0, None, 0, None) == 1


def test_kernel_timing_toggle_without_gpu(lib):
    """Per-kernel timing is off by default, toggles, and reports no records
    when nothing was launched."""
    from paper_2607_29221_gb300 import mosaic as M
    assert M.mosaic_kernel_timing(True) is False
    assert M.mosaic_kernel_timing(False) is True
    assert M.mosaic_kernel_times(reset=True) == {}
