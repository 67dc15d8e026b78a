"""mosaic_mask(kind, ...): the single mask-generation entry point of the C ABI
(Sec. 3.2 box: Init W steps 1-3 and 5, Init X steps 1a-1c) against the
oracle, for each of its three kinds -- public chains, weight mask, activation
mask -- bit-exact on every ring output."""
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
    yield


def _u32(t):
    torch.cuda.synchronize()
    return t.cpu().numpy().view(np.uint32)


def _i32(*shape):
    return torch.zeros(*shape, dtype=torch.int32, device="cuda")


@pytest.mark.parametrize("act_nested", [1, 0])
def test_mosaic_mask_each_kind_matches_oracle(act_nested):
    from paper_2607_29221_gb300 import mosaic as M
    p = M.default_params(act_nested=act_nested)
    po = O.Params(act_nested=bool(act_nested))
    key = M.make_key(KEY)
    m, n, l, n_pad, matrix_id, pass_id = 300, 500, 40, 512, 12, 31
    Sr, rd = sum(po.r), po.r[-1]
    ws = torch.empty(max(M.mosaic_workspace_bytes(op, m, n_pad, l, p)
                         for op in (M.OP_MASK_CHAINS, M.OP_MASK_WEIGHT, M.OP_MASK_ACTIVATION)),
                     dtype=torch.uint8, device="cuda")
    # public chains
    P, C, CT = _i32(Sr, n_pad), _i32(n_pad, Sr), _i32(Sr, n_pad)
    M.mosaic_mask(M.MASK_CHAINS, p, key, n_pad, 0, n_pad, 0, dict(P=P, C=C, CT=CT), M.GEMM_AUTO, ws)
    Po, Co = O.chains(KEY, po, n_pad)
    assert np.array_equal(_u32(P), np.vstack(Po))
    assert np.array_equal(_u32(C), np.hstack(Co))
    assert np.array_equal(_u32(CT), np.hstack(Co).T)
    # weight mask
    W = wl.weights(m, n, seed=77)
    Wd = torch.from_numpy(W).cuda()
    sw, s_w, L = _i32(n_pad // 32), torch.empty(m, dtype=torch.float32, device="cuda"), _i32(m, rd)
    nsp = sum(po.t) * m
    S_idx, S_val, Wp, J = _i32(nsp), _i32(nsp), _i32(m + Sr, n_pad), _i32(m, Sr)
    M.mosaic_mask(M.MASK_WEIGHT, p, key, matrix_id, m, n_pad, 0,
                  dict(W=Wd, ldw=n, n=n, P=P, CT=CT, sign_words=sw, s_w=s_w, L=L, S_idx=S_idx, S_val=S_val,
                       Wp=Wp, J=J), M.GEMM_AUTO, ws)
    wo = O.init_w(KEY, po, W, matrix_id, Po, Co, n_pad)
    assert np.array_equal(_u32(sw), wo.sign_words)
    assert np.array_equal(s_w.cpu().numpy(), wo.s_w)
    assert np.array_equal(_u32(L), wo.L)
    assert np.array_equal(_u32(Wp)[:m], wo.W_masked)
    assert np.array_equal(_u32(Wp)[m:], np.vstack(Po))
    Jg = _u32(J)
    assert np.array_equal(Jg[:, :sum(po.r[:len(wo.J)])], np.hstack(wo.J))
    off = 0
    for i in range(1, po.d):
        t = po.t[i - 1]
        assert np.array_equal(_u32(S_idx)[off:off + m * t].reshape(m, t), wo.S[i + 1][0])
        assert np.array_equal(_u32(S_val)[off:off + m * t].reshape(m, t), wo.S[i + 1][1])
        off += m * t
    # activation mask (Init X of one pass)
    Ux, K = _i32(l, n_pad), _i32(l, m)
    M.mosaic_mask(M.MASK_ACTIVATION, p, key, pass_id, m, n_pad, l, dict(C=C, J=J, Ux_tm=Ux, K_tm=K),
                  M.GEMM_AUTO, ws)
    M.mosaic_device_status()
    xo = O.init_x(KEY, po, l, pass_id, Co, wo.J, n_pad)
    assert np.array_equal(_u32(Ux), xo.U_x.T)
    assert np.array_equal(_u32(K), xo.K.T)


@pytest.mark.parametrize("l,nested", [(96, 1), (12, 1), (96, 0)])
def test_init_x_in_two_phases_matches_one_call(l, nested):
    """mosaic_mask_activation_phase: the DRAWS call then the COMPOSE call on
    the same workspace give U_x and K bit-identical to one
    mosaic_mask_activation_ex call (tensor-core product, the streaming
    product at 12 tokens, and the LWE-only activation mask); the draws alone
    leave K untouched."""
    import torch
    from paper_2607_29221_gb300 import mosaic as M
    from paper_2607_29221_gb300 import protocol as PR
    from paper_2607_29221_gb300 import workloads as wl
    proto = PR.Protocol(wl.mask_key(), M.default_params(d=3, r=[96, 64, 40], t=[0, 8, 4], act_nested=nested),
                        variant=M.GEMM_TC)
    m, n = 200, 256
    ch = PR.Chains(proto, PR.pad_width(n))
    layer = PR.SecureLinear(proto, torch.from_numpy(wl.weights(m, n, std=1.0)).cuda(), 4, ch)
    one = layer.init_x(l, 42)
    ws = torch.empty(layer.init_x_workspace_bytes(l), dtype=torch.uint8, device="cuda")
    two = PR.PassMask(42, l, torch.empty_like(one.Ux), torch.full_like(one.K, 7))
    layer.init_x(l, 42, out=two, phase=M.INITX_DRAWS, ws=ws)
    torch.cuda.synchronize()
    assert bool((two.K == 7).all())
    layer.init_x(l, 42, out=two, phase=M.INITX_COMPOSE, ws=ws)
    torch.cuda.synchronize()
    assert torch.equal(one.Ux, two.Ux) and torch.equal(one.K, two.K)
    with pytest.raises(M.MosaicError):
        layer.init_x(l, 42, out=two, phase=0, ws=ws)


def test_weight_mask_workspace_sizes_match_oracle():
    """Init W with three workspaces: the full size (tensor-core products, P_d^T
    and P^T carved for the L P_d product and the tiled gather of the sparse
    terms), room for the transposes only (CUDA-core products against P_d^T,
    tiled gather), and the minimum (CUDA-core products reading P_d strided,
    row gather of P).  W' and J are bit-identical to the oracle for all three."""
    from paper_2607_29221_gb300 import mosaic as M
    p = M.default_params()
    po = O.Params()
    key = M.make_key(KEY)
    m, n, n_pad, matrix_id = 300, 500, 512, 13
    Sr, rd = sum(po.r), po.r[-1]
    od = Sr - rd
    full = M.mosaic_workspace_bytes(M.OP_MASK_WEIGHT, m, n_pad, 0, p)
    ws_c = torch.empty(M.mosaic_workspace_bytes(M.OP_MASK_CHAINS, m, n_pad, 0, p), dtype=torch.uint8,
                       device="cuda")
    P, C, CT = _i32(Sr, n_pad), _i32(n_pad, Sr), _i32(Sr, n_pad)
    M.mosaic_mask(M.MASK_CHAINS, p, key, n_pad, 0, n_pad, 0, dict(P=P, C=C, CT=CT), M.GEMM_AUTO, ws_c)
    Po, Co = O.chains(KEY, po, n_pad)
    W = wl.weights(m, n, seed=78)
    wo = O.init_w(KEY, po, W, matrix_id, Po, Co, n_pad)

    def up(v):
        return (v + 255) // 256 * 256

    minimum = up(m * n_pad * 4)
    sizes = [full, minimum + up(n_pad * max(rd, od) * 4), minimum]
    assert sizes[0] > sizes[1] > sizes[2]
    for size in sizes:
        ws = torch.empty(size, dtype=torch.uint8, device="cuda")
        sw, s_w, L = _i32(n_pad // 32), torch.empty(m, dtype=torch.float32, device="cuda"), _i32(m, rd)
        nsp = sum(po.t) * m
        S_idx, S_val, Wp, J = _i32(nsp), _i32(nsp), _i32(m + Sr, n_pad), _i32(m, Sr)
        M.mosaic_mask(M.MASK_WEIGHT, p, key, matrix_id, m, n_pad, 0,
                      dict(W=torch.from_numpy(W).cuda(), ldw=n, n=n, P=P, CT=CT, sign_words=sw, s_w=s_w, L=L,
                           S_idx=S_idx, S_val=S_val, Wp=Wp, J=J), M.GEMM_AUTO, ws)
        M.mosaic_device_status()
        assert np.array_equal(_u32(Wp)[:m], wo.W_masked), size
        assert np.array_equal(_u32(Wp)[m:], np.vstack(Po)), size
        assert np.array_equal(_u32(J), np.hstack(wo.J)), size
