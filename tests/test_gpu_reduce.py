"""Parity of the gated reducer (Eq. 1) kernel with the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_26744_gb300 import hdf
from paper_2606_26744_gb300 import workloads as W
from _util import TOL_BF16, TOL_F32_REDUCE, TOL_F32_REDUCE_BWD, exact_fraction, rowwise_rel, to64

pytestmark = pytest.mark.gpu


@pytest.fixture(params=["general", "cluster", "tile"])
def reduce_path(request):
    """Runs a test on each kernel of the reducer, chosen per call (the
    cluster and tile kernels take the bf16 shapes they support; the others
    fall back to the general kernel)."""
    return request.param


def _run(inp, **kw):
    H = inp["H"].cuda()
    N, m, d = H.shape
    a = torch.full((N, m), -7.0, device="cuda")
    y = hdf.hdf_gated_reduce(H, inp["Wf"].cuda(), inp["b"].cuda(), alpha_out=a, **kw)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    return y.cpu(), a.cpu()


@pytest.mark.parametrize("N,m,d,dtype,std", [
    (64, 4, 256, "f32", 0.02),      # tiny workload
    (37, 4, 2048, "bf16", 0.1),     # decode width, ragged token count
    (5, 4, 7168, "bf16", 0.1),      # large width: W_f read through L1
    (130, 2, 512, "bf16", 0.1),
    (9, 8, 256, "bf16", 0.1),
    (7, 3, 128, "f32", 0.1),
    (1, 4, 4096, "bf16", 0.1),
    (3, 1, 64, "bf16", 0.1),
    (4099, 4, 2048, "bf16", 0.1),   # many batches per cluster: ring and exchange buffers wrap
    (50, 1, 1024, "bf16", 0.1),
    (777, 2, 7168, "bf16", 0.1),
    (32, 4, 512, "bf16", 0.1),      # one whole 32-token tile, one 64-element block per CTA
    (33, 1, 512, "bf16", 0.1),      # a tile of one token after a full one
    (1000, 4, 7168, "bf16", 0.1),   # 56 k-blocks per CTA: the stage ring wraps in both passes
    (300, 4, 16384, "bf16", 0.1),   # the widest d: 16-token tiles in 8-CTA clusters
    (333, 2, 7168, "bf16", 0.1),    # m = 2 at the sweep width: 8-CTA clusters
    (70, 4, 256, "bf16", 0.1),      # the narrowest tile width: one plane per slice
    (50, 4, 9728, "bf16", 0.1),     # 8-CTA clusters, a three-plane tail box
    (20, 4, 9984, "bf16", 0.1),     # no tile geometry fits: m = 4 takes the general kernel
])
def test_reduce_parity(N, m, d, dtype, std, reduce_path):
    inp = W.make_reduce_inputs(N, m, d, dtype, std, seed=N * 131 + d)
    y, a = _run(inp, kernel=reduce_path)
    y_ref, a_ref = O.gated_reduce(to64(inp["H"]), to64(inp["Wf"]), to64(inp["b"]), out_dtype=dtype)
    tol = TOL_F32_REDUCE if dtype == "f32" else TOL_BF16
    assert rowwise_rel(to64(y), y_ref) <= tol
    np.testing.assert_allclose(to64(a), a_ref, rtol=0, atol=1e-4)
    if dtype == "bf16":
        assert exact_fraction(to64(y), y_ref) >= 0.99


def test_reduce_scale_offset_and_path_norm():
    N, m, d = 33, 4, 1024
    inp = W.make_reduce_inputs(N, m, d, "bf16", 0.1, seed=5)
    g = torch.Generator().manual_seed(9)
    pnw = (1 + 0.1 * torch.randn(m, d, generator=g)).to(torch.bfloat16)
    y, a = _run(inp, gate_scale=0.7, gate_offset=0.05, rms_eps=1e-3, path_norm_w=pnw.cuda(),
                path_norm_eps=1e-5)
    y_ref, a_ref = O.gated_reduce(to64(inp["H"]), to64(inp["Wf"]), to64(inp["b"]), rms_eps=1e-3,
                                  gate_scale=0.7, gate_offset=0.05, path_norm_w=to64(pnw),
                                  path_norm_eps=1e-5, out_dtype="bf16")
    assert rowwise_rel(to64(y), y_ref) <= TOL_BF16
    np.testing.assert_allclose(to64(a), a_ref, atol=1e-4)


def test_reduce_m1_identity_bit_exact():
    inp = W.make_reduce_inputs(19, 1, 512, "bf16", 0.1, seed=3)
    H = inp["H"].cuda()
    y = hdf.hdf_gated_reduce(H, None, None, alpha_override=torch.ones(19, 1, device="cuda"))
    assert torch.equal(y, H[:, 0, :])


def test_reduce_one_hot_selects_path_bit_exact(reduce_path):
    inp = W.make_reduce_inputs(21, 4, 2048, "bf16", 0.1, seed=4)
    H = inp["H"].cuda()
    for j in range(4):
        a = torch.zeros(21, 4, device="cuda")
        a[:, j] = 1
        y = hdf.hdf_gated_reduce(H, inp["Wf"].cuda(), inp["b"].cuda(), alpha_override=a, kernel=reduce_path)
        assert torch.equal(y, H[:, j, :])


def test_reduce_mean_pool_matches_oracle():
    inp = W.make_reduce_inputs(16, 4, 256, "f32", 0.02, seed=8)
    H = inp["H"].cuda()
    y = hdf.hdf_gated_reduce(H, None, None, alpha_override=torch.full((16, 4), 0.25, device="cuda"))
    np.testing.assert_allclose(to64(y), to64(inp["H"]).mean(axis=1), rtol=0, atol=1e-6)


def test_reduce_empty_is_noop():
    y = hdf.hdf_gated_reduce(torch.empty(0, 4, 256, device="cuda"), torch.empty(4, 1024, device="cuda"),
                             torch.zeros(4, device="cuda"))
    assert y.shape == (0, 256)


def test_reduce_sweep_width_sampled_rows(reduce_path):
    # reducer-only workload width (m=4, d=7168) at 65536 tokens, checked on sampled tokens
    N, m, d = 65536, 4, 7168
    inp = W.make_reduce_inputs(N, m, d, "bf16", 0.1, seed=11, device="cuda")
    y = hdf.hdf_gated_reduce(inp["H"], inp["Wf"], inp["b"], kernel=reduce_path)
    torch.cuda.synchronize()
    rows = torch.cat([torch.tensor([0, 1, 2, N - 2, N - 1]), torch.randperm(N, generator=torch.Generator().manual_seed(0))[:59]])
    Hs = to64(inp["H"][rows.cuda()])
    y_ref, _ = O.gated_reduce(Hs, to64(inp["Wf"]), to64(inp["b"]), out_dtype="bf16")
    assert rowwise_rel(to64(y[rows.cuda()]), y_ref) <= TOL_BF16
    assert exact_fraction(to64(y[rows.cuda()]), y_ref) >= 0.99


def test_reduce_rows_do_not_depend_on_the_call():
    """A token's y is the same bits whether it is reduced with many others or
    in a call of its own (the default kernel choice does not depend on the
    token count): a serving round that reduces only its new tokens matches the
    reduction of the whole context."""
    N, m, d = 5000, 4, 2048
    inp = W.make_reduce_inputs(N, m, d, "bf16", 0.1, seed=21, device="cuda")
    H, Wf, b = inp["H"], inp["Wf"], inp["b"]
    y_all = hdf.hdf_gated_reduce(H, Wf, b)
    for lo, hi in [(0, 1), (4095, 4101), (17, 60), (4990, 5000)]:
        y_part = hdf.hdf_gated_reduce(H[lo:hi].contiguous(), Wf, b)
        assert torch.equal(y_part.view(torch.int16), y_all[lo:hi].view(torch.int16))
    # an explicit kernel choice in one call does not change what the next
    # default call runs (no state is kept between calls)
    hdf.hdf_gated_reduce(H[:64].contiguous(), Wf, b, kernel="general")
    assert torch.equal(hdf.hdf_gated_reduce(H, Wf, b).view(torch.int16), y_all.view(torch.int16))


# ------------------------------------------------ gradient w.r.t. W_f and b
def _bwd_inputs(N, m, d, dtype, std, seed):
    inp = W.make_reduce_inputs(N, m, d, dtype, std, seed=seed)
    g = torch.Generator().manual_seed(seed + 7)
    dy = torch.randn((N, d), generator=g).to(inp["H"].dtype)
    b = torch.randn(m, generator=g) * 0.5
    return inp["H"], inp["Wf"], b, dy


@pytest.mark.parametrize("N,m,d,dtype,std", [
    (1, 4, 2048, "bf16", 0.1),      # one token
    (37, 4, 512, "bf16", 0.1),      # ragged token count
    (2048, 4, 2048, "bf16", 0.1),   # the decode workload's context
    (300, 2, 256, "bf16", 0.1),
    (100, 8, 128, "bf16", 0.1),
    (1001, 3, 384, "bf16", 0.05),
    (64, 4, 256, "f32", 0.02),      # the tiny workload
    (5, 1, 64, "f32", 0.3),
    (3, 4, 7168, "bf16", 0.1),      # the large width
])
def test_reduce_backward_parity(N, m, d, dtype, std):
    H, Wf, b, dy = _bwd_inputs(N, m, d, dtype, std, seed=4000 + N + m)
    dWf, db = hdf.hdf_gated_reduce_backward(H.cuda(), Wf.cuda(), b.cuda(), dy.cuda(), rms_eps=1e-6, gate_scale=1.0)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    dWf_ref, db_ref = O.gated_reduce_backward(to64(H), to64(Wf), to64(b), to64(dy), rms_eps=1e-6, gate_scale=1.0)
    assert dWf.shape == (m, m * d) and db.shape == (m,)
    err_w = rowwise_rel(to64(dWf), dWf_ref)
    err_b = np.abs(to64(db) - db_ref).max() / max(np.abs(db_ref).max(), 1e-30)
    assert err_w <= TOL_F32_REDUCE_BWD, f"dW_f row-normwise error {err_w}"
    assert err_b <= TOL_F32_REDUCE_BWD, f"db error {err_b}"


def test_reduce_backward_gate_scale_and_reproducible():
    H, Wf, b, dy = _bwd_inputs(513, 4, 1024, "bf16", 0.05, seed=4100)
    args = (H.cuda(), Wf.cuda(), b.cuda(), dy.cuda())
    dW1, db1 = hdf.hdf_gated_reduce_backward(*args, rms_eps=1e-3, gate_scale=0.7)
    dW2, db2 = hdf.hdf_gated_reduce_backward(*args, rms_eps=1e-3, gate_scale=0.7)
    torch.cuda.synchronize()
    assert torch.equal(dW1, dW2) and torch.equal(db1, db2)   # fixed summation order
    dWf_ref, db_ref = O.gated_reduce_backward(to64(H), to64(Wf), to64(b), to64(dy), rms_eps=1e-3, gate_scale=0.7)
    assert rowwise_rel(to64(dW1), dWf_ref) <= TOL_F32_REDUCE_BWD
    assert np.abs(to64(db1) - db_ref).max() <= TOL_F32_REDUCE_BWD * np.abs(db_ref).max()


def test_reduce_backward_no_tokens_gives_zero_gradients():
    m, d = 4, 256
    dWf = torch.full((m, m * d), 7.0, device="cuda")
    db = torch.full((m,), 7.0, device="cuda")
    H = torch.empty((0, m, d), dtype=torch.bfloat16, device="cuda")
    hdf.hdf_gated_reduce_backward(H, torch.zeros((m, m * d), dtype=torch.bfloat16, device="cuda"),
                                  torch.zeros(m, device="cuda"), torch.empty((0, d), dtype=torch.bfloat16,
                                                                             device="cuda"), dWf=dWf, db=db)
    torch.cuda.synchronize()
    assert not dWf.any() and not db.any()
