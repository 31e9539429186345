"""KL distillation target (Eq. 2, Sec. 2.3) on the GPU against the fp64 oracle."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_26744_gb300 import hdf
from paper_2606_26744_gb300 import workloads as W
from _util import to64

pytestmark = pytest.mark.gpu


def _log_softmax_f32(z, t_kd):
    s = torch.log_softmax(torch.as_tensor(z, dtype=torch.float64) / t_kd, dim=1)
    return s.to(torch.float32)


def _oracle_kl(ls_t, ls_s, t_kd):
    # the inputs are log-softmax rows at t_kd: their softmax at temperature 1
    # is the same distribution, so the oracle runs at 1 and the T^2 factor is applied here
    return t_kd * t_kd * O.kl_distill(to64(ls_t), to64(ls_s), 1.0)


@pytest.mark.parametrize("rows,V,t_kd", [(2, 1000, 1.0), (4, 32768, 2.0), (3, 1001, 0.5), (16, 129280, 1.0),
                                         (1, 8193, 1.5)])
def test_kl_matches_oracle(rows, V, t_kd):
    g = torch.Generator().manual_seed(rows * 31 + V)
    zt = torch.randn(rows, V, generator=g) * 3
    zs = zt + torch.randn(rows, V, generator=g)
    ls_t, ls_s = _log_softmax_f32(zt, t_kd), _log_softmax_f32(zs, t_kd)
    kl_rows, kl_mean = hdf.hdf_kl_distill(ls_t.cuda(), ls_s.cuda(), t_kd=t_kd)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    ref_rows = np.array([O.kl_distill(to64(ls_t[r:r + 1]), to64(ls_s[r:r + 1]), 1.0) for r in range(rows)])
    np.testing.assert_allclose(to64(kl_rows), ref_rows, rtol=1e-4, atol=1e-6)
    np.testing.assert_allclose(float(kl_mean[0]), _oracle_kl(ls_t, ls_s, t_kd), rtol=1e-4, atol=1e-6)


def test_kl_identical_is_zero_and_scales_with_t_squared():
    g = torch.Generator().manual_seed(3)
    ls = _log_softmax_f32(torch.randn(4, 5000, generator=g), 1.0).cuda()
    _, m = hdf.hdf_kl_distill(ls, ls, t_kd=1.0)
    assert float(m[0]) == 0.0                       # KL(p || p) = 0 exactly
    ls_s = _log_softmax_f32(torch.randn(4, 5000, generator=g), 1.0).cuda()
    _, m1 = hdf.hdf_kl_distill(ls, ls_s, t_kd=1.0)
    _, m2 = hdf.hdf_kl_distill(ls, ls_s, t_kd=2.0)
    assert float(m1[0]) > 0
    assert float(m2[0]) == 4 * float(m1[0])         # same rows, the T^2 factor alone


def test_kl_infinities():
    ls_t = torch.log(torch.tensor([[0.5, 0.5, 0.0, 0.0]], dtype=torch.float32))   # p = (.5, .5, 0, 0)
    ls_s = torch.log(torch.tensor([[0.25, 0.25, 0.25, 0.25]], dtype=torch.float32))
    rows, _ = hdf.hdf_kl_distill(ls_t.cuda(), ls_s.cuda())
    np.testing.assert_allclose(float(rows[0]), np.log(2.0), rtol=1e-6)            # teacher zeros contribute 0
    ls_s2 = torch.log(torch.tensor([[1.0, 0.0, 0.0, 0.0]], dtype=torch.float32))  # q = 0 where p > 0
    rows2, _ = hdf.hdf_kl_distill(ls_t.cuda(), ls_s2.cuda())
    assert float(rows2[0]) == float("inf")


def test_kl_empty_is_noop():
    r, m = hdf.hdf_kl_distill(torch.empty(0, 64, device="cuda"), torch.empty(0, 64, device="cuda"))
    assert r.shape == (0,)


def test_kl_teacher_from_path_mean_and_lm_head():
    """Teacher = LM head on the path-mean residual (the reducer with alpha = 1/m),
    student = LM head on other hidden rows; both log-softmax at T_KD from the GPU
    LM head, KL on the GPU, against the oracle fed the same bf16 hidden rows."""
    cfg = W.CONFIGS["tiny"]
    P, t_kd = 2, 2.0
    g = torch.Generator().manual_seed(11)
    H = torch.randn(P, 4, 256, generator=g).to(torch.bfloat16)
    W_lm = (torch.randn(1024, 256, generator=g) * 0.02).to(torch.bfloat16)
    h_s = torch.randn(P, 256, generator=g).to(torch.bfloat16)
    h_t = hdf.hdf_gated_reduce(H.cuda(), None, None, alpha_override=torch.full((P, 4), 0.25, device="cuda"))
    _, _, ls_t = hdf.hdf_lm_head_argmax(h_t, W_lm.cuda(), inv_temp=1 / t_kd, logsoftmax=True)
    _, _, ls_s = hdf.hdf_lm_head_argmax(h_s.cuda(), W_lm.cuda(), inv_temp=1 / t_kd, logsoftmax=True)
    _, m = hdf.hdf_kl_distill(ls_t, ls_s, t_kd=t_kd)
    torch.cuda.synchronize()
    # stage-wise: the oracle gets the GPU's bf16 teacher rows (exact values) and computes the rest in fp64
    h_mean_ref, _ = O.gated_reduce(to64(H), None, None, alpha_override=np.full((P, 4), 0.25), out_dtype="bf16")
    np.testing.assert_array_equal(to64(h_t), h_mean_ref)
    zt = O.lm_head(to64(h_t), to64(W_lm))["z"]
    zs = O.lm_head(to64(h_s), to64(W_lm))["z"]
    ref = O.kl_distill(zt, zs, t_kd)
    np.testing.assert_allclose(float(m[0]), ref, rtol=2e-3, atol=1e-6)


# -------------------------------------------------- Eq. 3: L = L_CE + alpha L_KL
def _loss_inputs(batch, block, P, V, seed, unsup=0.2):
    """Student and teacher log-softmax rows at temperature 1 (fp32) and labels
    with a share of unsupervised (-1) positions."""
    g = torch.Generator().manual_seed(seed)
    zs = torch.randn(batch * block, V, generator=g, dtype=torch.float64) * 3
    zt = torch.stack([zs[i * block + 1:i * block + 1 + P] for i in range(batch)]) + \
        torch.randn(batch, P, V, generator=g, dtype=torch.float64)
    ls_s = torch.log_softmax(zs, dim=-1).float()
    ls_t = torch.log_softmax(zt, dim=-1).float()
    labels = torch.randint(0, V, (batch, block - 1), generator=g, dtype=torch.int32)
    labels[torch.rand(batch, block - 1, generator=g) < unsup] = -1
    return ls_t, ls_s, labels


def _check_loss(ls_t, ls_s, labels, block, t_kd, alpha, out):
    loss, ce_rows, kl_rows = out
    ref = O.draft_loss(to64(ls_t), to64(ls_s), labels.numpy(), block=block, P=ls_t.shape[1], t_kd=t_kd, alpha=alpha)
    ce = to64(ce_rows).reshape(-1)
    sup = labels.numpy().reshape(-1) >= 0
    assert np.all(np.isnan(ce[~sup]))
    np.testing.assert_allclose(ce[sup], ref["ce_rows"][sup], rtol=1e-5, atol=1e-5)
    np.testing.assert_allclose(to64(kl_rows).reshape(-1), ref["kl_rows"], rtol=1e-4, atol=1e-6)
    np.testing.assert_allclose(to64(loss), [ref["loss"], ref["ce"], ref["kl"]], rtol=1e-4, atol=1e-6)


@pytest.mark.parametrize("batch,block,P,V,t_kd,alpha", [
    (1, 8, 2, 1024, 1.0, 0.1),        # tiny workload's block and vocabulary
    (1, 16, 2, 32768, 2.0, 0.2),      # decode
    (3, 5, 4, 1001, 0.5, 1.0),        # ragged vocabulary (no 16-byte rows), P = block - 1
    (8, 16, 2, 129280, 1.0, 0.15),    # large workload
    (2, 16, 0, 4099, 1.0, 0.1),       # CE alone
    (5, 3, 1, 8193, 3.0, 0.0),        # a chunk of one vector past 8192
])
def test_draft_loss_matches_oracle(batch, block, P, V, t_kd, alpha):
    ls_t, ls_s, labels = _loss_inputs(batch, block, P, V, seed=batch * 1000 + V)
    out = hdf.hdf_draft_loss(ls_t.cuda() if P else None, ls_s.cuda(), labels.cuda(), block=block, t_kd=t_kd,
                             alpha=alpha)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    _check_loss(ls_t, ls_s, labels, block, t_kd, alpha, out)


def test_draft_loss_exact_properties():
    """KL exactly 0 for a teacher equal to the student's first P draft rows;
    two calls give the same bits; a label past the vocabulary is left out and
    recorded in the device status word; no supervised position gives L_CE 0."""
    batch, block, P, V = 4, 16, 2, 50000
    _, ls_s, labels = _loss_inputs(batch, block, P, V, seed=9)
    ls_t = torch.stack([ls_s[i * block + 1:i * block + 1 + P] for i in range(batch)])
    d_t, d_s, d_l = ls_t.cuda(), ls_s.cuda(), labels.cuda()
    a = hdf.hdf_draft_loss(d_t, d_s, d_l, block=block, t_kd=2.0, alpha=0.5)
    b = hdf.hdf_draft_loss(d_t, d_s, d_l, block=block, t_kd=2.0, alpha=0.5)
    torch.cuda.synchronize()
    assert float(a[0][2]) == 0.0 and torch.all(a[2] == 0)
    assert torch.equal(a[0], b[0]) and torch.equal(a[1].nan_to_num(), b[1].nan_to_num())
    assert float(a[0][0]) == float(a[0][1])                     # L = L_CE when L_KL = 0
    assert hdf.device_status() == 0
    bad = d_l.clone()
    bad[1, 3] = V                                              # outside the vocabulary
    loss, ce_rows, _ = hdf.hdf_draft_loss(d_t, d_s, bad, block=block, t_kd=2.0, alpha=0.5)
    torch.cuda.synchronize()
    assert hdf.load().hdf_device_status(1) != 0                 # recorded (and cleared)
    assert torch.isnan(ce_rows[1, 3])
    keep = labels.clone()
    keep[1, 3] = -1
    ref = O.draft_loss(to64(ls_t), to64(ls_s), keep.numpy(), block=block, P=P, t_kd=2.0, alpha=0.5)
    np.testing.assert_allclose(float(loss[1]), ref["ce"], rtol=1e-5)
    none = torch.full_like(d_l, -1)
    loss0, _, _ = hdf.hdf_draft_loss(d_t, d_s, none, block=block, t_kd=2.0, alpha=0.5)
    torch.cuda.synchronize()
    assert float(loss0[1]) == 0.0
    assert hdf.device_status() == 0


def test_draft_loss_from_the_lm_heads():
    """The whole objective from hidden rows: the student is the GPU LM head on
    draft hidden rows, the teacher the LM head on the path-mean residual
    (hdf_gated_reduce with alpha = 1/m), both log-softmax at temperature 1;
    checked against the oracle fed the same bf16 hidden rows."""
    batch, block, P, d, V, m = 2, 8, 2, 256, 1024, 4
    g = torch.Generator().manual_seed(21)
    W_lm = (torch.randn(V, d, generator=g) * 0.05).to(torch.bfloat16)
    h_s = torch.randn(batch * block, d, generator=g).to(torch.bfloat16)
    H = torch.randn(batch * P, m, d, generator=g).to(torch.bfloat16)
    labels = torch.randint(0, V, (batch, block - 1), generator=g, dtype=torch.int32)
    h_t = hdf.hdf_gated_reduce(H.cuda(), None, None, alpha_override=torch.full((batch * P, m), 1 / m, device="cuda"))
    _, _, ls_t = hdf.hdf_lm_head_argmax(h_t, W_lm.cuda(), inv_temp=1.0, logsoftmax=True)
    _, _, ls_s = hdf.hdf_lm_head_argmax(h_s.cuda(), W_lm.cuda(), inv_temp=1.0, logsoftmax=True)
    loss, _, _ = hdf.hdf_draft_loss(ls_t.view(batch, P, V), ls_s, labels.cuda(), block=block, t_kd=2.0, alpha=0.2)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    zt = O.lm_head(to64(h_t), to64(W_lm))["z"].reshape(batch, P, V)
    zs = O.lm_head(to64(h_s), to64(W_lm))["z"]
    ref = O.draft_loss(zt, zs, labels.numpy(), block=block, P=P, t_kd=2.0, alpha=0.2)
    np.testing.assert_allclose(to64(loss), [ref["loss"], ref["ce"], ref["kl"]], rtol=2e-3, atol=1e-5)
