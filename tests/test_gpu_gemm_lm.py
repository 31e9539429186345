"""Parity of the tcgen05 GEMM paths: the generic fc reducer (Table 1's
comparison path) and the LM head (logits, argmax, log-softmax)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_26744_gb300 import hdf
from paper_2606_26744_gb300 import workloads as W
from _util import TOL_BF16, TOL_F32_TF32, check_tokens, rowwise_rel, to64

pytestmark = pytest.mark.gpu


def _rand(shape, std, dtype, seed, device="cpu"):
    g = torch.Generator(device=device).manual_seed(seed)
    return (torch.randn(shape, generator=g, device=device) * std).to(dtype)


@pytest.mark.parametrize("N,m,d,dtype", [(200, 4, 256, torch.bfloat16), (129, 4, 384, torch.bfloat16),
                                         (64, 4, 256, torch.float32), (1, 2, 128, torch.bfloat16),
                                         (1000, 4, 512, torch.bfloat16)])
def test_fc_reduce_parity(N, m, d, dtype):
    H = _rand((N, m, d), 1.0, dtype, 1 + N)
    Wfc = _rand((d, m * d), 0.02, dtype, 2 + d)
    y = hdf.hdf_fc_reduce(H.cuda(), Wfc.cuda())
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    out = "bf16" if dtype == torch.bfloat16 else "f32"
    ref = O.store(to64(H).reshape(N, m * d) @ to64(Wfc).T, out)
    assert rowwise_rel(to64(y), ref) <= (TOL_BF16 if out == "bf16" else TOL_F32_TF32)


def test_fc_reduce_large_width_sampled_rows():
    N, m, d = 1024, 4, 7168
    H = _rand((N, m, d), 1.0, torch.bfloat16, 3, "cuda")
    Wfc = _rand((d, m * d), 0.02, torch.bfloat16, 4, "cuda")
    y = hdf.hdf_fc_reduce(H, Wfc)
    torch.cuda.synchronize()
    rows = torch.tensor([0, 127, 128, 511, 1023, 700, 33, 901])
    ref = O.store(to64(H[rows.cuda()]).reshape(len(rows), m * d) @ to64(Wfc).T, "bf16")
    assert rowwise_rel(to64(y[rows.cuda()]), ref) <= TOL_BF16


@pytest.mark.parametrize("N,m,d_in,d_out,dtype", [
    (300, 4, 200, 640, torch.bfloat16),    # narrower input, 128-wide tiles, K tail of 32
    (64, 2, 96, 256, torch.float32),       # tf32, wider output
    (7, 4, 4096, 7168, torch.bfloat16),    # a few rows, target 4096 -> drafter 7168
])
def test_fc_reduce_unequal_widths(N, m, d_in, d_out, dtype):
    """The fc fallback when the drafter width differs from the target's
    (Sec. 2.2): W_fc [d_out, m * d_in], against the oracle's fc_reduce."""
    H = _rand((N, m, d_in), 1.0, dtype, 5 + N)
    Wfc = _rand((d_out, m * d_in), 0.02, dtype, 6 + d_out)
    y = hdf.hdf_fc_reduce(H.cuda(), Wfc.cuda())
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    assert y.shape == (N, d_out)
    out = "bf16" if dtype == torch.bfloat16 else "f32"
    ref = O.fc_reduce(to64(H), to64(Wfc), out)
    assert rowwise_rel(to64(y), ref) <= (TOL_BF16 if out == "bf16" else TOL_F32_TF32)


def test_fc_reduce_7168_to_4096_sampled_rows():
    """Target width 7168 into a 4096-wide drafter on 1024 tokens (CTA-pair
    tiles), every column of 8 sampled rows against the oracle."""
    N, m, d_in, d_out = 1024, 4, 7168, 4096
    H = _rand((N, m, d_in), 1.0, torch.bfloat16, 7, "cuda")
    Wfc = _rand((d_out, m * d_in), 0.02, torch.bfloat16, 8, "cuda")
    y = hdf.hdf_fc_reduce(H, Wfc)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    rows = torch.tensor([0, 255, 256, 511, 1023, 700, 33, 901], device="cuda")
    ref = O.fc_reduce(to64(H[rows]), to64(Wfc), "bf16")
    assert rowwise_rel(to64(y[rows]), ref) <= TOL_BF16


@pytest.mark.parametrize("M,d,V,dtype,it,ls", [
    (8, 256, 1024, torch.float32, 1.0, True),     # tiny workload shape
    (16, 2048, 32768, torch.bfloat16, 1.0, False),  # decode shape
    (16, 2048, 32768, torch.bfloat16, 0.5, True),
    (37, 512, 1000, torch.bfloat16, 1.0, True),   # ragged rows and vocab
    (200, 256, 4099, torch.bfloat16, 2.0, True),
    (128, 7168, 129280, torch.bfloat16, 1.0, True),  # large workload LM head (every row)
])
def test_lm_head_parity(M, d, V, dtype, it, ls):
    dev = "cuda"
    h = _rand((M, d), 1.0, dtype, 10 + M, dev)
    Wl = _rand((V, d), 0.02, dtype, 20 + V, dev)
    tok, zmax, lsm = hdf.hdf_lm_head_argmax(h, Wl, inv_temp=it, logsoftmax=ls)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    ref = O.lm_head(to64(h), to64(Wl), inv_temp=it, logsoftmax=ls)
    ties = check_tokens(tok.cpu().numpy(), ref["z"])
    assert ties <= max(2, M // 20)
    np.testing.assert_allclose(to64(zmax), ref["zmax"], rtol=0, atol=2e-3)
    if ls:
        assert rowwise_rel(to64(lsm), ref["logsoftmax"]) <= TOL_BF16
        assert np.abs(to64(lsm) - ref["logsoftmax"]).max() <= 1e-2


def test_lm_head_ties_pick_lowest_index():
    d, V = 256, 512
    h = torch.zeros(3, d, dtype=torch.bfloat16)
    h[:, 0] = 1.0
    Wl = torch.zeros(V, d, dtype=torch.bfloat16)
    Wl[[7, 300, 301], 0] = 2.0      # exact three-way tie across two vocabulary tiles
    tok, zmax, _ = hdf.hdf_lm_head_argmax(h.cuda(), Wl.cuda())
    assert tok.cpu().tolist() == [7, 7, 7]
    assert torch.all(zmax.cpu() == 2.0)


def test_accept_len_bit_exact():
    g = torch.Generator().manual_seed(0)
    B, batch, V = 16, 300, 50
    tok = torch.randint(0, V, (batch * B,), generator=g, dtype=torch.int32)
    plan = torch.randint(0, B, (batch,), generator=g).tolist()
    plan[:3] = [0, B - 1, 5]
    draft = tok.view(batch, B)[:, 1:]
    tgt = W.make_targets(draft, plan, V, seed=1)
    acc = hdf.hdf_accept_len(tok.cuda()[1:], tgt.cuda(), n_draft=B - 1, draft_stride=B, batch=batch)
    ref = O.accept_len(draft.numpy(), tgt.numpy())
    assert np.array_equal(acc.cpu().numpy(), ref)
    assert np.array_equal(ref, np.array(plan))
    # no drafts -> nothing accepted
    acc0 = hdf.hdf_accept_len(tok.cuda(), tgt.cuda(), n_draft=0, draft_stride=B, batch=batch)
    assert int(acc0.abs().sum()) == 0


def test_rope_table_matches_definition():
    hd, P = 128, 16500
    c, s = hdf.hdf_rope_table(10000.0, hd, P, "cuda")
    pos = np.array([0, 1, 2, 1000, 8191, 16399, 16499])
    i = np.arange(hd // 2)
    ang = pos[:, None] * 10000.0 ** (-2.0 * i / hd)[None, :]
    np.testing.assert_allclose(to64(c[pos]), np.cos(ang), rtol=0, atol=2e-7)
    np.testing.assert_allclose(to64(s[pos]), np.sin(ang), rtol=0, atol=2e-7)


@pytest.mark.parametrize("batch,nd,ds,ts", [(1000, 15, 16, 15), (129, 47, 50, 47), (1 << 17, 7, 7, 9)])
def test_accept_len_staged_rows(batch, nd, ds, ts):
    """Ragged CTAs of 128 sequences, strides above n_draft, the largest n_draft."""
    g = torch.Generator().manual_seed(batch + nd)
    draft = torch.randint(0, 1000, (batch, ds), generator=g, dtype=torch.int32)
    keep = torch.randint(0, nd + 1, (batch,), generator=g)
    target = torch.randint(0, 1000, (batch, ts), generator=g, dtype=torch.int32)
    k = torch.arange(ts)[None, :]
    target = torch.where(k < keep[:, None], torch.nn.functional.pad(draft, (0, max(0, ts - ds)))[:, :ts], (target % 997) + 1001)
    acc = hdf.hdf_accept_len(draft.cuda(), target.cuda(), n_draft=nd, draft_stride=ds, batch=batch)
    ref = O.accept_len(draft[:, :nd].numpy(), target[:, :nd].numpy())
    assert np.array_equal(acc.cpu().numpy(), ref)
    assert np.array_equal(ref, keep.numpy())
