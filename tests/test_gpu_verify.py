"""Temperature-1 verification (speculative sampling) on the GPU: accept
lengths and next tokens must equal the oracle's exactly."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_26744_gb300 import hdf

pytestmark = pytest.mark.gpu


def _case(batch, nd, V, seed, agree=0.7):
    rng = np.random.default_rng(seed)
    logits_p = rng.standard_normal((batch, nd + 1, V)) * 2
    p = np.exp(logits_p - logits_p.max(-1, keepdims=True))
    p = (p / p.sum(-1, keepdims=True)).astype(np.float32)
    # draft distribution: a mix of the target and an independent one, so acceptance varies
    logits_q = rng.standard_normal((batch, nd, V)) * 2
    q = np.exp(logits_q - logits_q.max(-1, keepdims=True))
    q = q / q.sum(-1, keepdims=True)
    q = (agree * p[:, :nd] + (1 - agree) * q).astype(np.float32)
    draft = np.stack([[rng.choice(V, p=q[i, k] / q[i, k].sum()) for k in range(nd)] for i in range(batch)]).astype(np.int32) \
        if nd > 0 else np.zeros((batch, 0), np.int32)
    u = rng.integers(0, 2 ** 32, size=(batch, nd), dtype=np.uint64).astype(np.uint32)
    r = rng.integers(0, 2 ** 32, size=(batch,), dtype=np.uint64).astype(np.uint32)
    return p, q, draft, u, r


def _gpu(p, q, draft, u, r):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    acc, nxt = hdf.hdf_accept_sample(t(p), t(q), t(draft), t(u.view(np.int32)), t(r.view(np.int32)))
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    return acc.cpu().numpy(), nxt.cpu().numpy()


@pytest.mark.parametrize("batch,nd,V", [(33, 15, 1000), (8, 15, 32768), (5, 7, 1001), (3, 15, 129280), (17, 1, 64)])
def test_accept_sample_matches_oracle(batch, nd, V):
    p, q, draft, u, r = _case(batch, nd, V, seed=batch * 7 + V)
    acc, nxt = _gpu(p, q, draft, u, r)
    ref_acc, ref_nxt = O.accept_sample(p, q, draft, u, r)
    np.testing.assert_array_equal(acc, ref_acc)
    np.testing.assert_array_equal(nxt, ref_nxt)
    assert 0 < acc.mean() < nd or nd == 1      # the cases exercise both outcomes


def test_accept_sample_special_cases():
    V, nd = 50, 4
    p, _, _, _, _ = _case(1, nd, V, seed=3)
    u = np.full((1, nd), 2 ** 32 - 1, np.uint32)
    acc, nxt = _gpu(p, p[:, :nd].copy(), np.zeros((1, nd), np.int32), u, np.array([0], np.uint32))
    assert acc[0] == nd and nxt[0] == O.accept_sample(p, p[:, :nd], np.zeros((1, nd), int), u, np.array([0]))[1][0]
    q1 = np.zeros((1, nd, V), np.float32); q1[:, :, 2] = 1
    p1 = np.zeros((1, nd + 1, V), np.float32); p1[:, :, 5] = 1
    acc, nxt = _gpu(p1, q1, np.full((1, nd), 2, np.int32), np.zeros((1, nd), np.uint32), np.array([77], np.uint32))
    assert acc[0] == 0 and nxt[0] == 5
    acc, _ = _gpu(p, p[:, :nd].copy(), np.array([[0, 1, V, 2]], np.int32), u, np.array([0], np.uint32))
    assert acc[0] == 2                           # an id outside the vocabulary is rejected


def test_accept_sample_without_drafts_samples_p():
    p, _, _, _, r = _case(6, 0, 300, seed=9)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    acc, nxt = hdf.hdf_accept_sample(t(p), None, torch.zeros((6, 0), dtype=torch.int32, device="cuda"), None,
                                     t(r.view(np.int32)))
    ref_acc, ref_nxt = O.accept_sample(p, np.zeros((6, 0, 300), np.float32), np.zeros((6, 0), int),
                                       np.zeros((6, 0), np.uint32), r)
    np.testing.assert_array_equal(acc.cpu().numpy(), ref_acc)
    np.testing.assert_array_equal(nxt.cpu().numpy(), ref_nxt)


def test_accept_sample_reads_drafts_with_a_stride():
    # drafts straight out of the LM head's tok layout: row i at tok + 1 + i*B
    batch, nd, V = 4, 7, 500
    B = nd + 1
    p, q, draft, u, r = _case(batch, nd, V, seed=21)
    tok = np.zeros((batch, B), np.int32); tok[:, 1:] = draft
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    tok_d = t(tok)
    acc, nxt = hdf.hdf_accept_sample(t(p), t(q), tok_d.view(-1)[1:].as_strided((batch, nd), (B, 1)),
                                     t(u.view(np.int32)), t(r.view(np.int32)))
    ref_acc, ref_nxt = O.accept_sample(p, q, draft, u, r)
    np.testing.assert_array_equal(acc.cpu().numpy(), ref_acc)
    np.testing.assert_array_equal(nxt.cpu().numpy(), ref_nxt)
