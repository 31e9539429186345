"""Incremental (serving) form of the drafter: the context K/V cache.

hdf_ctx_append projects only the rows accepted since the last round into a
per-layer K_c / V_c cache; hdf_draft_block_cached runs the block forward over
it.  K_c[t] and V_c[t] depend only on row t's reduced state and on t, so a
context appended over any number of rounds must give exactly (bit for bit)
the output of hdf_draft_block over the whole context.  The cache starts
filled with NaN, so a read of a row that was never appended would show.
The warm path is also checked against the fp64 oracle directly."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_26744_gb300 import hdf
from paper_2606_26744_gb300 import workloads as W
from _util import TOL_BF16, TOL_F32_TF32, check_tokens, rowwise_rel, to64

pytestmark = pytest.mark.gpu


def _to_cuda(w):
    out = {k: v.cuda() for k, v in w.items() if k != "layers"}
    out["layers"] = [{k: v.cuda() for k, v in lw.items()} for lw in w["layers"]]
    return out


def _weights64(w):
    out = {k: to64(v) for k, v in w.items() if k != "layers"}
    out["layers"] = [{k: to64(v) for k, v in lw.items()} for lw in w["layers"]]
    return out


def _rounds(lens, n_rounds, rng):
    """Split every sequence's context into n_rounds consecutive pieces (some
    empty): pieces[r][i] rows of sequence i arrive in round r."""
    pieces = []
    for T in lens:
        cuts = np.sort(rng.integers(0, T + 1, size=n_rounds - 1)) if T > 0 else np.zeros(n_rounds - 1, int)
        edges = np.concatenate([[0], cuts, [T]])
        pieces.append(np.diff(edges))
    return np.array(pieces).T  # [rounds, batch]


def _setup(cfg, seed, lens, capacity_extra=7, device="cuda"):
    cfg = W.scaled(cfg, batch=len(lens), ctx_len=max(lens))
    inp = W.make_draft_inputs(cfg, seed)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    inp = dict(inp)
    inp["ctx_lens"] = list(lens)
    inp["cu_ctx"] = torch.tensor(cu)
    inp.update(W.make_reduce_inputs(int(cu[-1]), cfg.m, cfg.d, cfg.dtype, cfg.wf_std, seed=seed))
    max_ctx = max(lens)
    wc = _to_cuda(inp["weights"])
    drafter = hdf.Drafter(wc, n_heads=cfg.n_heads, head_dim=cfg.head_dim, rope_theta=cfg.rope_theta,
                          rope_max_pos=max_ctx + capacity_extra + cfg.block, norm_eps=cfg.norm_eps)
    return cfg, inp, drafter, wc, cu, max_ctx


def _cold(drafter, cfg, inp, max_ctx):
    H = inp["H"].cuda()
    y = hdf.hdf_gated_reduce(H, inp["Wf"].cuda(), inp["b"].cuda())
    h = drafter.hdf_draft_block(y, inp["cu_ctx"].cuda(), inp["anchor"].cuda(), block=cfg.block, max_ctx=max_ctx)
    return y, h


def _nan_cache(drafter, batch, capacity):
    cache = drafter.new_cache(batch, capacity, "cuda")
    cache.k.fill_(float("nan"))
    cache.v.fill_(float("nan"))
    return cache


def _append_rounds(drafter, cfg, inp, cu, pieces, cache, pad_rows=0):
    """Each round reduces the new rows' residuals and appends them."""
    H = inp["H"].cuda()
    Wf, b = inp["Wf"].cuda(), inp["b"].cuda()
    batch = len(cu) - 1
    done = np.zeros(batch, dtype=np.int64)
    for r in range(pieces.shape[0]):
        idx = []
        for i in range(batch):
            idx.extend(range(cu[i] + done[i], cu[i] + done[i] + pieces[r, i]))
        done += pieces[r]
        cu_new = torch.tensor(np.concatenate([[0], np.cumsum(pieces[r])]).astype(np.int32), device="cuda")
        n = len(idx)
        rows = torch.tensor(idx, dtype=torch.long, device="cuda")
        H_new = torch.empty((n + pad_rows,) + tuple(H.shape[1:]), dtype=H.dtype, device="cuda")
        H_new[:n] = H[rows]
        if pad_rows:
            H_new[n:] = torch.randn_like(H_new[n:], dtype=torch.float32).to(H.dtype)  # never appended
        y_new = hdf.hdf_gated_reduce(H_new, Wf, b)
        drafter.hdf_ctx_append(y_new, cu_new, cache, block=cfg.block)
    return done


def _check_warm_equals_cold(cfg_base, seed, lens, n_rounds, pad_rows=0, check_oracle=True):
    rng = np.random.default_rng(seed)
    cfg, inp, drafter, wc, cu, max_ctx = _setup(cfg_base, seed, lens)
    y, h_cold = _cold(drafter, cfg, inp, max_ctx)
    cache = _nan_cache(drafter, cfg.batch, max_ctx + 7)
    pieces = _rounds(lens, n_rounds, rng)
    _append_rounds(drafter, cfg, inp, cu, pieces, cache, pad_rows=pad_rows)
    anchor = inp["anchor"].cuda()
    h_warm = drafter.hdf_draft_block_cached(cache, anchor, block=cfg.block, max_ctx=max_ctx)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    assert cache.len.cpu().tolist() == list(lens)
    assert torch.equal(h_warm.view(torch.int16 if h_warm.dtype == torch.bfloat16 else torch.int32),
                       h_cold.view(torch.int16 if h_cold.dtype == torch.bfloat16 else torch.int32)), \
        f"warm/cold differ: max |diff| {float((h_warm.float() - h_cold.float()).abs().max())}"
    # rows past each sequence's length were never written
    for i, T in enumerate(lens):
        assert torch.isnan(cache.k[:, i, T:].float()).all() and torch.isnan(cache.v[:, i, T:].float()).all()
    if check_oracle:
        act = cfg.dtype
        w64 = _weights64(inp["weights"])
        y_ref, _ = O.gated_reduce(to64(inp["H"]), to64(inp["Wf"]), to64(inp["b"]), out_dtype=act)
        h_ref = O.draft_block(w64, y_ref, inp["cu_ctx"].tolist(), inp["anchor"].tolist(), block=cfg.block,
                              n_heads=cfg.n_heads, head_dim=cfg.head_dim, rope_theta=cfg.rope_theta,
                              norm_eps=cfg.norm_eps, act_dtype=act)
        tol = TOL_F32_TF32 if act == "f32" else TOL_BF16
        assert rowwise_rel(to64(h_warm), h_ref) <= tol
        tok, _, _ = hdf.hdf_lm_head_argmax(h_warm, wc["lm_head"])
        check_tokens(tok.cpu().numpy(), O.lm_head(to64(h_warm), w64["lm_head"])["z"])
    return drafter, cache, h_cold


def test_warm_equals_cold_tiny_fp32():
    _check_warm_equals_cold(W.CONFIGS["tiny"], 2001, [64], n_rounds=5)


def test_warm_equals_cold_ragged_two_layers():
    cfg = W.DraftConfig("ragged", m=4, d=512, block=16, n_layers=2, n_heads=4, head_dim=128, ffn=1024,
                        vocab=4096, batch=5, ctx_len=300)
    _check_warm_equals_cold(cfg, 2002, [0, 1, 63, 65, 300], n_rounds=4)


def test_warm_equals_cold_decode_widths():
    """The decode workload's widths, context appended over 6 rounds."""
    _check_warm_equals_cold(W.CONFIGS["decode"], 2003, [2048], n_rounds=6)


def test_warm_equals_cold_head_dim_64():
    cfg = W.DraftConfig("hd64", m=4, d=256, block=8, n_layers=1, n_heads=4, head_dim=64, ffn=512,
                        vocab=2048, batch=3, ctx_len=257)
    _check_warm_equals_cold(cfg, 2004, [10, 130, 257], n_rounds=3)


def test_padded_rows_are_skipped():
    """Rows past cu_new[batch] (a graph captured for the largest round) are
    reduced and normed but never appended."""
    cfg = W.DraftConfig("pad", m=4, d=512, block=16, n_layers=1, n_heads=4, head_dim=128, ffn=1024,
                        vocab=4096, batch=3, ctx_len=200)
    _check_warm_equals_cold(cfg, 2005, [200, 77, 5], n_rounds=3, pad_rows=37, check_oracle=False)


def test_append_in_cuda_graph():
    """One captured append (fixed row bound, device-side counts) replayed
    round after round with new rows gives the cold result."""
    cfg_base = W.DraftConfig("graph", m=4, d=512, block=16, n_layers=2, n_heads=4, head_dim=128, ffn=1024,
                             vocab=4096, batch=4, ctx_len=160)
    lens = [160, 99, 3, 128]
    cfg, inp, drafter, wc, cu, max_ctx = _setup(cfg_base, 2006, lens)
    y, h_cold = _cold(drafter, cfg, inp, max_ctx)
    cache = _nan_cache(drafter, cfg.batch, max_ctx + 7)
    pieces = _rounds(lens, 5, np.random.default_rng(2006))
    bound = int(pieces.sum(axis=1).max()) + 3
    y_new = torch.zeros((bound, cfg.d), dtype=y.dtype, device="cuda")
    cu_new = torch.zeros(cfg.batch + 1, dtype=torch.int32, device="cuda")
    ws = torch.empty(drafter.append_workspace_size(cfg.batch, cfg.block, bound), dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    # one eager append (every row skipped) into a scratch cache first, so
    # that no first-use setup happens under capture
    scratch = drafter.new_cache(cfg.batch, max_ctx + 7, "cuda", zero=True)
    drafter.hdf_ctx_append(y_new, cu_new, scratch, block=cfg.block, ws=ws)
    torch.cuda.synchronize()
    assert scratch.len.cpu().tolist() == [0] * cfg.batch
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        drafter.hdf_ctx_append(y_new, cu_new, cache, block=cfg.block, ws=ws, stream=s)
    cache.len.zero_()  # capture does not run the work
    done = np.zeros(cfg.batch, dtype=np.int64)
    for r in range(pieces.shape[0]):
        idx = [cu[i] + done[i] + j for i in range(cfg.batch) for j in range(pieces[r, i])]
        done += pieces[r]
        y_new.zero_()
        if idx:
            y_new[:len(idx)] = y[torch.tensor(idx, device="cuda")]
        cu_new.copy_(torch.tensor(np.concatenate([[0], np.cumsum(pieces[r])]).astype(np.int32)))
        torch.cuda.synchronize()
        with torch.cuda.stream(s):
            g.replay()
        s.synchronize()
    h_warm = drafter.hdf_draft_block_cached(cache, inp["anchor"].cuda(), block=cfg.block, max_ctx=max_ctx)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    assert cache.len.cpu().tolist() == lens
    assert torch.equal(h_warm.view(torch.int16), h_cold.view(torch.int16))


def test_capacity_overflow_is_skipped_and_recorded():
    """Rows that would pass the capacity are not written (the next
    sequence's rows stay untouched), len stops at the capacity and the
    device status word records the violation."""
    cfg = W.DraftConfig("ovf", m=4, d=256, block=8, n_layers=1, n_heads=2, head_dim=128, ffn=512,
                        vocab=1024, batch=2, ctx_len=12)
    cfg, inp, drafter, wc, cu, max_ctx = _setup(cfg, 2007, [12, 4])
    cache = _nan_cache(drafter, 2, 8)
    assert hdf.device_status(reset=True) == 0
    y = hdf.hdf_gated_reduce(inp["H"].cuda(), inp["Wf"].cuda(), inp["b"].cuda())
    drafter.hdf_ctx_append(y, inp["cu_ctx"].cuda(), cache, block=cfg.block)
    torch.cuda.synchronize()
    assert hdf.device_status(reset=True) == 8
    assert cache.len.cpu().tolist() == [8, 4]
    assert not torch.isnan(cache.k[0, 0, :8].float()).any()
    assert not torch.isnan(cache.k[0, 1, :4].float()).any()
    assert torch.isnan(cache.k[0, 1, 4:].float()).all()
    assert hdf.device_status() == 0


def test_length_above_max_ctx_is_recorded():
    cfg = W.DraftConfig("lenchk", m=4, d=256, block=8, n_layers=1, n_heads=2, head_dim=128, ffn=512,
                        vocab=1024, batch=2, ctx_len=40)
    cfg, inp, drafter, wc, cu, max_ctx = _setup(cfg, 2008, [40, 20])
    cache = drafter.new_cache(2, 48, "cuda", zero=True)
    y = hdf.hdf_gated_reduce(inp["H"].cuda(), inp["Wf"].cuda(), inp["b"].cuda())
    drafter.hdf_ctx_append(y, inp["cu_ctx"].cuda(), cache, block=cfg.block)
    torch.cuda.synchronize()
    assert hdf.device_status(reset=True) == 0
    h = drafter.hdf_draft_block_cached(cache, inp["anchor"].cuda(), block=cfg.block, max_ctx=32)  # 40 > 32
    torch.cuda.synchronize()
    assert hdf.device_status(reset=True) == 8
    assert torch.isfinite(h.float()).all()


def test_large_workload_full_size_warm_equals_cold():
    """The large workload (m4 d7168 T16384 B16, 2 layers 56x128, F18432,
    batch 8) at full size: the last 20 rows of every sequence arrive in four
    rounds of five (a mean accepted length of four, plus the bonus token)."""
    cfg = W.CONFIGS["large"]
    seed = 2009
    inp = W.make_draft_inputs(cfg, seed, device="cuda")
    lens = inp["ctx_lens"]
    max_ctx = max(lens)
    drafter = hdf.Drafter(inp["weights"], n_heads=cfg.n_heads, head_dim=cfg.head_dim, rope_theta=cfg.rope_theta,
                          rope_max_pos=max_ctx + 64 + cfg.block, norm_eps=cfg.norm_eps)
    cu = inp["cu_ctx"].numpy() if inp["cu_ctx"].device.type == "cpu" else inp["cu_ctx"].cpu().numpy()
    y = hdf.hdf_gated_reduce(inp["H"], inp["Wf"], inp["b"])
    anchor = inp["anchor"].cuda()
    h_cold = drafter.hdf_draft_block(y, torch.as_tensor(cu, device="cuda"), anchor, block=cfg.block,
                                     max_ctx=max_ctx)
    torch.cuda.synchronize()
    del inp["H"]
    cache = drafter.new_cache(cfg.batch, max_ctx + 64, "cuda")
    pieces = np.array([[T - 20 for T in lens]] + [[5] * len(lens)] * 4)
    done = np.zeros(len(lens), dtype=np.int64)
    for r in range(pieces.shape[0]):
        idx = torch.cat([torch.arange(cu[i] + done[i], cu[i] + done[i] + pieces[r, i]) for i in range(len(lens))])
        done += pieces[r]
        cu_new = torch.tensor(np.concatenate([[0], np.cumsum(pieces[r])]).astype(np.int32), device="cuda")
        drafter.hdf_ctx_append(y[idx.cuda()], cu_new, cache, block=cfg.block)
    h_warm = drafter.hdf_draft_block_cached(cache, anchor, block=cfg.block, max_ctx=max_ctx)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    assert cache.len.cpu().tolist() == list(lens)
    assert torch.equal(h_warm.view(torch.int16), h_cold.view(torch.int16))


def _check_round_equals_two_calls(cfg_base, seed, lens, n_rounds, pad_rows=0):
    """hdf_draft_round (the first block path beside the append) against
    hdf_ctx_append + hdf_draft_block_cached, round after round: the same
    h_out, cache rows and lengths, bit for bit; after the last round both
    equal the cold step."""
    rng = np.random.default_rng(seed)
    cfg, inp, drafter, wc, cu, max_ctx = _setup(cfg_base, seed, lens)
    y, h_cold = _cold(drafter, cfg, inp, max_ctx)
    cap = max_ctx + 7
    c_round = _nan_cache(drafter, cfg.batch, cap)
    c_two = _nan_cache(drafter, cfg.batch, cap)
    c_round.len.zero_()
    c_two.len.zero_()
    pieces = _rounds(lens, n_rounds, rng)
    anchor = inp["anchor"].cuda()
    bits = torch.int16 if h_cold.dtype == torch.bfloat16 else torch.int32
    done = np.zeros(cfg.batch, dtype=np.int64)
    for r in range(pieces.shape[0]):
        idx = [cu[i] + done[i] + j for i in range(cfg.batch) for j in range(pieces[r, i])]
        done += pieces[r]
        n = len(idx)
        y_new = torch.zeros((n + pad_rows, cfg.d), dtype=y.dtype, device="cuda")
        if n:
            y_new[:n] = y[torch.tensor(idx, device="cuda")]
        if pad_rows:
            y_new[n:] = torch.randn_like(y_new[n:], dtype=torch.float32).to(y.dtype)  # never appended
        cu_new = torch.tensor(np.concatenate([[0], np.cumsum(pieces[r])]).astype(np.int32), device="cuda")
        h_round = drafter.hdf_draft_round(y_new, cu_new, c_round, anchor, block=cfg.block, max_ctx=max_ctx)
        drafter.hdf_ctx_append(y_new, cu_new, c_two, block=cfg.block)
        h_two = drafter.hdf_draft_block_cached(c_two, anchor, block=cfg.block, max_ctx=max_ctx)
        torch.cuda.synchronize()
        assert hdf.device_status() == 0
        assert torch.equal(c_round.len, c_two.len)
        assert torch.equal(h_round.view(bits), h_two.view(bits)), f"round {r}: round / two calls differ"
        for i, T in enumerate(done):
            assert torch.equal(c_round.k[:, i, :T].view(bits), c_two.k[:, i, :T].view(bits))
            assert torch.equal(c_round.v[:, i, :T].view(bits), c_two.v[:, i, :T].view(bits))
    assert c_round.len.cpu().tolist() == list(lens)
    assert torch.equal(h_round.view(bits), h_cold.view(bits))


def test_round_equals_two_calls_decode_widths():
    _check_round_equals_two_calls(W.CONFIGS["decode"], 2010, [2048], n_rounds=5)


def test_round_equals_two_calls_ragged_two_layers():
    cfg = W.DraftConfig("ragged", m=4, d=512, block=16, n_layers=2, n_heads=4, head_dim=128, ffn=1024,
                        vocab=4096, batch=5, ctx_len=300)
    _check_round_equals_two_calls(cfg, 2011, [0, 1, 63, 65, 300], n_rounds=4, pad_rows=9)


def test_round_equals_two_calls_tiny_fp32():
    _check_round_equals_two_calls(W.CONFIGS["tiny"], 2012, [64], n_rounds=4)


def test_round_in_cuda_graph():
    """One captured round (fixed row bound, device-side counts: the fork and
    join of the block path are captured too) replayed round after round
    gives the cold result."""
    cfg_base = W.DraftConfig("graph", m=4, d=512, block=16, n_layers=2, n_heads=4, head_dim=128, ffn=1024,
                             vocab=4096, batch=4, ctx_len=160)
    lens = [160, 99, 3, 128]
    cfg, inp, drafter, wc, cu, max_ctx = _setup(cfg_base, 2013, lens)
    y, h_cold = _cold(drafter, cfg, inp, max_ctx)
    cache = _nan_cache(drafter, cfg.batch, max_ctx + 7)
    pieces = _rounds(lens, 5, np.random.default_rng(2013))
    bound = int(pieces.sum(axis=1).max()) + 3
    y_new = torch.zeros((bound, cfg.d), dtype=y.dtype, device="cuda")
    cu_new = torch.zeros(cfg.batch + 1, dtype=torch.int32, device="cuda")
    anchor = inp["anchor"].cuda()
    h = torch.empty((cfg.batch * cfg.block, cfg.d), dtype=y.dtype, device="cuda")
    ws = torch.empty(drafter.round_workspace_size(cfg.batch, cfg.block, bound, max_ctx), dtype=torch.uint8,
                     device="cuda")
    s = torch.cuda.Stream()
    # one eager round (every row skipped) on a scratch cache first, so that
    # no first-use setup happens under capture
    scratch = drafter.new_cache(cfg.batch, max_ctx + 7, "cuda", zero=True)
    drafter.hdf_draft_round(y_new, cu_new, scratch, anchor, block=cfg.block, max_ctx=max_ctx, h_out=h, ws=ws)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        drafter.hdf_draft_round(y_new, cu_new, cache, anchor, block=cfg.block, max_ctx=max_ctx, h_out=h, ws=ws,
                                stream=s)
    cache.len.zero_()  # capture does not run the work
    done = np.zeros(cfg.batch, dtype=np.int64)
    for r in range(pieces.shape[0]):
        idx = [cu[i] + done[i] + j for i in range(cfg.batch) for j in range(pieces[r, i])]
        done += pieces[r]
        y_new.zero_()
        if idx:
            y_new[:len(idx)] = y[torch.tensor(idx, device="cuda")]
        cu_new.copy_(torch.tensor(np.concatenate([[0], np.cumsum(pieces[r])]).astype(np.int32)))
        torch.cuda.synchronize()
        with torch.cuda.stream(s):
            g.replay()
        s.synchronize()
    assert hdf.device_status() == 0
    assert cache.len.cpu().tolist() == lens
    assert torch.equal(h.view(torch.int16), h_cold.view(torch.int16))
