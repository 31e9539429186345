"""Parity of the serve and large workloads at their full sizes.

    serve  32 sequences, ragged T_i ~ U[512, 8192], m4 d4096, 1 layer 32x128,
           F11008, V65536, bf16
    large  8 sequences x T16384, m4 d7168, 2 layers 56x128, F18432, V129280,
           bf16, log-softmax on

The GPU runs the whole batch exactly as bench.py does (reduce, draft block
with its two-stream context path, LM head).  A full fp64 oracle of these
steps would take hours, so each stage is checked stage by stage: the
oracle of a stage is fed the GPU's own output of the stage before (exact
bf16 values, read from the draft workspace through
hdf_draft_block_workspace_layout), on every row of the cheap stages, on 512
sampled rows of the context projection and on every head of two full
sequences of the attention.  Two full sequences also run end to end
through the oracle from the raw inputs (reduce, block forward, LM head).
The block's attention and MLP are those of the last layer."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2606_26744_gb300 import hdf
from paper_2606_26744_gb300 import workloads as W
from _util import TOL_BF16, check_tokens, exact_fraction, rowwise_rel, to64

pytestmark = pytest.mark.gpu

SAMPLED_ROWS = 512


@pytest.fixture(scope="module", params=["serve", "large"])
def step(request):
    cfg = W.CONFIGS[request.param]
    seed = {"serve": 4003, "large": 4004}[cfg.name]
    inp = W.make_draft_inputs(cfg, seed, device="cuda")
    lens = inp["ctx_lens"]
    n_ctx, max_ctx, B, batch = sum(lens), max(lens), cfg.block, cfg.batch
    drafter = hdf.Drafter(inp["weights"], n_heads=cfg.n_heads, head_dim=cfg.head_dim, rope_theta=cfg.rope_theta,
                          rope_max_pos=max_ctx + B, norm_eps=cfg.norm_eps)
    y = hdf.hdf_gated_reduce(inp["H"], inp["Wf"], inp["b"])
    cu = inp["cu_ctx"].cuda()
    anchor = inp["anchor"].cuda()
    ws = torch.empty(drafter.workspace_size(batch, B, n_ctx, max_ctx), dtype=torch.uint8, device="cuda")
    h = drafter.hdf_draft_block(y, cu, anchor, block=B, max_ctx=max_ctx, ws=ws)
    tok, zmax, ls = hdf.hdf_lm_head_argmax(h, inp["weights"]["lm_head"], logsoftmax=cfg.logsoftmax)
    torch.cuda.synchronize()
    assert hdf.device_status() == 0
    views = drafter.workspace_views(ws, batch, B, n_ctx, max_ctx)
    cu_np = inp["cu_ctx"].cpu().numpy().astype(np.int64)
    # the two sequences checked in full: the longest and the shortest
    order = np.argsort(lens, kind="stable")
    full = sorted({int(order[-1]), int(order[0])})
    yield dict(cfg=cfg, inp=inp, y=y, h=h, tok=tok, ls=ls, v=views, cu=cu_np, lens=lens, full=full,
               rng=np.random.default_rng(seed))
    del inp, y, h, ws, views
    torch.cuda.empty_cache()


def _rows(st, n):
    """n sampled context rows: both ends of every checked sequence plus random ones."""
    cu, rng = st["cu"], st["rng"]
    edge = [int(cu[i]) for i in st["full"]] + [int(cu[i + 1]) - 1 for i in st["full"]]
    rest = rng.choice(int(cu[-1]), size=n - len(edge), replace=False)
    return np.unique(np.concatenate([edge, rest]))


def _pos(cu, t):
    b = np.searchsorted(cu, t, side="right") - 1
    return t - cu[b]


def test_reduce_sampled_rows(step):
    t = _rows(step, SAMPLED_ROWS)
    ti = torch.as_tensor(t, device="cuda")
    inp = step["inp"]
    y_ref, _ = O.gated_reduce(to64(inp["H"][ti]), to64(inp["Wf"]), to64(inp["b"]), out_dtype="bf16")
    got = to64(step["y"][ti])
    assert rowwise_rel(got, y_ref) <= TOL_BF16
    assert exact_fraction(got, y_ref) >= 0.99


def test_context_norm_sampled_rows(step):
    cfg, t = step["cfg"], _rows(step, SAMPLED_ROWS)
    ti = torch.as_tensor(t, device="cuda")
    c_ref = O.store(O.rmsnorm(to64(step["y"][ti]), to64(step["inp"]["weights"]["ctx_norm"]), cfg.norm_eps), "bf16")
    got = to64(step["v"]["c"][ti])
    assert rowwise_rel(got, c_ref) <= TOL_BF16
    assert exact_fraction(got, c_ref) >= 0.99


def test_context_projection_sampled_rows(step):
    """K_c, V_c of the last layer on 512 rows of the whole context, from the
    GPU's normed rows c, at each row's position in its sequence."""
    cfg, t = step["cfg"], _rows(step, SAMPLED_ROWS)
    ti = torch.as_tensor(t, device="cuda")
    lw = step["inp"]["weights"]["layers"][-1]
    K_ref, V_ref = O.context_kv(to64(step["v"]["c"][ti]), to64(lw["wk"]), to64(lw["wv"]), _pos(step["cu"], t),
                                n_heads=cfg.n_heads, head_dim=cfg.head_dim, theta=cfg.rope_theta, act_dtype="bf16")
    assert rowwise_rel(to64(step["v"]["k_ctx"][ti]), K_ref) <= TOL_BF16
    assert rowwise_rel(to64(step["v"]["v_ctx"][ti]), V_ref) <= TOL_BF16


def test_attention_every_head_of_two_full_sequences(step):
    """Non-causal attention of the block's queries over all T_i context keys
    and the B block keys, every head, from the GPU's Q, K, V."""
    cfg, cu, v = step["cfg"], step["cu"], step["v"]
    B, hd = cfg.block, cfg.head_dim
    for i in step["full"]:
        rows = slice(i * B, (i + 1) * B)
        ctx = slice(int(cu[i]), int(cu[i + 1]))
        Q = to64(v["q"][rows])
        Kall = np.concatenate([to64(v["k_ctx"][ctx]), to64(v["k_blk"][rows])])
        Vall = np.concatenate([to64(v["v_ctx"][ctx]), to64(v["v_blk"][rows])])
        ref = np.empty((B, cfg.d))
        for hh in range(cfg.n_heads):
            cols = slice(hh * hd, (hh + 1) * hd)
            ref[:, cols] = O.softmax_attention(Q[:, cols], Kall[:, cols], Vall[:, cols])
        err = rowwise_rel(to64(v["o"][rows]), O.store(ref, "bf16"))
        assert err <= TOL_BF16, f"sequence {i} (T = {step['lens'][i]}): attention error {err}"


def test_mlp_and_final_norm_every_row(step):
    cfg, v = step["cfg"], step["v"]
    w = step["inp"]["weights"]
    lw = w["layers"][-1]
    x = to64(v["x"])
    act_ref = O.store(O.silu(x @ to64(lw["wg"]).T) * (x @ to64(lw["wu"]).T), "bf16")
    assert rowwise_rel(to64(v["act"]), act_ref) <= TOL_BF16
    h_ref = O.store(O.rmsnorm(to64(v["h"]), to64(w["final_norm"]), cfg.norm_eps), "bf16")
    assert rowwise_rel(to64(step["h"]), h_ref) <= TOL_BF16
    assert exact_fraction(to64(step["h"]), h_ref) >= 0.99


def test_lm_head_every_row(step):
    """Drafts bit-exact against the oracle's argmax of the GPU's h_out
    (outside the 1e-3 tie band); log-softmax within the bf16 bar."""
    cfg = step["cfg"]
    lm = O.lm_head(to64(step["h"]), to64(step["inp"]["weights"]["lm_head"]), logsoftmax=cfg.logsoftmax)
    ties = check_tokens(step["tok"].cpu().numpy(), lm["z"])
    print(f"[{cfg.name}] LM head rows in the tie band: {ties}/{lm['z'].shape[0]}")
    if cfg.logsoftmax:
        assert rowwise_rel(to64(step["ls"]), lm["logsoftmax"]) <= TOL_BF16


def test_two_full_sequences_end_to_end(step):
    """The oracle's whole step for two full sequences from the raw inputs:
    reduce (Eq. 1), block forward, LM head.  h_out within the bf16 bar;
    drafts equal outside a tie band of 6 sigma of the logit noise that bf16
    re-rounding at every storage point leaves (measured here)."""
    cfg, inp, cu, B = step["cfg"], step["inp"], step["cu"], step["cfg"].block
    seqs = step["full"]
    w = inp["weights"]
    anchors = inp["anchor"].cpu().numpy()
    w64 = {k: to64(w[k]) for k in ("mask_vec", "ctx_norm", "final_norm")}
    w64["embed"] = to64(w["embed"][torch.as_tensor(anchors[seqs], device=w["embed"].device)])
    w64["layers"] = [{k: to64(t) for k, t in lw.items()} for lw in w["layers"]]
    idx = np.concatenate([np.arange(cu[i], cu[i + 1]) for i in seqs])
    sub_cu = np.concatenate([[0], np.cumsum([cu[i + 1] - cu[i] for i in seqs])])
    y_ref, _ = O.gated_reduce(to64(inp["H"][torch.as_tensor(idx, device="cuda")]), to64(inp["Wf"]), to64(inp["b"]),
                              out_dtype="bf16")
    h_ref = O.draft_block(w64, y_ref, sub_cu.tolist(), list(range(len(seqs))), block=B, n_heads=cfg.n_heads,
                          head_dim=cfg.head_dim, rope_theta=cfg.rope_theta, norm_eps=cfg.norm_eps, act_dtype="bf16")
    rows = np.concatenate([np.arange(i * B, (i + 1) * B) for i in seqs])
    h_gpu = to64(step["h"][torch.as_tensor(rows, device="cuda")])
    err = rowwise_rel(h_gpu, h_ref)
    assert err <= TOL_BF16, f"h_out error {err}"
    W_lm = to64(w["lm_head"])
    z_ref = O.lm_head(h_ref, W_lm)["z"]
    z_gpu_h = O.lm_head(h_gpu, W_lm)["z"]
    sigma = float(np.sqrt(np.mean((z_gpu_h - z_ref) ** 2)))
    band = max(1e-3, 6 * sigma)
    ties = check_tokens(step["tok"].cpu().numpy()[rows], z_ref, band=band)
    print(f"[{cfg.name}] sequences {seqs}: h_out err {err:.2e}, logit noise sigma {sigma:.2e}, "
          f"rows in band {ties}/{len(rows)}")
