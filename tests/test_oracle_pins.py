"""Pins for the fp64 oracle: closed forms, invariants, special cases and the
paper's printed numbers.  None of these re-types an oracle formula; each is
chosen so that a plausible slip (a dropped term, a wrong sign or index, a
transposed operand) fails at least one of them."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


# --------------------------------------------------------------------------
# storage rounding
# --------------------------------------------------------------------------

def test_bf16_round_matches_torch_conversion():
    # torch's float32 -> bfloat16 cast is an independent round-to-nearest-even.
    x32 = torch.randn(200000, dtype=torch.float32) * 10
    # add exact ties: values halfway between two bf16 neighbours
    base = torch.randn(1000, dtype=torch.float32).to(torch.bfloat16).float()
    ulp = torch.ldexp(torch.ones_like(base), torch.frexp(base).exponent - 8)
    ties = base + ulp / 2
    x32 = torch.cat([x32, ties])
    ref = x32.to(torch.bfloat16).double().numpy()
    got = O.bf16_round(x32.double().numpy())
    assert np.array_equal(ref, got)


def _bf16_nearest(y, exact):
    """y holds bfloat16 values (each survives torch's float32 -> bfloat16 cast
    unchanged) within half a bfloat16 ulp of the exact values."""
    y = np.asarray(y, np.float64)
    survives = np.array_equal(torch.from_numpy(y).float().to(torch.bfloat16).double().numpy(), y)
    half_ulp = np.ldexp(1.0, np.frexp(np.asarray(exact, np.float64))[1] - 9)
    return survives and bool(np.all(np.abs(y - exact) <= half_ulp))


def test_reducer_and_fc_outputs_are_rounded_where_they_are_stored():
    # y of Eq. 1 and the fc output are stored in bf16 (the precision contract):
    # every value is the bf16 nearest to the exact one, and random data is
    # not bf16-exact, so the rounding shows
    r = np.random.default_rng(81)
    H = r.standard_normal((6, 3, 16))
    Wf, b = 0.1 * r.standard_normal((3, 48)), r.standard_normal(3)
    y, _ = O.gated_reduce(H, Wf, b, out_dtype="bf16")
    y64, _ = O.gated_reduce(H, Wf, b, out_dtype="f64")
    assert _bf16_nearest(y, y64) and not np.array_equal(y, y64)
    W = r.standard_normal((8, 48))
    f, f64 = O.fc_reduce(H, W, out_dtype="bf16"), O.fc_reduce(H, W, out_dtype="f64")
    assert _bf16_nearest(f, f64) and not np.array_equal(f, f64)


def test_store_f32_is_float32_rounding():
    x = rng.standard_normal(1000)
    assert np.array_equal(O.store(x, "f32"), x.astype(np.float32).astype(np.float64))


# --------------------------------------------------------------------------
# Eq. 1 reducer
# --------------------------------------------------------------------------

def _H(N, m, d):
    return rng.standard_normal((N, m, d))


def test_reduce_m1_identity_under_unit_gate():
    H = O.bf16_round(_H(5, 1, 16))
    y, _ = O.gated_reduce(H, np.zeros((1, 16)), np.zeros(1),
                          alpha_override=np.ones((5, 1)), out_dtype="bf16")
    assert np.array_equal(y, H[:, 0, :])


def test_reduce_one_hot_selects_path():
    H = O.bf16_round(_H(6, 4, 32))
    for j in range(4):
        a = np.zeros((6, 4))
        a[:, j] = 1.0
        y, _ = O.gated_reduce(H, np.zeros((4, 128)), np.zeros(4),
                              alpha_override=a, out_dtype="bf16")
        assert np.array_equal(y, H[:, j, :])


def test_reduce_equal_weights_is_path_mean():
    H = _H(7, 4, 24)
    y, _ = O.gated_reduce(H, np.zeros((4, 96)), np.zeros(4),
                          alpha_override=np.full((7, 4), 0.25), out_dtype="f64")
    np.testing.assert_allclose(y, H.mean(axis=1), rtol=1e-15, atol=1e-15)


def test_reduce_zero_gate_weight_gives_sigmoid_of_bias():
    # sigmoid(0) = 1/2, sigmoid(ln 3) = 3/4, sigmoid(-ln 3) = 1/4, sigmoid(ln 9) = 9/10
    b = np.array([0.0, math.log(3.0), -math.log(3.0), math.log(9.0)])
    H = _H(3, 4, 8)
    y, a = O.gated_reduce(H, np.zeros((4, 32)), b, out_dtype="f64")
    expect_a = np.array([0.5, 0.75, 0.25, 0.9])
    np.testing.assert_allclose(a, np.broadcast_to(expect_a, (3, 4)), rtol=1e-14)
    np.testing.assert_allclose(
        y, 0.5 * H[:, 0] + 0.75 * H[:, 1] + 0.25 * H[:, 2] + 0.9 * H[:, 3], rtol=1e-13)


def test_reduce_gate_reads_path_major_vec_with_sign_and_scale():
    # H = +1 everywhere except one entry -1 => mean(H^2) = 1, r = 1 (eps 0).
    # W_f picks that single entry for gate 2 with weight 1: logit_2 = s*(-1) + b_2.
    m, d = 4, 8
    p, e = 2, 5
    H = np.ones((1, m, d))
    H[0, p, e] = -1.0
    Wf = np.zeros((m, m * d))
    Wf[2, p * d + e] = 1.0
    b = np.array([0.0, 0.0, 0.25, 0.0])
    s = 1.7
    g = O.gate_logits(H, Wf, b, rms_eps=0.0, gate_scale=s)
    np.testing.assert_allclose(g[0], [0.0, 0.0, -s + 0.25, 0.0], rtol=0, atol=1e-15)
    # the transposed (element-major) vec would have read a +1 entry
    assert g[0, 2] < 0


def test_reduce_rms_uses_all_md_entries_and_eps():
    # H = c everywhere -> x~ = c / sqrt(c^2 + eps); W_f = 1/(md) sums x~ once.
    m, d, c, eps = 2, 4, 3.0, 7.0
    H = np.full((1, m, d), c)
    Wf = np.full((m, m * d), 1.0 / (m * d))
    g = O.gate_logits(H, Wf, np.zeros(m), rms_eps=eps)
    np.testing.assert_allclose(g[0], c / math.sqrt(c * c + eps), rtol=1e-15)  # 3/4


def test_reduce_scale_invariance():
    H = _H(4, 4, 16)
    Wf = rng.standard_normal((4, 64)) * 0.1
    b = rng.standard_normal(4)
    y1, a1 = O.gated_reduce(H, Wf, b, rms_eps=0.0, out_dtype="f64")
    y2, a2 = O.gated_reduce(3.5 * H, Wf, b, rms_eps=0.0, out_dtype="f64")
    np.testing.assert_allclose(a1, a2, rtol=1e-13)
    np.testing.assert_allclose(y2, 3.5 * y1, rtol=1e-12)


def _reduce_loss(H, Wf, b, dy, s, eps):
    y, _ = O.gated_reduce(H, Wf, b, rms_eps=eps, gate_scale=s, gate_offset=0.25, out_dtype="f64")
    return float(np.sum(np.asarray(dy) * y))


def test_reduce_backward_matches_central_differences():
    """dL/dW_f and dL/db of L = sum dy . y (Eq. 1, forward oracle in fp64)
    against central differences of that loss, entry by entry; the offset
    (0.25 here) must not enter."""
    N, m, d, s, eps = 5, 3, 8, 1.7, 1e-3
    H = rng.standard_normal((N, m, d))
    Wf = rng.standard_normal((m, m * d)) * 0.3
    b = rng.standard_normal(m) * 0.5
    dy = rng.standard_normal((N, d))
    dWf, db = O.gated_reduce_backward(H, Wf, b, dy, rms_eps=eps, gate_scale=s)
    assert dWf.shape == (m, m * d) and db.shape == (m,)
    h = 1e-6
    fd = np.zeros_like(Wf)
    for j in range(m):
        for k in range(m * d):
            Wp, Wm = Wf.copy(), Wf.copy()
            Wp[j, k] += h
            Wm[j, k] -= h
            fd[j, k] = (_reduce_loss(H, Wp, b, dy, s, eps) - _reduce_loss(H, Wm, b, dy, s, eps)) / (2 * h)
    fdb = np.zeros(m)
    for j in range(m):
        bp, bm = b.copy(), b.copy()
        bp[j] += h
        bm[j] -= h
        fdb[j] = (_reduce_loss(H, Wf, bp, dy, s, eps) - _reduce_loss(H, Wf, bm, dy, s, eps)) / (2 * h)
    scale = max(np.abs(fd).max(), 1.0)
    assert np.abs(dWf - fd).max() <= 1e-7 * scale
    assert np.abs(db - fdb).max() <= 1e-7 * max(np.abs(fdb).max(), 1.0)


def test_reduce_backward_zero_cotangent_and_bias_is_gate_sum():
    H = _H(6, 4, 16)
    Wf = rng.standard_normal((4, 64)) * 0.1
    b = rng.standard_normal(4)
    dWf, db = O.gated_reduce_backward(H, Wf, b, np.zeros((6, 16)))
    assert not dWf.any() and not db.any()
    # W_f = 0: every gate is sigmoid(b), so dL/db_j = sigmoid'(b_j) * sum_t dy_t . H_tj
    dy = rng.standard_normal((6, 16))
    _, db0 = O.gated_reduce_backward(H, np.zeros((4, 64)), b, dy)
    sg = 1.0 / (1.0 + np.exp(-b))
    np.testing.assert_allclose(db0, sg * (1 - sg) * np.einsum("nd,njd->j", dy, H), rtol=1e-13)


def test_reduce_gates_are_not_a_softmax():
    H = _H(16, 4, 32)
    _, a = O.gated_reduce(H, rng.standard_normal((4, 128)) * 0.1, np.zeros(4), out_dtype="f64")
    assert np.all((a > 0) & (a < 1))
    assert np.max(np.abs(a.sum(axis=1) - 1.0)) > 1e-3


def test_reduce_offset_and_scale_terms():
    H = _H(3, 4, 8)
    Wf = rng.standard_normal((4, 32))
    b = rng.standard_normal(4)
    _, a0 = O.gated_reduce(H, Wf, b, out_dtype="f64")
    _, a1 = O.gated_reduce(H, Wf, b, gate_offset=0.125, out_dtype="f64")
    np.testing.assert_allclose(a1 - a0, 0.125, rtol=0, atol=1e-15)
    _, az = O.gated_reduce(H, Wf, b, gate_scale=0.0, out_dtype="f64")
    np.testing.assert_allclose(az, np.broadcast_to(1 / (1 + np.exp(-b)), az.shape), rtol=1e-14)


def test_reduce_path_norm_constant_magnitude_paths():
    # path j = +-c_j -> RMSNorm_gamma(H_j) = sign * gamma_j (eps 0)
    m, d = 3, 6
    c = np.array([0.5, 2.0, 7.0])
    sign = np.where(rng.standard_normal((1, m, d)) > 0, 1.0, -1.0)
    H = sign * c[None, :, None]
    gamma = rng.standard_normal((m, d))
    a = np.array([[0.2, 0.3, 0.9]])
    y, _ = O.gated_reduce(H, np.zeros((m, m * d)), np.zeros(m), alpha_override=a,
                          path_norm_w=gamma, path_norm_eps=0.0, out_dtype="f64")
    expect = (a[0, :, None] * sign[0] * gamma).sum(axis=0)
    np.testing.assert_allclose(y[0], expect, rtol=1e-14)


def test_table1_parameter_counts():
    g = json.load(open(os.path.join(GOLDEN, "table1_reducer_params.json")))
    m, d = g["m"], g["d"]
    hc = O.hc_gate_param_count(m, d)
    fc = O.fc_param_count(m, d)
    assert hc == 65536
    assert hc // 1000 == g["hc_gate_thousands_printed"]   # printed "65K"
    assert fc // 10**6 == g["fc_millions_printed"]         # printed "67M"
    assert fc // hc == d // m == 1024       # "three orders of magnitude fewer"


# --------------------------------------------------------------------------
# drafter pieces
# --------------------------------------------------------------------------

def test_rmsnorm_constant_vector():
    x = np.where(rng.standard_normal(10) > 0, 4.0, -4.0)
    w = rng.standard_normal(10)
    np.testing.assert_allclose(O.rmsnorm(x, w, 0.0), np.sign(x) * w, rtol=1e-15)


def test_rmsnorm_eps_inside_the_square_root():
    # a constant vector c normalises to c / sqrt(c^2 + eps) * w; with eps far
    # above c^2 that is about c / sqrt(eps), ten times c / (|c| + eps) here
    c, eps = 1e-3, 1e-2
    w = np.random.default_rng(95).standard_normal(6)
    np.testing.assert_allclose(O.rmsnorm(np.full(6, c), w, eps), c / math.sqrt(c * c + eps) * w, rtol=1e-14)


def test_rope_head_dim_two_is_plain_rotation():
    x = np.array([[[1.0, 0.0]], [[0.0, 1.0]]])       # [n=2, heads=1, hd=2]
    p = np.array([0.3, 1.1])
    out = O.rope(x, p, theta=10000.0)
    np.testing.assert_allclose(out[0, 0], [math.cos(0.3), math.sin(0.3)], rtol=1e-15)
    np.testing.assert_allclose(out[1, 0], [-math.sin(1.1), math.cos(1.1)], rtol=1e-15)


def test_rope_second_pair_frequency():
    # hd = 4, pair i = 1 turns at theta^(-2/4) = 1/10 for theta = 100
    x = np.array([[[0.0, 0.0, 1.0, 0.0]]])
    out = O.rope(x, np.array([5.0]), theta=100.0)
    np.testing.assert_allclose(out[0, 0], [0, 0, math.cos(0.5), math.sin(0.5)], atol=1e-15)


def test_rope_position_zero_identity_and_norm():
    x = rng.standard_normal((3, 2, 8))
    np.testing.assert_allclose(O.rope(x, np.zeros(3), 10000.0), x, rtol=0, atol=0)
    y = O.rope(x, np.array([3.0, 77.0, 1234.0]), 10000.0)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-14)


def test_rope_scores_depend_on_relative_position_only():
    q = rng.standard_normal((1, 1, 16))
    k = rng.standard_normal((1, 1, 16))
    s1 = (O.rope(q, [40.0], 1e4) * O.rope(k, [13.0], 1e4)).sum()
    s2 = (O.rope(q, [527.0], 1e4) * O.rope(k, [500.0], 1e4)).sum()
    np.testing.assert_allclose(s1, s2, rtol=1e-10)


def test_attention_zero_query_is_value_mean():
    k = rng.standard_normal((9, 8))
    v = rng.standard_normal((9, 8))
    out = O.softmax_attention(np.zeros((2, 8)), k, v)
    np.testing.assert_allclose(out, np.broadcast_to(v.mean(0), (2, 8)), rtol=1e-14)


def test_attention_single_key_returns_value():
    v = rng.standard_normal((1, 8))
    out = O.softmax_attention(rng.standard_normal((3, 8)), rng.standard_normal((1, 8)), v)
    np.testing.assert_allclose(out, np.broadcast_to(v, (3, 8)), rtol=1e-14)


def test_attention_two_keys_closed_form():
    q = rng.standard_normal((1, 4))
    k = rng.standard_normal((2, 4))
    v = rng.standard_normal((2, 4))
    delta = (q[0] @ k[0] - q[0] @ k[1]) / 2.0     # sqrt(hd) = 2
    w0 = 1.0 / (1.0 + math.exp(-delta))
    np.testing.assert_allclose(O.softmax_attention(q, k, v)[0], w0 * v[0] + (1 - w0) * v[1], rtol=1e-13)


def test_attention_key_permutation_invariance():
    q = rng.standard_normal((4, 8))
    k = rng.standard_normal((11, 8))
    v = rng.standard_normal((11, 8))
    perm = rng.permutation(11)
    np.testing.assert_allclose(O.softmax_attention(q, k, v),
                               O.softmax_attention(q, k[perm], v[perm]), rtol=1e-13)


def test_silu_points():
    assert O.silu(np.array([0.0]))[0] == 0.0
    np.testing.assert_allclose(O.silu(np.array([math.log(3.0)]))[0], 0.75 * math.log(3.0), rtol=1e-15)
    np.testing.assert_allclose(O.silu(np.array([-40.0]))[0], -40.0 / (1 + math.exp(40.0)), rtol=1e-12)


# --------------------------------------------------------------------------
# draft block wiring
# --------------------------------------------------------------------------

def _tiny_weights(d=16, F=32, V=50, L=1, seed=0):
    r = np.random.default_rng(seed)
    W = {"embed": r.standard_normal((V, d)) * 0.5, "mask_vec": r.standard_normal(d) * 0.5,
         "ctx_norm": 1 + 0.1 * r.standard_normal(d), "final_norm": 1 + 0.1 * r.standard_normal(d),
         "layers": []}
    for _ in range(L):
        W["layers"].append({
            "attn_norm": 1 + 0.1 * r.standard_normal(d), "mlp_norm": 1 + 0.1 * r.standard_normal(d),
            "wq": r.standard_normal((d, d)) * 0.3, "wk": r.standard_normal((d, d)) * 0.3,
            "wv": r.standard_normal((d, d)) * 0.3, "wo": r.standard_normal((d, d)) * 0.3,
            "wg": r.standard_normal((F, d)) * 0.3, "wu": r.standard_normal((F, d)) * 0.3,
            "wd": r.standard_normal((d, F)) * 0.3})
    return W


def test_draft_block_zero_output_projections_keep_block_input():
    # W_o = W_d = 0: the residual stream stays the block input, so the output is
    # RMSNorm_final of [embed[anchor]; mask_vec ...].  With +-a entries that is
    # sign * final_norm exactly (eps 0).
    d = 16
    W = _tiny_weights(d=d)
    W["embed"] = np.where(W["embed"] > 0, 0.25, -0.25)
    W["mask_vec"] = np.where(W["mask_vec"] > 0, 2.0, -2.0)
    for lw in W["layers"]:
        lw["wo"][:] = 0
        lw["wd"][:] = 0
    ctx = rng.standard_normal((10, d))
    out = O.draft_block(W, ctx, [0, 4, 10], [7, 3], block=4, n_heads=2, head_dim=8,
                        rope_theta=1e4, norm_eps=0.0, act_dtype="f64")
    for i, a in enumerate([7, 3]):
        np.testing.assert_allclose(out[i * 4], np.sign(W["embed"][a]) * W["final_norm"], rtol=1e-14)
        for k in range(1, 4):
            np.testing.assert_allclose(out[i * 4 + k], np.sign(W["mask_vec"]) * W["final_norm"], rtol=1e-14)


def test_draft_block_zero_query_averages_own_sequence_context_and_block():
    # W_q = 0 -> uniform attention over this sequence's T_i context keys plus its
    # B block keys, and over nothing else (ragged sequences do not mix).
    d, B = 16, 4
    W = _tiny_weights(d=d)
    W["layers"][0]["wq"][:] = 0
    ctx = rng.standard_normal((10, d))
    cu = [0, 3, 10]
    inter = {}
    O.draft_block(W, ctx, cu, [1, 2], block=B, n_heads=2, head_dim=8, rope_theta=1e4,
                  norm_eps=1e-6, act_dtype="f64", intermediates=inter)
    L0 = inter["layers"][0]
    for i in range(2):
        v_all = np.concatenate([L0["Vc"][cu[i]:cu[i + 1]], L0["Vb"][i * B:(i + 1) * B]], axis=0)
        for k in range(B):
            np.testing.assert_allclose(L0["O"][i * B + k], v_all.mean(axis=0), rtol=1e-12)


def test_zero_keys_attend_uniformly_with_values_from_w_v_and_output_through_w_o():
    # W_k = 0: every score is 0, so each block row's attention output is the
    # plain mean of the values of its own sequence's T_i context rows and B
    # block rows.  Context rows are constant vectors a_t * 1 and the block
    # input rows are 0.5 * 1, so at eps 0 their norms are the norm weights:
    # every context value row is ctx_norm W_v^T and every block value row
    # attn_norm W_v^T.  In every head, per sequence,
    #     O = (T_i ctx_norm W_v^T + B attn_norm W_v^T) / (T_i + B),
    # and the attention residual is h = 0.5 + O W_o^T.  Keys or values taken
    # from another projection, heads reading another head's columns, or W_o
    # applied untransposed each move O or h.
    d, B, nh, hd = 16, 4, 2, 8
    W = _tiny_weights(d=d, seed=91)
    lw = W["layers"][0]
    lw["wk"][:] = 0
    W["embed"] = np.full_like(W["embed"], 0.5)
    W["mask_vec"] = np.full_like(W["mask_vec"], 0.5)
    cu = [0, 3, 10]
    ctx = np.repeat(np.random.default_rng(92).uniform(0.5, 2.0, 10)[:, None], d, axis=1)
    inter = {}
    O.draft_block(W, ctx, cu, [1, 2], block=B, n_heads=nh, head_dim=hd, rope_theta=1e4,
                  norm_eps=0.0, act_dtype="f64", intermediates=inter)
    L0 = inter["layers"][0]
    vc = W["ctx_norm"] @ lw["wv"].T
    vb = lw["attn_norm"] @ lw["wv"].T
    for i in range(2):
        T = cu[i + 1] - cu[i]
        want = (T * vc + B * vb) / (T + B)
        for k in range(B):
            np.testing.assert_allclose(L0["O"][i * B + k], want, rtol=1e-12, atol=1e-12)
            np.testing.assert_allclose(L0["h_attn"][i * B + k], 0.5 + want @ lw["wo"].T, rtol=1e-6, atol=1e-6)


def test_a_layer_with_zero_output_projections_adds_nothing():
    # a second layer whose W_o and W_d are 0 leaves the residual stream as the
    # first layer left it, so two layers equal the first alone, bit for bit;
    # layers that read another layer's weights would not
    d, B = 16, 4
    W1 = _tiny_weights(d=d, L=1, seed=93)
    extra = _tiny_weights(d=d, L=1, seed=94)["layers"][0]
    extra["wo"][:] = 0
    extra["wd"][:] = 0
    W2 = dict(W1)
    W2["layers"] = [W1["layers"][0], extra]
    ctx = np.random.default_rng(96).standard_normal((9, d))
    cu = [0, 4, 9]
    kw = dict(block=B, n_heads=2, head_dim=8, rope_theta=1e4, norm_eps=1e-6, act_dtype="f64")
    np.testing.assert_array_equal(O.draft_block(W2, ctx, cu, [3, 7], **kw), O.draft_block(W1, ctx, cu, [3, 7], **kw))


def test_draft_tokens_are_block_slots_one_to_b_minus_one():
    # slot 0 of each block is the anchor; drafts d_1 .. d_{B-1} are slots 1 .. B-1
    B, batch = 5, 2
    tok = np.arange(batch * B) * 10
    np.testing.assert_array_equal(O.draft_tokens(tok, batch, B), [[10, 20, 30, 40], [60, 70, 80, 90]])


def test_draft_block_sequences_are_independent():
    d, B = 16, 4
    W = _tiny_weights(d=d)
    ctx = rng.standard_normal((10, d))
    cu = [0, 3, 10]
    a = O.draft_block(W, ctx, cu, [1, 2], block=B, n_heads=2, head_dim=8, rope_theta=1e4,
                      norm_eps=1e-6, act_dtype="f64")
    ctx2 = ctx.copy()
    ctx2[5:] += 1.0                     # only sequence 1's context changes
    b = O.draft_block(W, ctx2, cu, [1, 2], block=B, n_heads=2, head_dim=8, rope_theta=1e4,
                      norm_eps=1e-6, act_dtype="f64")
    np.testing.assert_array_equal(a[:B], b[:B])
    assert np.abs(a[B:] - b[B:]).max() > 1e-6


# --------------------------------------------------------------------------
# LM head, accept, tau, KL
# --------------------------------------------------------------------------

def test_lm_head_argmax_first_index_on_ties_brute_force():
    # small integers: every dot product is exact whatever order the matmul
    # sums in, so duplicate weight rows give an exact tie
    h = rng.integers(-8, 9, (6, 8)).astype(np.float64)
    W = rng.integers(-8, 9, (40, 8)).astype(np.float64)
    W[17] = W[5]                       # exact duplicate rows -> exact tie in z
    h[2] = W[5] * 10                   # row 2's max is the (5, 17) tie
    res = O.lm_head(h, W)
    z = h @ W.T
    for i in range(6):
        best, bi = -math.inf, -1
        for v in range(40):
            if z[i, v] > best:
                best, bi = z[i, v], v
        assert res["tok"][i] == bi
    assert res["tok"][2] == 5


def test_logsoftmax_normalised_and_argmax_preserved():
    h = rng.standard_normal((5, 8))
    W = rng.standard_normal((30, 8))
    for it in (1.0, 0.5, 3.0):
        res = O.lm_head(h, W, inv_temp=it, logsoftmax=True)
        np.testing.assert_allclose(np.log(np.exp(res["logsoftmax"]).sum(1)), 0.0, atol=1e-13)
        assert np.array_equal(np.argmax(res["logsoftmax"], 1), res["tok"])


def test_logsoftmax_two_class_closed_form():
    h = np.array([[1.0]])
    W = np.array([[2.0], [0.5]])
    res = O.lm_head(h, W, inv_temp=1.0, logsoftmax=True)
    np.testing.assert_allclose(res["logsoftmax"][0], [-math.log1p(math.exp(-1.5)),
                                                      -math.log1p(math.exp(1.5))], rtol=1e-14)


def test_accept_len_against_cumprod_and_edges():
    d = rng.integers(0, 5, size=(200, 7))
    t = rng.integers(0, 5, size=(200, 7))
    t[::3] = d[::3]
    expect = np.cumprod(d == t, axis=1).sum(axis=1)
    assert np.array_equal(O.accept_len(d, t), expect)
    assert O.accept_len(d[:1], d[:1])[0] == 7
    t2 = d[:1].copy()
    t2[0, 0] += 1
    assert O.accept_len(d[:1], t2)[0] == 0


def test_tau_counts_bonus_token_table2():
    g = json.load(open(os.path.join(GOLDEN, "table2_mtp3_tau.json")))
    k = g["drafted_steps"]
    taus = list(g["tau_per_benchmark"].values())
    # a drafts-only count can never exceed k; the printed values do
    assert max(taus) > k
    # with the bonus token tau lies in [1, k + 1] and reaches k + 1 on full acceptance
    assert all(1.0 <= t <= k + 1 for t in taus)
    assert O.mean_accepted_length([k, k]) == k + 1
    assert O.mean_accepted_length([0]) == 1.0
    # the Average column is the arithmetic mean of the seven benchmarks
    assert round(sum(taus) / len(taus), 2) == g["tau_average_printed"]


def test_kl_pins():
    z = rng.standard_normal((2, 9))
    assert abs(O.kl_distill(z, z, 1.0)) < 1e-14
    assert O.kl_distill(z, rng.standard_normal((2, 9)), 2.0) > 0
    # two classes: p = (3/4, 1/4), q = (1/2, 1/2) -> KL = 3/4 ln 3/2 + 1/4 ln 1/2
    t = np.array([[math.log(3.0), 0.0]])
    s = np.array([[0.0, 0.0]])
    np.testing.assert_allclose(O.kl_distill(t, s, 1.0),
                               0.75 * math.log(1.5) + 0.25 * math.log(0.5), rtol=1e-14)
    # T^2 factor: logits scaled with T keep p, q fixed, loss scales by T^2
    np.testing.assert_allclose(O.kl_distill(2 * t, 2 * s, 2.0),
                               4 * O.kl_distill(t, s, 1.0), rtol=1e-13)


# ---------------------------------------------- speculative-sampling verification
def _dist(rng, V):
    w = rng.random(V).astype(np.float64) + 0.05
    return (w / w.sum()).astype(np.float32)


def test_accept_sample_output_is_distributed_as_p():
    """The defining property of speculative sampling: with x ~ q, accept with
    probability min(1, p(x)/q(x)), else draw from norm(max(0, p - q)), the
    emitted token is distributed exactly as p.  Integrated over dense grids of
    the two uniforms (u, r) and exactly over x."""
    rng = np.random.default_rng(5)
    V, G = 5, 96
    p0, q0 = _dist(rng, V), _dist(rng, V)
    grid = ((np.arange(G) + 0.5) * 2.0 ** 32 / G).astype(np.uint64)
    freq = np.zeros(V)
    for x in range(V):
        # batch over (u, r) pairs for this drafted x
        uu, rr = np.meshgrid(grid, grid, indexing="ij")
        n = uu.size
        p = np.broadcast_to(np.stack([p0, p0])[None], (n, 2, V))
        q = np.broadcast_to(q0[None, None], (n, 1, V))
        acc, nxt = O.accept_sample(p, q, np.full((n, 1), x), uu.reshape(n, 1), rr.reshape(n))
        first = np.where(acc == 1, x, nxt)
        freq += q0[x] * np.bincount(first, minlength=V) / n
    np.testing.assert_allclose(freq, p0, atol=2.5 / G)


def test_accept_sample_special_cases():
    rng = np.random.default_rng(6)
    V, nd = 7, 4
    p = np.stack([_dist(rng, V) for _ in range(nd + 1)])[None]
    u = np.full((1, nd), 2 ** 32 - 1, dtype=np.uint64)          # the largest uniform
    acc, nxt = O.accept_sample(p, p[:, :nd], np.zeros((1, nd), int), u, np.array([0]))
    assert acc[0] == nd and nxt[0] == 0                          # q == p: ratio 1 > u, bonus from p[nd]
    q1 = np.zeros((1, nd, V), np.float32); q1[:, :, 2] = 1       # draft certain of token 2
    p1 = np.zeros((1, nd + 1, V), np.float32); p1[:, :, 5] = 1   # target certain of token 5
    acc, nxt = O.accept_sample(p1, q1, np.full((1, nd), 2), np.zeros((1, nd), np.uint64), np.array([123]))
    assert acc[0] == 0 and nxt[0] == 5                           # p/q = 0: rejected, residual = p
    acc, _ = O.accept_sample(p, p[:, :nd], np.array([[0, 1, V, 2]]), u, np.array([0]))
    assert acc[0] == 2                                           # an id outside the vocabulary is rejected


def test_accept_sample_bonus_token_comes_from_the_slot_after_the_drafts():
    # Every draft accepted (q == p, so the ratio is 1 and any u < 2^32 passes):
    # the emitted token is drawn from p at slot n_draft, the position after the
    # block.  The draft slots put all their mass on token 1, so a draw from any
    # of them would show.  With r = 2^32 - 1 the inverse CDF picks the last
    # token with weight.
    V, nd = 6, 3
    p = np.zeros((2, nd + 1, V), np.float32)
    p[:, :nd, 1] = 1.0
    p[0, nd, 4] = 1.0
    p[1, nd, 2] = 0.5
    p[1, nd, 5] = 0.5
    u = np.zeros((2, nd), np.uint64)
    acc, nxt = O.accept_sample(p, p[:, :nd], np.full((2, nd), 1), u, np.array([0, 2 ** 32 - 1], np.uint64))
    assert list(acc) == [nd, nd]
    assert nxt[0] == 4 and nxt[1] == 5


def test_accept_sample_inverse_cdf_boundaries():
    # uniform residual over 4 tokens: weights 2^38 each, R = 2^40, threshold = r * 2^8
    p = np.zeros((1, 2, 4), np.float32); p[0, 0] = 0.25
    q = np.zeros((1, 1, 4), np.float32)
    draft = np.array([[0]])
    u = np.array([[2 ** 32 - 1]], dtype=np.uint64)                # p/q = inf: accepted ... so use p at slot 1
    p[0, 1] = 0.25
    for r, want in [(0, 0), (2 ** 30 - 1, 0), (2 ** 30, 1), (2 ** 31, 2), (2 ** 32 - 1, 3)]:
        _, nxt = O.accept_sample(p, q, draft, u, np.array([r], dtype=np.uint64))
        assert nxt[0] == want, (r, nxt[0])


# --------------------------------------------------------------------------
# drafter wiring pins: each fixes one place where the drafter reading could
# be slipped (MLP wiring, where RoPE goes, block and context positions, the
# context norm, the gate under the per-path norm, the log-softmax temperature)
# with a closed form of a special case
# --------------------------------------------------------------------------

def _const_block_weights(d, F, gamma_mlp, seed=3):
    """Drafter weights whose block input rows are all 0.5 (so RMSNorm(h) is
    the norm weight itself at eps 0) and whose attention adds nothing (W_o = 0)."""
    W = _tiny_weights(d=d, F=F, seed=seed)
    W["embed"] = np.full_like(W["embed"], 0.5)
    W["mask_vec"] = np.full_like(W["mask_vec"], 0.5)
    lw = W["layers"][0]
    lw["wo"][:] = 0.0
    lw["mlp_norm"] = gamma_mlp
    return W


def test_swiglu_gate_closes_the_mlp_when_the_gate_logit_is_very_negative():
    # x2 = mlp_norm = gamma for every block row (h0 = 0.5 * ones, eps 0).  Gate
    # rows with gamma . W_g[f] = -60 give silu(-60) ~ -5e-25: the MLP adds
    # nothing and the output is RMSNorm_final(0.5 * ones) = final_norm exactly.
    # With the gate and up projections swapped the MLP adds silu(u) * (-60).
    d, F = 16, 8
    r = np.random.default_rng(71)
    gamma = 1.0 + 0.2 * r.random(d)
    W = _const_block_weights(d, F, gamma)
    lw = W["layers"][0]
    lw["wg"] = np.tile(-60.0 * gamma / np.dot(gamma, gamma), (F, 1))
    lw["wu"] = r.standard_normal((F, d))
    lw["wd"] = r.standard_normal((d, F))
    out = O.draft_block(W, r.standard_normal((5, d)), [0, 5], [3], block=4, n_heads=2, head_dim=8,
                        rope_theta=1e4, norm_eps=0.0, act_dtype="f64")
    np.testing.assert_allclose(out, np.broadcast_to(W["final_norm"], out.shape), rtol=0, atol=1e-12)


def test_swiglu_is_linear_in_the_up_projection_when_the_gate_saturates_high():
    # gamma . W_g[f] = 40: silu(40) = 40 to 1e-16, so act = 40 * (W_u gamma) and
    # h = 0.5 * ones + 40 * W_d W_u gamma, out = h / rms(h) * final_norm.
    d, F = 16, 8
    r = np.random.default_rng(72)
    gamma = 1.0 + 0.2 * r.random(d)
    W = _const_block_weights(d, F, gamma)
    lw = W["layers"][0]
    lw["wg"] = np.tile(40.0 * gamma / np.dot(gamma, gamma), (F, 1))
    lw["wu"] = r.standard_normal((F, d)) * 0.1
    lw["wd"] = r.standard_normal((d, F)) * 0.1
    out = O.draft_block(W, r.standard_normal((5, d)), [0, 5], [3], block=4, n_heads=2, head_dim=8,
                        rope_theta=1e4, norm_eps=0.0, act_dtype="f64")
    h = 0.5 + 40.0 * (lw["wd"] @ (lw["wu"] @ gamma))
    expect = h / math.sqrt(np.mean(h * h)) * W["final_norm"]
    # the block residual h is stored in fp32 (the precision contract), so
    # agreement is to fp32 rounding of h
    np.testing.assert_allclose(out, np.broadcast_to(expect, out.shape), rtol=4e-7, atol=0)


def _rot(pairs, angle):
    """Rotate 2-vectors (last axis) by angle, as complex multiplication."""
    z = (pairs[..., 0] + 1j * pairs[..., 1]) * np.exp(1j * np.asarray(angle, np.float64))
    return np.stack([z.real, z.imag], axis=-1)


def test_context_projection_rotates_keys_and_not_values():
    # head_dim 2 (frequency theta^0 = 1: the angle is the position), identity
    # projections: K_c[t] is c_t turned by t radians per head, V_c[t] is c_t.
    c = rng.standard_normal((3, 4))
    pos = np.array([0.0, 3.0, 7.0])
    K, V = O.context_kv(c, np.eye(4), np.eye(4), pos, n_heads=2, head_dim=2, theta=10000.0, act_dtype="f64")
    expect_k = _rot(c.reshape(3, 2, 2), pos[:, None]).reshape(3, 4)
    np.testing.assert_allclose(K, expect_k, rtol=1e-14, atol=1e-15)
    np.testing.assert_array_equal(V, c)


def test_block_attention_positions_rotary_and_context_norm_closed_form():
    """Identity Q/K/V projections, head_dim 2: per head the score of a block
    query (slot k, position T_i + k) and a key at position p is
    Re(z_q e^{i(T_i+k)} conj(z_k e^{ip})) / sqrt(2) for the complex pairs z of
    the normed rows, and the values are the unrotated pairs.  The normed
    context rows are y / rms(y) * ctx_norm, the normed block rows
    h0 / rms(h0) * attn_norm.  Checks block slot k at exactly T_i + k, context
    row t at t, RoPE on Q and both kinds of keys, none on either kind of
    values, the context norm weight and the 1/sqrt(hd) scale."""
    d, B, hd = 4, 3, 2
    W = _tiny_weights(d=d, F=8, V=6, seed=9)
    lw = W["layers"][0]
    for k in ("wq", "wk", "wv"):
        lw[k] = np.eye(d)
    lw["wo"][:] = 0.0
    ctx = rng.standard_normal((5, d))
    cu, anchor = [0, 3, 5], [4, 1]
    inter = {}
    O.draft_block(W, ctx, cu, anchor, block=B, n_heads=2, head_dim=hd, rope_theta=1e4, norm_eps=0.0,
                  act_dtype="f64", intermediates=inter)
    got = inter["layers"][0]["O"]

    def normed(rows, w):
        return rows / np.sqrt(np.mean(rows * rows, axis=1, keepdims=True)) * w
    c = normed(ctx, W["ctx_norm"])
    for i in range(2):
        T = cu[i + 1] - cu[i]
        # the block residual starts as the fp32 copy of its input rows
        h0 = np.stack([W["embed"][anchor[i]]] + [W["mask_vec"]] * (B - 1)).astype(np.float32).astype(np.float64)
        x = normed(h0, W["layers"][0]["attn_norm"])
        keys = np.concatenate([c[cu[i]:cu[i + 1]], x])            # [T + B, d], unrotated
        kpos = np.concatenate([np.arange(T), T + np.arange(B)])
        for hh in range(2):
            kz = keys[:, 2 * hh] + 1j * keys[:, 2 * hh + 1]
            for k in range(B):
                qz = (x[k, 2 * hh] + 1j * x[k, 2 * hh + 1]) * np.exp(1j * (T + k))
                s = np.real(qz * np.conj(kz * np.exp(1j * kpos))) / math.sqrt(hd)
                p = np.exp(s - s.max())
                p /= p.sum()
                np.testing.assert_allclose(got[i * B + k, 2 * hh:2 * hh + 2], p @ keys[:, 2 * hh:2 * hh + 2],
                                           rtol=1e-12, atol=1e-14)


def test_per_path_norm_leaves_the_gate_on_the_raw_residual():
    # m = 2, d = 4, path 0 = 1 and path 1 = 3 everywhere: mean(H^2) = 5, so
    # r = 1/sqrt(5) (eps 0).  W_f row 0 reads H[1][0] (+1), row 1 reads
    # H[0][2] (-2): gates sigmoid(3/sqrt5 + b0), sigmoid(-2/sqrt5 + b1) whether
    # or not the drafter-side per-path norm is on; with it on each normed path
    # is its weight gamma_j, so y = alpha_0 gamma_0 + alpha_1 gamma_1.
    m, d = 2, 4
    H = np.concatenate([np.ones((1, 1, d)), 3.0 * np.ones((1, 1, d))], axis=1)
    Wf = np.zeros((m, m * d))
    Wf[0, 1 * d + 0] = 1.0
    Wf[1, 0 * d + 2] = -2.0
    b = np.array([0.1, -0.2])
    gamma = np.array([[0.5, 1.5, -1.0, 2.0], [1.0, -0.5, 0.25, 3.0]])
    y, a = O.gated_reduce(H, Wf, b, rms_eps=0.0, path_norm_w=gamma, path_norm_eps=0.0, out_dtype="f64")
    s5 = math.sqrt(5.0)
    expect_a = 1.0 / (1.0 + np.exp(-np.array([3.0 / s5 + 0.1, -2.0 / s5 - 0.2])))
    np.testing.assert_allclose(a[0], expect_a, rtol=1e-14)
    np.testing.assert_allclose(y[0], expect_a[0] * gamma[0] + expect_a[1] * gamma[1], rtol=1e-14)


def test_logsoftmax_two_class_closed_form_at_temperature():
    # z = (2, 0.5): at inv_temp t the two classes differ by 1.5 t
    h = np.array([[1.0]])
    W = np.array([[2.0], [0.5]])
    for t in (0.5, 3.0):
        res = O.lm_head(h, W, inv_temp=t, logsoftmax=True)
        np.testing.assert_allclose(res["logsoftmax"][0], [-math.log1p(math.exp(-1.5 * t)),
                                                          -math.log1p(math.exp(1.5 * t))], rtol=1e-13)
        assert res["tok"][0] == 0 and res["zmax"][0] == 2.0


# --------------------------------------------------------------------------
# generic fc reducer (Sec. 2.2, Table 1): the fallback for unequal widths
# --------------------------------------------------------------------------

def test_fc_reduce_identity_blocks_sum_the_paths():
    """W_fc = [I I ... I] maps vec(H_t) to the plain path sum; a block of
    the identity's first d_out rows truncates each path to d_out features
    (a narrower drafter), and the position of a block picks its path."""
    N, m, d_in = 5, 3, 8
    H = rng.standard_normal((N, m, d_in))
    I = np.eye(d_in)
    np.testing.assert_array_equal(O.fc_reduce(H, np.concatenate([I] * m, axis=1)), H.sum(axis=1))
    d_out = 4
    W = np.zeros((d_out, m * d_in))
    W[:, 2 * d_in:2 * d_in + d_out] = np.eye(d_out)        # path 2, first d_out features
    np.testing.assert_array_equal(O.fc_reduce(H, W), H[:, 2, :d_out])
    # a wider drafter: path 0 placed twice, the second copy negated
    W = np.zeros((2 * d_in, m * d_in))
    W[:d_in, :d_in] = I
    W[d_in:, :d_in] = -I
    np.testing.assert_array_equal(O.fc_reduce(H, W), np.concatenate([H[:, 0], -H[:, 0]], axis=1))


def test_fc_reduce_brute_force_loops():
    N, m, d_in, d_out = 3, 2, 5, 7
    H = rng.standard_normal((N, m, d_in))
    W = rng.standard_normal((d_out, m * d_in))
    ref = np.zeros((N, d_out))
    for t in range(N):
        for o in range(d_out):
            ref[t, o] = sum(W[o, j * d_in + e] * H[t, j, e] for j in range(m) for e in range(d_in))
    np.testing.assert_allclose(O.fc_reduce(H, W), ref, rtol=1e-13, atol=1e-13)


# --------------------------------------------------------------------------
# training objective, Eq. 3: L = L_CE + alpha * L_KL
# --------------------------------------------------------------------------

def test_cross_entropy_closed_forms():
    # two classes with logits (0, x): CE of class 1 = log(1 + e^-x), of class 0 = log(1 + e^x)
    for x in (-3.0, 0.0, 0.7, 5.0):
        z = np.array([[0.0, x], [0.0, x]])
        np.testing.assert_allclose(O.cross_entropy(z, [1, 0]),
                                   [math.log1p(math.exp(-x)), math.log1p(math.exp(x))], rtol=1e-12)
    # uniform logits over V classes: log V whatever the label; a shift changes nothing
    z = np.full((3, 10), 2.5)
    np.testing.assert_allclose(O.cross_entropy(z, [0, 4, 9]), math.log(10.0), rtol=1e-14)
    # an unsupervised row is NaN (kept out of any mean)
    assert np.isnan(O.cross_entropy(z, [-1, 0, 0])[0])


def _two_class_kl(a, b, T):
    p1 = 1.0 / (1.0 + math.exp(-a / T))
    q1 = 1.0 / (1.0 + math.exp(-b / T))
    return p1 * math.log(p1 / q1) + (1 - p1) * math.log((1 - p1) / (1 - q1))


def test_draft_loss_two_class_closed_form():
    """batch 2, block 3, P = 2, two classes.  Logit rows are (0, x).  Student
    rows: anchor slots get a logit the loss must ignore, draft k of block i
    gets s[i][k-1]; teacher row k - 1 of block i gets t[i][k-1].  Labels make
    each CE a log1p term.  Every term is written out by hand."""
    s = [[0.4, -1.2], [2.0, 0.3]]
    t = [[1.5, -0.5], [0.0, 3.0]]
    lab = [[1, 0], [0, 1]]
    S = np.zeros((6, 2))
    for i in range(2):
        S[i * 3, 1] = 40.0  # anchor rows: neither CE nor KL may read them
        for k in (1, 2):
            S[i * 3 + k, 1] = s[i][k - 1]
    Tt = np.zeros((2, 2, 2))
    for i in range(2):
        for k in range(2):
            Tt[i, k, 1] = t[i][k]

    def ce(x, y):
        return math.log1p(math.exp(-x)) if y == 1 else math.log1p(math.exp(x))
    for T, a in ((1.0, 0.1), (2.0, 0.2), (0.5, 1.0)):
        out = O.draft_loss(Tt, S, lab, block=3, P=2, t_kd=T, alpha=a)
        l_ce = sum(ce(s[i][k], lab[i][k]) for i in range(2) for k in range(2)) / 4
        l_kl = T * T / 2 * sum(_two_class_kl(t[i][k], s[i][k], T) for i in range(2) for k in range(2)) / 2
        np.testing.assert_allclose(out["ce"], l_ce, rtol=1e-13)
        np.testing.assert_allclose(out["kl"], l_kl, rtol=1e-12)
        np.testing.assert_allclose(out["loss"], l_ce + a * l_kl, rtol=1e-12)


def test_draft_loss_kl_covers_the_first_P_positions_only():
    """Teacher equal to the student on positions 1..P gives L_KL = 0 whatever
    positions past P and the anchor slot hold; changing position P + 1 or the
    anchor leaves the loss's KL part alone, changing position P does not."""
    batch, B, P, V = 3, 5, 2, 7
    S = rng.standard_normal((batch * B, V))
    Tt = np.stack([S[i * B + 1:i * B + 1 + P] for i in range(batch)])
    lab = rng.integers(0, V, (batch, B - 1))
    base = O.draft_loss(Tt, S, lab, block=B, P=P, t_kd=1.7, alpha=0.3)
    assert abs(base["kl"]) < 1e-14
    S2 = S.copy()
    S2[0] += 5.0 * rng.standard_normal(V)            # anchor of block 0
    S2[1 * B + P + 1] += 5.0 * rng.standard_normal(V)  # position P + 1 of block 1
    assert abs(O.draft_loss(Tt, S2, lab, block=B, P=P, t_kd=1.7, alpha=0.3)["kl"]) < 1e-14
    S3 = S.copy()
    S3[2 * B + P] += 5.0 * rng.standard_normal(V)      # position P of block 2
    assert O.draft_loss(Tt, S3, lab, block=B, P=P, t_kd=1.7, alpha=0.3)["kl"] > 1e-3


def test_draft_loss_ce_is_at_temperature_one_and_skips_unlabelled_rows():
    batch, B, V = 2, 4, 6
    S = rng.standard_normal((batch * B, V))
    Tt = rng.standard_normal((batch, 2, V))
    lab = np.array([[3, -1, 0], [-1, -1, 5]])
    a = O.draft_loss(Tt, S, lab, block=B, P=2, t_kd=1.0, alpha=0.0)
    b = O.draft_loss(Tt, S, lab, block=B, P=2, t_kd=4.0, alpha=0.0)
    assert a["ce"] == b["ce"] and a["loss"] == a["ce"]
    # the mean runs over the three supervised positions, each a brute-force -log softmax
    def nll(z, y):
        return -(z[y] - math.log(sum(math.exp(v) for v in z)))
    ref = (nll(S[1], 3) + nll(S[3], 0) + nll(S[7], 5)) / 3
    np.testing.assert_allclose(a["ce"], ref, rtol=1e-13)
    # a constant shift of any row changes nothing (log-softmax rows may be passed)
    S4 = S + rng.standard_normal((batch * B, 1))
    T4 = Tt + rng.standard_normal((batch, 2, 1))
    c = O.draft_loss(T4, S4, lab, block=B, P=2, t_kd=2.0, alpha=0.5)
    d = O.draft_loss(Tt, S, lab, block=B, P=2, t_kd=2.0, alpha=0.5)
    np.testing.assert_allclose(c["loss"], d["loss"], rtol=1e-12)
