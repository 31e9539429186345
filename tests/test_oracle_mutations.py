"""Planted mistakes in the oracle must each turn a pin red.

Each entry below is a plausible slip in ``oracle/hdf_oracle.py`` (a swapped
operand, a dropped term or weight, a rotation in the wrong place, an index
off by one).  The test plants it in a copy of the oracle source, on the CPU,
loads ``tests/test_oracle_pins.py`` against that copy and runs every pin:
at least one must fail.  The unmutated source must pass them all, so the
harness itself is checked too.  Nothing here touches the CUDA library."""
import importlib.util
import os
import sys
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE_SRC = os.path.join(ROOT, "oracle", "hdf_oracle.py")
PINS = os.path.join(ROOT, "tests", "test_oracle_pins.py")

# name -> (text in the oracle source, replacement)
MUTATIONS = {
    # ------------------------------------- reducer, its gradient, verification
    "inverse RMS over the sum of squares, not the mean": (
        "r = 1.0 / np.sqrt(np.mean(x * x, axis=1) + rms_eps)  # inverse RMS",
        "r = 1.0 / np.sqrt(np.sum(x * x, axis=1) + rms_eps)  # inverse RMS"),
    "inverse RMS dropped from the gate": (
        "x_tilde = x * r[:, None]",
        "x_tilde = x"),
    "RMS eps outside the square root": (
        "r = 1.0 / np.sqrt(np.mean(x * x, axis=1) + rms_eps)  # inverse RMS",
        "r = 1.0 / (np.sqrt(np.mean(x * x, axis=1)) + rms_eps)  # inverse RMS"),
    "gate scale applied to the bias too": (
        "return gate_scale * (x_tilde @ np.asarray(Wf, np.float64).T) + np.asarray(b, np.float64)[None, :]",
        "return gate_scale * (x_tilde @ np.asarray(Wf, np.float64).T + np.asarray(b, np.float64)[None, :])"),
    "gate offset inside the sigmoid": (
        "alpha = sigmoid(gate_logits(H, Wf, b, rms_eps, gate_scale)) + gate_offset",
        "alpha = sigmoid(gate_logits(H, Wf, b, rms_eps, gate_scale) + gate_offset)"),
    "gate offset dropped": (
        "alpha = sigmoid(gate_logits(H, Wf, b, rms_eps, gate_scale)) + gate_offset",
        "alpha = sigmoid(gate_logits(H, Wf, b, rms_eps, gate_scale))"),
    "sigmoid of negative logits inverted": (
        "out[~pos] = e / (1.0 + e)",
        "out[~pos] = 1.0 / (1.0 + e)"),
    "per-path norm RMS over the whole token": (
        "rp = 1.0 / np.sqrt(np.mean(H * H, axis=2) + path_norm_eps)   # [N, m]",
        "rp = (1.0 / np.sqrt(np.mean(H * H, axis=(1, 2)) + path_norm_eps))[:, None] * np.ones((1, H.shape[1]))"),
    "per-path norm weight dropped": (
        "Hh = H * rp[:, :, None] * np.asarray(path_norm_w, np.float64)[None, :, :]",
        "Hh = H * rp[:, :, None]"),
    "weighted sum normalised by the gate sum": (
        "y = np.einsum(\"nj,njd->nd\", alpha, Hh)",
        "y = np.einsum(\"nj,njd->nd\", alpha, Hh) / alpha.sum(axis=1, keepdims=True)"),
    "backward: sigmoid derivative dropped": (
        "dg = a * sg * (1.0 - sg)",
        "dg = a"),
    "backward: sign flipped": (
        "dg = a * sg * (1.0 - sg)",
        "dg = -a * sg * (1.0 - sg)"),
    "backward: inverse RMS dropped from dW_f": (
        "dWf = (gate_scale * r[:, None] * dg).T @ x",
        "dWf = (gate_scale * dg).T @ x"),
    "backward: gate scale dropped from dW_f": (
        "dWf = (gate_scale * r[:, None] * dg).T @ x",
        "dWf = (r[:, None] * dg).T @ x"),
    "backward: dy paired with the paths reversed": (
        "a = np.einsum(\"nd,njd->nj\", dy, H)",
        "a = np.einsum(\"nd,njd->nj\", dy, H[:, ::-1])"),
    "rope frequency exponent without the factor 2": (
        "inv_freq = theta ** (-2.0 * i / hd)",
        "inv_freq = theta ** (-1.0 * i / hd)"),
    "rope rotation direction reversed": (
        "out[..., 0::2] = x0 * c - x1 * s\n    out[..., 1::2] = x0 * s + x1 * c",
        "out[..., 0::2] = x0 * c + x1 * s\n    out[..., 1::2] = -x0 * s + x1 * c"),
    "rope pairs rotate-half instead of interleaved": (
        "    x0 = x[..., 0::2]\n    x1 = x[..., 1::2]\n    out = np.empty_like(x)\n"
        "    out[..., 0::2] = x0 * c - x1 * s\n    out[..., 1::2] = x0 * s + x1 * c",
        "    x0 = x[..., : hd // 2]\n    x1 = x[..., hd // 2:]\n    out = np.empty_like(x)\n"
        "    out[..., : hd // 2] = x0 * c - x1 * s\n    out[..., hd // 2:] = x0 * s + x1 * c"),
    "attention softmax normalised over the queries": (
        "p = p / p.sum(axis=1, keepdims=True)",
        "p = p / p.sum(axis=0, keepdims=True)"),
    "log-softmax without the log-sum-exp": (
        "ls = s - lse",
        "ls = s - smax"),
    "accept length counts the first mismatch": (
        "        out[i] = n\n    return out",
        "        out[i] = min(n + 1, draft.shape[1])\n    return out"),
    "accept length compares with the next target slot": (
        "while n < draft.shape[1] and draft[i, n] == target[i, n]:",
        "while n < draft.shape[1] and draft[i, n] == target[i, min(n + 1, draft.shape[1] - 1)]:"),
    "T=1 acceptance test inverted": (
        "if float(u[i, n]) / 2.0 ** 32 < float(ratio):",
        "if float(u[i, n]) / 2.0 ** 32 > float(ratio):"),
    "T=1 rejection resamples from p, not max(0, p - q)": (
        "res = np.maximum(p_target[i, n] - q_draft[i, n], np.float32(0))      # fp32 subtraction",
        "res = p_target[i, n]      # fp32 subtraction"),
    "T=1 bonus token drawn at the last draft slot": (
        "v = draw(p_target[i, nd], r[i])",
        "v = draw(p_target[i, nd - 1], r[i])"),
    "tau without the bonus token": (
        "return float(np.mean(np.asarray(accept, np.float64) + 1.0))",
        "return float(np.mean(np.asarray(accept, np.float64)))"),
    # ------------------------------------------ drafter projections and layers
    "context keys projected with the value weights": (
        "K = (_f64(c) @ _f64(wk).T).reshape(n, n_heads, head_dim)",
        "K = (_f64(c) @ _f64(wv).T).reshape(n, n_heads, head_dim)"),
    "block keys projected with the query weights": (
        "Kb = store(rope((x @ _f64(lw[\"wk\"]).T).reshape(M, n_heads, head_dim),",
        "Kb = store(rope((x @ _f64(lw[\"wq\"]).T).reshape(M, n_heads, head_dim),"),
    "block values projected with the key weights": (
        "Vb = store(x @ _f64(lw[\"wv\"]).T, A)",
        "Vb = store(x @ _f64(lw[\"wk\"]).T, A)"),
    "block attention skips the block's own keys": (
        "k_all = np.concatenate([Kc[ctx_rows, cols], Kb[rows, cols]], axis=0)\n"
        "                v_all = np.concatenate([Vc[ctx_rows, cols], Vb[rows, cols]], axis=0)",
        "k_all = Kc[ctx_rows, cols] if cu[i + 1] > cu[i] else Kb[rows, cols]\n"
        "                v_all = Vc[ctx_rows, cols] if cu[i + 1] > cu[i] else Vb[rows, cols]"),
    "block attention reads every sequence's context": (
        "ctx_rows = slice(cu[i], cu[i + 1])",
        "ctx_rows = slice(0, cu[-1])"),
    "context positions continue across sequences": (
        "pos_ctx = np.concatenate([np.arange(t) for t in lens]) if cu[-1] else np.zeros(0)",
        "pos_ctx = np.arange(cu[-1])"),
    "a head's output written into another head's columns": (
        "O[rows, cols] = softmax_attention(Q[rows, cols], k_all, v_all)",
        "O[rows, slice((n_heads - 1 - hh) * head_dim, (n_heads - hh) * head_dim)] = softmax_attention(Q[rows, cols], k_all, v_all)"),
    "output projection transposed": (
        "h = store(h + O @ _f64(lw[\"wo\"]).T, \"f32\")",
        "h = store(h + O @ _f64(lw[\"wo\"]), \"f32\")"),
    "down projection applied to the MLP input": (
        "h = store(h + act @ _f64(lw[\"wd\"]).T, \"f32\")",
        "h = store(h + silu(x2 @ _f64(lw[\"wg\"]).T) @ _f64(lw[\"wd\"]).T, \"f32\")"),
    "context rows normalised with the final norm weight": (
        "c = store(rmsnorm(ctx, W[\"ctx_norm\"], norm_eps), A)",
        "c = store(rmsnorm(ctx, W[\"final_norm\"], norm_eps), A)"),
    "every block slot gets the anchor embedding": (
        "h[i * B + 1:(i + 1) * B] = _f64(W[\"mask_vec\"])[None, :]",
        "h[i * B + 1:(i + 1) * B] = _f64(W[\"embed\"])[int(anchor[i])][None, :]"),
    "layers share the first layer's weights": (
        "    for lw in W[\"layers\"]:\n        rec = {}",
        "    for lw in [W[\"layers\"][0]] * len(W[\"layers\"]):\n        rec = {}"),
    "context K/V from the raw reducer output": (
        "        Kc, Vc = context_kv(c, lw[\"wk\"], lw[\"wv\"], pos_ctx, n_heads=n_heads,",
        "        Kc, Vc = context_kv(ctx, lw[\"wk\"], lw[\"wv\"], pos_ctx, n_heads=n_heads,"),
    "draft tokens taken from slots 0..B-2": (
        "return tok[:, 1:]",
        "return tok[:, :-1]"),
    # ----------------------------------------- storage rounding and helpers
    "bf16 rounding half away from zero": (
        "q = np.rint(mant * 256.0) / 256.0        # np.rint: round half to even",
        "q = np.sign(mant) * np.floor(np.abs(mant) * 256.0 + 0.5) / 256.0        # np.rint: round half to even"),
    "bf16 rounding by truncation": (
        "q = np.rint(mant * 256.0) / 256.0        # np.rint: round half to even",
        "q = np.trunc(mant * 256.0) / 256.0        # np.rint: round half to even"),
    "bf16 keeps 9 significant bits": (
        "q = np.rint(mant * 256.0) / 256.0        # np.rint: round half to even",
        "q = np.rint(mant * 512.0) / 512.0        # np.rint: round half to even"),
    "drafter RMSNorm eps outside the square root": (
        "r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)",
        "r = 1.0 / (np.sqrt(np.mean(x * x, axis=-1, keepdims=True)) + eps)"),
    "drafter RMSNorm over the sum of squares": (
        "r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)",
        "r = 1.0 / np.sqrt(np.sum(x * x, axis=-1, keepdims=True) + eps)"),
    "silu is the sigmoid alone": (
        "return x * sigmoid(x)",
        "return sigmoid(x)"),
    "KL divided by the vocabulary size": (
        "return float(t_kd * t_kd / P * np.sum(p * (lp - lq)))",
        "return float(t_kd * t_kd / t.shape[1] * np.sum(p * (lp - lq)))"),
    "reducer output not rounded at its storage point": (
        "    y = np.einsum(\"nj,njd->nd\", alpha, Hh)\n    return store(y, out_dtype), alpha",
        "    y = np.einsum(\"nj,njd->nd\", alpha, Hh)\n    return y, alpha"),
    "attention scale applied twice": (
        "s = (q @ k.T) / math.sqrt(q.shape[-1])",
        "s = (q @ k.T) / q.shape[-1]"),
    "zmax taken from the tempered logits": (
        "zmax = z[np.arange(z.shape[0]), tok]",
        "zmax = z[np.arange(z.shape[0]), tok] * inv_temp"),
    "cross-entropy sign flipped": (
        "out[on] = -ls[np.nonzero(on)[0], labels[on]]",
        "out[on] = ls[np.nonzero(on)[0], labels[on]]"),
    "T=1 residual of q - p instead of p - q": (
        "res = np.maximum(p_target[i, n] - q_draft[i, n], np.float32(0))      # fp32 subtraction",
        "res = np.maximum(q_draft[i, n] - p_target[i, n], np.float32(0))      # fp32 subtraction"),
    "T=1 acceptance ratio q/p": (
        "ratio = np.float32(p_target[i, n, x]) / np.float32(q_draft[i, n, x])   # IEEE fp32 division",
        "ratio = np.float32(q_draft[i, n, x]) / np.float32(p_target[i, n, x])   # IEEE fp32 division"),
    "fc output not rounded at its storage point": (
        "return store(x @ _f64(W_fc).T, out_dtype)",
        "return x @ _f64(W_fc).T"),
    "backward: bias gradient summed over paths": (
        "db = dg.sum(axis=0)",
        "db = np.full(dg.shape[1], dg.sum())"),
    # ---------------------------------------------------------- drafter block
    "swiglu gate and up projections swapped": (
        'act = store(silu(x2 @ _f64(lw["wg"]).T) * (x2 @ _f64(lw["wu"]).T), A)',
        'act = store(silu(x2 @ _f64(lw["wu"]).T) * (x2 @ _f64(lw["wg"]).T), A)'),
    "rotary embedding applied to the context values": (
        "V = store(_f64(c) @ _f64(wv).T, act_dtype)",
        "V = store(rope((_f64(c) @ _f64(wv).T).reshape(n, n_heads, head_dim), pos, theta),"
        " act_dtype).reshape(n, n_heads * head_dim)"),
    "rotary embedding dropped from the context keys": (
        "K = store(rope(K, pos, theta), act_dtype).reshape(n, n_heads * head_dim)",
        "K = store(K, act_dtype).reshape(n, n_heads * head_dim)"),
    "block slot k placed at T + 1 + k": (
        "pos_blk = np.concatenate([lens[i] + np.arange(B) for i in range(batch)])",
        "pos_blk = np.concatenate([lens[i] + 1 + np.arange(B) for i in range(batch)])"),
    "context row t placed at t + 1": (
        "pos_ctx = np.concatenate([np.arange(t) for t in lens]) if cu[-1] else np.zeros(0)",
        "pos_ctx = np.concatenate([np.arange(t) + 1 for t in lens]) if cu[-1] else np.zeros(0)"),
    "context norm weight dropped": (
        'c = store(rmsnorm(ctx, W["ctx_norm"], norm_eps), A)',
        "c = store(rmsnorm(ctx, np.ones(d), norm_eps), A)"),
    "rotary embedding applied to the block values": (
        'Vb = store(x @ _f64(lw["wv"]).T, A)',
        'Vb = store(rope((x @ _f64(lw["wv"]).T).reshape(M, n_heads, head_dim), pos_blk, rope_theta),'
        " A).reshape(M, d)"),
    "block queries not rotated": (
        'Q = store(rope((x @ _f64(lw["wq"]).T).reshape(M, n_heads, head_dim),\n'
        "                       pos_blk, rope_theta), A).reshape(M, d)",
        'Q = store((x @ _f64(lw["wq"]).T), A).reshape(M, d)'),
    "block keys not rotated": (
        'Kb = store(rope((x @ _f64(lw["wk"]).T).reshape(M, n_heads, head_dim),\n'
        "                        pos_blk, rope_theta), A).reshape(M, d)",
        'Kb = store((x @ _f64(lw["wk"]).T), A).reshape(M, d)'),
    "attention keys and values swapped": (
        "O[rows, cols] = softmax_attention(Q[rows, cols], k_all, v_all)",
        "O[rows, cols] = softmax_attention(Q[rows, cols], v_all, k_all)"),
    "attention 1/sqrt(head_dim) scale dropped": (
        "s = (q @ k.T) / math.sqrt(q.shape[-1])",
        "s = q @ k.T"),
    "attention residual dropped": (
        'h = store(h + O @ _f64(lw["wo"]).T, "f32")',
        'h = store(O @ _f64(lw["wo"]).T, "f32")'),
    "MLP residual dropped": (
        'h = store(h + act @ _f64(lw["wd"]).T, "f32")',
        'h = store(act @ _f64(lw["wd"]).T, "f32")'),
    "MLP norm takes the attention norm weight": (
        'x2 = store(rmsnorm(h, lw["mlp_norm"], norm_eps), A)',
        'x2 = store(rmsnorm(h, lw["attn_norm"], norm_eps), A)'),
    "final norm dropped": (
        'return store(rmsnorm(h, W["final_norm"], norm_eps), A)',
        "return store(h, A)"),
    "anchor slot gets the mask vector": (
        'h[i * B] = _f64(W["embed"])[int(anchor[i])]',
        'h[i * B] = _f64(W["mask_vec"])'),
    # ---------------------------------------------------------------- reducer
    "gate computed from the per-path-normed residual": (
        "        alpha = sigmoid(gate_logits(H, Wf, b, rms_eps, gate_scale)) + gate_offset\n",
        "        Hg = H if path_norm_w is None else (H / np.sqrt(np.mean(H * H, axis=2, keepdims=True)"
        " + path_norm_eps) * np.asarray(path_norm_w, np.float64)[None])\n"
        "        alpha = sigmoid(gate_logits(Hg, Wf, b, rms_eps, gate_scale)) + gate_offset\n"),
    "vec() taken element-major": (
        "x = H.reshape(N, m * d)                              # vec(H_t), path-major",
        "x = H.transpose(0, 2, 1).reshape(N, m * d)"),
    "gate bias dropped": (
        "return gate_scale * (x_tilde @ np.asarray(Wf, np.float64).T) + np.asarray(b, np.float64)[None, :]",
        "return gate_scale * (x_tilde @ np.asarray(Wf, np.float64).T)"),
    # ---------------------------------------------------------------- LM head
    "log-softmax temperature ignored": (
        "s = z * inv_temp",
        "s = z"),
    "argmax takes the last index on ties": (
        "tok = np.argmax(z, axis=1)          # numpy returns the first maximiser",
        "tok = z.shape[1] - 1 - np.argmax(z[:, ::-1], axis=1)"),
    # --------------------------------------------------------- fc reducer
    "fc vec() taken element-major": (
        "x = H.reshape(N, m * d_in)                       # vec(H_t), path-major",
        "x = H.transpose(0, 2, 1).reshape(N, m * d_in)"),
    # ------------------------------------------------------ Eq. 3 training loss
    "CE reads the label's neighbour": (
        "out[on] = -ls[np.nonzero(on)[0], labels[on]]",
        "out[on] = -ls[np.nonzero(on)[0], (labels[on] + 1) % ls.shape[1]]"),
    "CE mean over every draft row, supervised or not": (
        "l_ce = float(np.nansum(ce) / n_sup) if n_sup else 0.0",
        "l_ce = float(np.nansum(ce) / len(ce))"),
    "draft positions start at the anchor slot": (
        "draft_rows = np.array([i * block + k for i in range(batch) for k in range(1, block)], np.int64)",
        "draft_rows = np.array([i * block + k - 1 for i in range(batch) for k in range(1, block)], np.int64)"),
    "KL student row off by one": (
        "lq = _log_softmax(S[i * block + k] / t_kd)",
        "lq = _log_softmax(S[i * block + k - 1] / t_kd)"),
    "loss KL without the temperature-squared factor": (
        "l_kl = float(t_kd * t_kd / P * np.sum(kl_rows) / batch) if P",
        "l_kl = float(1.0 / P * np.sum(kl_rows) / batch) if P"),
    "loss KL summed over the batch instead of averaged": (
        "l_kl = float(t_kd * t_kd / P * np.sum(kl_rows) / batch) if P",
        "l_kl = float(t_kd * t_kd / P * np.sum(kl_rows)) if P"),
    "loss KL weight applied to CE": (
        'return {"loss": l_ce + alpha * l_kl,',
        'return {"loss": alpha * l_ce + l_kl,'),
    # --------------------------------------------------------------------- KL
    "KL direction reversed": (
        "return float(t_kd * t_kd / P * np.sum(p * (lp - lq)))",
        "return float(t_kd * t_kd / P * np.sum(np.exp(lq) * (lq - lp)))"),
    "KL temperature-squared factor dropped": (
        "return float(t_kd * t_kd / P * np.sum(p * (lp - lq)))",
        "return float(1.0 / P * np.sum(p * (lp - lq)))"),
}


def _load_oracle(src: str) -> types.ModuleType:
    mod = types.ModuleType("oracle")
    mod.__file__ = ORACLE_SRC
    exec(compile(src, ORACLE_SRC, "exec"), mod.__dict__)
    return mod


def _red_pins(oracle_mod: types.ModuleType):
    """Names of the pins that fail against ``oracle_mod``."""
    saved = sys.modules.get("oracle")
    sys.modules["oracle"] = oracle_mod
    try:
        spec = importlib.util.spec_from_file_location("_pins_against_planted_oracle", PINS)
        pins = importlib.util.module_from_spec(spec)
        spec.loader.exec_module(pins)
    finally:
        if saved is not None:
            sys.modules["oracle"] = saved
        else:
            del sys.modules["oracle"]
    red = []
    for name in sorted(n for n in dir(pins) if n.startswith("test_")):
        try:
            getattr(pins, name)()
        except Exception:  # an assertion, or the slip breaking a shape
            red.append(name)
    return red


def test_unplanted_oracle_passes_every_pin():
    assert _red_pins(_load_oracle(open(ORACLE_SRC).read())) == []


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_turns_a_pin_red(name):
    old, new = MUTATIONS[name]
    src = open(ORACLE_SRC).read()
    assert src.count(old) == 1, f"the text to plant '{name}' in is not in the oracle once"
    red = _red_pins(_load_oracle(src.replace(old, new)))
    assert red, f"no pin fails when the oracle has: {name}"
    print(f"{name}: caught by {', '.join(red)}")
