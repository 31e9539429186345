"""Plain fp64 CPU oracle for the HyperDFlash block-drafting path.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports this module:
only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may call it.  It shares no code with the CUDA library (no
kernels, headers, tables or helpers); the two meet only through the seeded
inputs of ``paper_2606_26744_gb300.workloads``, which hold no arithmetic.

Every function is the definition written out in numpy float64, step by step
in the paper's order and notation, with a library matmul as the only
primitive.  Where the CUDA path stores an intermediate in bf16 (or fp32),
the oracle rounds to that format at the same point (``store``), so that the
only remaining differences are fp32 accumulation order.

Passages followed (HyperDFlash paper):
  * Eq. 1 (Sec. 2.2): inherited HC-Gate reducer,
        x~ = RMSNorm(vec H_t), alpha = sigmoid(W_f x~ + b), y = sum_j alpha_j H_tj
    with the implementation detail of Sec. 2.2 (scale factor, small offset)
    and the drafter-side per-path RMSNorm (Sec. 2.2, last paragraph).
  * Sec. 2.1 / 2.3: anchor-plus-mask block, draft slot k predicts a+k.
  * Sec. 2.3, Eq. 2: log-softmax at temperature T_KD for the KL target.
  * Sec. 3.4: accepted length; tau counts the bonus token.
  * Sec. 1 / Tables 2-3 (T = 1 rows): speculative-sampling verification,
    accept with probability min(1, p/q) and resample from max(0, p - q).

Readings of passages the paper leaves open are listed in the design notes;
the ones used here are: RMSNorm over all m*d entries with eps and no weight
(the weight folds into W_f), gate alpha_j = sigmoid(s*r*(W_f vec H)_j + b_j)
+ eps_alpha, vec() path-major; drafter = pre-norm MHA + SwiGLU layers whose
context K/V are the layer's W_k/W_v applied to RMSNorm(y); interleaved-pair
RoPE (theta 10000) at positions t (context) and T+k (block slot k).
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np

# ----------------------------------------------------------------------------
# storage formats
# ----------------------------------------------------------------------------


def bf16_round(x) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 (8 significant bits),
    ties to even, returned as float64.  bfloat16 keeps float32's exponent
    range, so for the magnitudes used here (no overflow, no subnormals)
    rounding the frexp mantissa to 8 bits is the whole definition."""
    x = np.asarray(x, dtype=np.float64)
    mant, expo = np.frexp(x)                 # x = mant * 2**expo, |mant| in [0.5, 1)
    q = np.rint(mant * 256.0) / 256.0        # np.rint: round half to even
    return np.ldexp(q, expo)


def store(x, dtype: str) -> np.ndarray:
    """Value after being written in ``dtype`` ('bf16' | 'f32' | 'f64')."""
    x = np.asarray(x, dtype=np.float64)
    if dtype == "bf16":
        return bf16_round(x)
    if dtype == "f32":
        return x.astype(np.float32).astype(np.float64)
    if dtype == "f64":
        return x
    raise ValueError(dtype)


def sigmoid(g) -> np.ndarray:
    g = np.asarray(g, dtype=np.float64)
    out = np.empty_like(g)
    pos = g >= 0
    out[pos] = 1.0 / (1.0 + np.exp(-g[pos]))
    e = np.exp(g[~pos])
    out[~pos] = e / (1.0 + e)
    return out


# ----------------------------------------------------------------------------
# (1) gated residual reducer, Eq. 1
# ----------------------------------------------------------------------------


def gate_logits(H, Wf, b, rms_eps: float = 1e-6, gate_scale: float = 1.0):
    """Pre-sigmoid gate of Eq. 1 for every token: s * (W_f x~_t) + b with
    x~_t = vec(H_t) / sqrt(mean(vec(H_t)^2) + eps).  H: [N, m, d]."""
    H = np.asarray(H, dtype=np.float64)
    N, m, d = H.shape
    x = H.reshape(N, m * d)                              # vec(H_t), path-major
    r = 1.0 / np.sqrt(np.mean(x * x, axis=1) + rms_eps)  # inverse RMS
    x_tilde = x * r[:, None]
    return gate_scale * (x_tilde @ np.asarray(Wf, np.float64).T) + np.asarray(b, np.float64)[None, :]


def gated_reduce(H, Wf, b, *, rms_eps: float = 1e-6, gate_scale: float = 1.0,
                 gate_offset: float = 0.0, path_norm_w=None,
                 path_norm_eps: float = 1e-6, alpha_override=None,
                 out_dtype: str = "bf16"):
    """Eq. 1: y_t = sum_j alpha_tj * H^_tj, alpha = sigmoid(gate) + offset.

    ``path_norm_w`` [m, d] switches on the drafter-side per-path RMSNorm:
    H^_tj = H_tj / rms(H_tj) * gamma_j (the gate still reads the raw H).
    ``alpha_override`` [N, m] replaces the gate (mean pooling, one-hot
    selection).  Returns (y stored in out_dtype, alpha in fp64)."""
    H = np.asarray(H, dtype=np.float64)
    if alpha_override is None:
        alpha = sigmoid(gate_logits(H, Wf, b, rms_eps, gate_scale)) + gate_offset
    else:
        alpha = np.asarray(alpha_override, dtype=np.float64)
    if path_norm_w is None:
        Hh = H
    else:
        rp = 1.0 / np.sqrt(np.mean(H * H, axis=2) + path_norm_eps)   # [N, m]
        Hh = H * rp[:, :, None] * np.asarray(path_norm_w, np.float64)[None, :, :]
    y = np.einsum("nj,njd->nd", alpha, Hh)
    return store(y, out_dtype), alpha


def gated_reduce_backward(H, Wf, b, dy, *, rms_eps: float = 1e-6, gate_scale: float = 1.0):
    """Gradient of Eq. 1 with respect to the reducer's trainable parameters,
    the gate W_f and b (the 65K parameters of Table 1), for the loss
    L = sum_t dy_t . y_t, with H held fixed (the frozen target's residual),
    no per-path norm and no gate override.  The chain rule written out:
        g_tj   = s * r_t * (W_f vec H_t)_j + b_j        (gate_logits)
        a_tj   = dL/dalpha_tj = dy_t . H_tj
        dg_tj  = a_tj * sigmoid(g_tj) * (1 - sigmoid(g_tj))
        dL/db_j    = sum_t dg_tj
        dL/dW_f[j] = sum_t dg_tj * s * r_t * vec(H_t)
    The offset eps_alpha does not enter.  Returns (dW_f [m, m*d], db [m]),
    fp64."""
    H = np.asarray(H, dtype=np.float64)
    N, m, d = H.shape
    dy = np.asarray(dy, dtype=np.float64).reshape(N, d)
    x = H.reshape(N, m * d)
    r = 1.0 / np.sqrt(np.mean(x * x, axis=1) + rms_eps)
    sg = sigmoid(gate_logits(H, Wf, b, rms_eps, gate_scale))
    a = np.einsum("nd,njd->nj", dy, H)
    dg = a * sg * (1.0 - sg)
    db = dg.sum(axis=0)
    dWf = (gate_scale * r[:, None] * dg).T @ x
    return dWf, db


def hc_gate_param_count(m: int, d: int) -> int:
    """Trainable parameters of W_f in Eq. 1 (W_f in R^{m x md})."""
    return m * (m * d)


def fc_param_count(m: int, d: int) -> int:
    """Parameters of the generic fc: R^{md} -> R^d collapse (Sec. 2.2)."""
    return (m * d) * d


def fc_reduce(H, W_fc, out_dtype: str = "f64") -> np.ndarray:
    """Generic fc collapse of vanilla DFlash (Sec. 2.2, Table 1): the learned
    linear map of the flattened residual, y_t = W_fc vec(H_t), vec() path-major
    as in Eq. 1.  W_fc is [d_out, m * d_in]; with d_out != d_in it is the
    fallback the paper names for a drafter narrower or wider than the target."""
    H = _f64(H)
    N, m, d_in = H.shape
    x = H.reshape(N, m * d_in)                       # vec(H_t), path-major
    return store(x @ _f64(W_fc).T, out_dtype)


# ----------------------------------------------------------------------------
# (2) drafter block forward
# ----------------------------------------------------------------------------


def rmsnorm(x, w, eps: float):
    x = np.asarray(x, dtype=np.float64)
    r = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    return x * r * np.asarray(w, np.float64)


def rope(x, pos, theta: float):
    """Rotary embedding on the last axis (head_dim), pairs (2i, 2i+1) turned
    by angle pos * theta^(-2i/head_dim).  x: [n, heads, hd]; pos: [n]."""
    x = np.asarray(x, dtype=np.float64)
    hd = x.shape[-1]
    i = np.arange(hd // 2, dtype=np.float64)
    inv_freq = theta ** (-2.0 * i / hd)
    ang = np.asarray(pos, np.float64)[:, None] * inv_freq[None, :]   # [n, hd/2]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x0 = x[..., 0::2]
    x1 = x[..., 1::2]
    out = np.empty_like(x)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def softmax_attention(q, k, v):
    """softmax(q k^T / sqrt(hd)) v for one head, no mask.  q [nq,hd], k,v [nk,hd]."""
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    s = (q @ k.T) / math.sqrt(q.shape[-1])
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=1, keepdims=True)
    return p @ v


def silu(x):
    x = np.asarray(x, np.float64)
    return x * sigmoid(x)


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def context_kv(c, wk, wv, pos, *, n_heads: int, head_dim: int, theta: float,
               act_dtype: str):
    """Conditioning projection of one layer: K = RoPE(c W_k^T), V = c W_v^T
    for already-normalised context rows c [n, d] at positions pos [n]."""
    n = c.shape[0]
    K = (_f64(c) @ _f64(wk).T).reshape(n, n_heads, head_dim)
    K = store(rope(K, pos, theta), act_dtype).reshape(n, n_heads * head_dim)
    V = store(_f64(c) @ _f64(wv).T, act_dtype)
    return K, V


def draft_block(weights: Dict, ctx, cu_ctx: Sequence[int], anchor: Sequence[int],
                *, block: int, n_heads: int, head_dim: int, rope_theta: float,
                norm_eps: float, act_dtype: str, intermediates: Optional[Dict] = None):
    """One block-drafting forward (Sec. 2.1/2.3 with the drafter reading).

    ctx [N_ctx, d] is the reducer output y; rows cu_ctx[b]:cu_ctx[b+1] belong
    to sequence b.  The block of sequence b is [anchor_b, mask x (B-1)] at
    positions T_b .. T_b+B-1.  Returns the final-normed hidden [batch*B, d]
    stored in act_dtype."""
    W = weights
    ctx = _f64(ctx)
    cu = [int(v) for v in cu_ctx]
    batch = len(cu) - 1
    d = ctx.shape[1]
    B = block
    M = batch * B
    A = act_dtype
    lens = [cu[i + 1] - cu[i] for i in range(batch)]
    pos_ctx = np.concatenate([np.arange(t) for t in lens]) if cu[-1] else np.zeros(0)
    pos_blk = np.concatenate([lens[i] + np.arange(B) for i in range(batch)])

    c = store(rmsnorm(ctx, W["ctx_norm"], norm_eps), A)
    h = np.empty((M, d))
    for i in range(batch):
        h[i * B] = _f64(W["embed"])[int(anchor[i])]
        h[i * B + 1:(i + 1) * B] = _f64(W["mask_vec"])[None, :]
    h = store(h, "f32")
    if intermediates is not None:
        intermediates["c"] = c
        intermediates["h0"] = h.copy()
        intermediates["layers"] = []

    for lw in W["layers"]:
        rec = {}
        Kc, Vc = context_kv(c, lw["wk"], lw["wv"], pos_ctx, n_heads=n_heads,
                            head_dim=head_dim, theta=rope_theta, act_dtype=A)
        x = store(rmsnorm(h, lw["attn_norm"], norm_eps), A)
        Q = store(rope((x @ _f64(lw["wq"]).T).reshape(M, n_heads, head_dim),
                       pos_blk, rope_theta), A).reshape(M, d)
        Kb = store(rope((x @ _f64(lw["wk"]).T).reshape(M, n_heads, head_dim),
                        pos_blk, rope_theta), A).reshape(M, d)
        Vb = store(x @ _f64(lw["wv"]).T, A)
        O = np.empty((M, d))
        for i in range(batch):
            rows = slice(i * B, (i + 1) * B)
            ctx_rows = slice(cu[i], cu[i + 1])
            for hh in range(n_heads):
                cols = slice(hh * head_dim, (hh + 1) * head_dim)
                k_all = np.concatenate([Kc[ctx_rows, cols], Kb[rows, cols]], axis=0)
                v_all = np.concatenate([Vc[ctx_rows, cols], Vb[rows, cols]], axis=0)
                O[rows, cols] = softmax_attention(Q[rows, cols], k_all, v_all)
        O = store(O, A)
        h = store(h + O @ _f64(lw["wo"]).T, "f32")
        h_attn = h.copy()
        x2 = store(rmsnorm(h, lw["mlp_norm"], norm_eps), A)
        act = store(silu(x2 @ _f64(lw["wg"]).T) * (x2 @ _f64(lw["wu"]).T), A)
        h = store(h + act @ _f64(lw["wd"]).T, "f32")
        if intermediates is not None:
            rec.update(Kc=Kc, Vc=Vc, x=x, Q=Q, Kb=Kb, Vb=Vb, O=O, h_attn=h_attn,
                       x2=x2, act=act, h=h.copy())
            intermediates["layers"].append(rec)
    return store(rmsnorm(h, W["final_norm"], norm_eps), A)


# ----------------------------------------------------------------------------
# (3) LM head: logits, argmax drafts, log-softmax at T_KD (Eq. 2)
# ----------------------------------------------------------------------------


def lm_head(h, W_lm, inv_temp: float = 1.0, logsoftmax: bool = False):
    """z = h W_lm^T; tok = first index of the row maximum; optional
    log-softmax of z * inv_temp (the q^{T_KD} of Eq. 2 in log form).
    Returns dict(z, tok, zmax, logsoftmax|None)."""
    z = _f64(h) @ _f64(W_lm).T
    tok = np.argmax(z, axis=1)          # numpy returns the first maximiser
    zmax = z[np.arange(z.shape[0]), tok]
    ls = None
    if logsoftmax:
        s = z * inv_temp
        smax = s.max(axis=1, keepdims=True)
        lse = smax + np.log(np.exp(s - smax).sum(axis=1, keepdims=True))
        ls = s - lse
    return {"z": z, "tok": tok.astype(np.int64), "zmax": zmax, "logsoftmax": ls}


def top2_gap(z) -> np.ndarray:
    """Per row: largest logit minus the second largest (tie detector)."""
    z = _f64(z)
    part = np.partition(z, -2, axis=1)
    return part[:, -1] - part[:, -2]


def draft_tokens(tok, batch: int, block: int) -> np.ndarray:
    """Draft tokens d_1..d_{B-1} of every sequence: block slots 1..B-1
    (slot k predicts the token at a+k; slot 0 is the anchor)."""
    tok = np.asarray(tok).reshape(batch, block)
    return tok[:, 1:]


# ----------------------------------------------------------------------------
# (4) verification
# ----------------------------------------------------------------------------


def accept_len(draft, target) -> np.ndarray:
    """Longest prefix n with draft[i,k] == target[i,k] for all k < n."""
    draft = np.asarray(draft)
    target = np.asarray(target)
    out = np.zeros(draft.shape[0], dtype=np.int64)
    for i in range(draft.shape[0]):
        n = 0
        while n < draft.shape[1] and draft[i, n] == target[i, n]:
            n += 1
        out[i] = n
    return out


def accept_sample(p_target, q_draft, draft, u, r):
    """Temperature-1 verification of one drafted block per sequence by
    speculative sampling (the T = 1 rows of Tables 2 and 3; the rule is the
    standard one the paper relies on without restating it):
      * draft slot k is accepted when u[i,k] / 2^32 < p(x) / q(x), x = draft[i,k],
        with the ratio one IEEE fp32 division; the first rejection ends the block;
      * the next token is drawn from norm(max(0, p - q)) at the rejected slot
        (from p there if that residual is empty), or from p at the bonus slot
        n_draft when every draft is accepted;
      * the draw is an inverse-CDF lookup with the 32-bit uniform r[i] over
        integer weights floor(w * 2^40): the first v whose prefix sum exceeds
        floor(r * R / 2^32), R = total weight (exact integer arithmetic).
    p_target [batch, n_draft + 1, V], q_draft [batch, n_draft, V] float32
    probabilities; draft [batch, n_draft] ids; u [batch, n_draft], r [batch]
    uint32.  Returns (accept [batch], next [batch]); next = -1 when the chosen
    distribution has no weight at all (invalid input)."""
    p_target = np.asarray(p_target, dtype=np.float32)
    q_draft = np.asarray(q_draft, dtype=np.float32)
    draft = np.asarray(draft)
    u = np.asarray(u, dtype=np.uint64)
    r = np.asarray(r, dtype=np.uint64)
    batch, nd = draft.shape
    acc = np.zeros(batch, dtype=np.int64)
    nxt = np.zeros(batch, dtype=np.int64)

    def draw(w32, ri):
        wi = [int(np.floor(float(x) * 2.0 ** 40)) for x in w32]   # exact: w <= 1, float64 product exact
        total = sum(wi)
        if total == 0:
            return None
        thr = (int(ri) * total) >> 32
        run = 0
        for v, x in enumerate(wi):
            run += x
            if run > thr:
                return v
        return len(wi) - 1

    for i in range(batch):
        n = 0
        while n < nd:
            x = int(draft[i, n])
            if x < 0 or x >= p_target.shape[2]:   # an id outside the vocabulary is rejected
                break
            with np.errstate(divide="ignore", invalid="ignore"):   # p/0 = inf (accept), 0/0 = nan (reject)
                ratio = np.float32(p_target[i, n, x]) / np.float32(q_draft[i, n, x])   # IEEE fp32 division
            if float(u[i, n]) / 2.0 ** 32 < float(ratio):
                n += 1
            else:
                break
        acc[i] = n
        if n < nd:
            res = np.maximum(p_target[i, n] - q_draft[i, n], np.float32(0))      # fp32 subtraction
            v = draw(res, r[i])
            if v is None:
                v = draw(p_target[i, n], r[i])
        else:
            v = draw(p_target[i, nd], r[i])
        nxt[i] = -1 if v is None else v
    return acc, nxt


def mean_accepted_length(accept) -> float:
    """tau of Sec. 3.4 per verification round, counting the bonus token the
    target emits after the accepted prefix (tau = mean(n + 1))."""
    return float(np.mean(np.asarray(accept, np.float64) + 1.0))


# ----------------------------------------------------------------------------
# KL distillation target, Eq. 2 (next item on the path; oracle side)
# ----------------------------------------------------------------------------


def kl_distill(teacher_logits, student_logits, t_kd: float = 1.0) -> float:
    """T_KD^2 / P * sum_{k<=P} KL(p_k^T || q_k^T) for P rows of logits, with
    p, q the softmax of the teacher / student logits divided by T_KD."""
    t = _f64(teacher_logits) / t_kd
    s = _f64(student_logits) / t_kd
    lp = t - (t.max(1, keepdims=True) + np.log(np.exp(t - t.max(1, keepdims=True)).sum(1, keepdims=True)))
    lq = s - (s.max(1, keepdims=True) + np.log(np.exp(s - s.max(1, keepdims=True)).sum(1, keepdims=True)))
    p = np.exp(lp)
    P = t.shape[0]
    return float(t_kd * t_kd / P * np.sum(p * (lp - lq)))


# ----------------------------------------------------------------------------
# Training objective of the drafter, Eq. 3 (Sec. 2.3)
# ----------------------------------------------------------------------------


def _log_softmax(z) -> np.ndarray:
    z = _f64(z)
    zmax = z.max(axis=-1, keepdims=True)
    return z - (zmax + np.log(np.exp(z - zmax).sum(axis=-1, keepdims=True)))


def cross_entropy(logits, labels) -> np.ndarray:
    """One-hot supervision of Sec. 2.3 per row: -log softmax(z_r)[label_r].
    A negative label marks a row without supervision; it gets NaN here and
    takes no part in any mean."""
    ls = _log_softmax(logits)
    labels = np.asarray(labels, np.int64)
    out = np.full(ls.shape[0], np.nan)
    on = labels >= 0
    out[on] = -ls[np.nonzero(on)[0], labels[on]]
    return out


def draft_loss(teacher_logits, student_logits, labels, *, block: int, P: int = 2, t_kd: float = 1.0,
               alpha: float = 0.1) -> Dict[str, float]:
    """L = L_CE + alpha * L_KL (Eq. 3) for a batch of drafted blocks.

    student_logits [batch * block, V]: row i * block + k holds z_k of block i
        (k = 0 is the anchor slot, k >= 1 draft position k, which predicts the
        token at a + k);
    labels [batch, block - 1]: the true token at a + k for draft position k
        (negative = unsupervised);
    teacher_logits [batch, P, V]: LMHead(h_{a+k-1}) for k = 1..P.
    L_CE is the mean of the per-position cross-entropy over every supervised
    draft position of the batch (one-hot supervision of the draft logits, at
    temperature 1); L_KL is Eq. 2, T_KD^2 / P * sum_{k=1..P} KL(p_k^T || q_k^T),
    with the expectation taken as the mean over the blocks of the batch.
    Any logits may be passed, log-softmax rows included: both softmaxes are
    unchanged by a constant shift of a row."""
    S = _f64(student_logits)
    Tt = _f64(teacher_logits)
    batch, Pt, V = Tt.shape
    assert Pt == P and S.shape == (batch * block, V)
    labels = np.asarray(labels, np.int64).reshape(batch, block - 1)
    draft_rows = np.array([i * block + k for i in range(batch) for k in range(1, block)], np.int64)
    ce = cross_entropy(S[draft_rows], labels.reshape(-1))
    n_sup = int(np.sum(labels >= 0))
    l_ce = float(np.nansum(ce) / n_sup) if n_sup else 0.0
    kl_rows = np.empty((batch, P))
    for i in range(batch):
        for k in range(1, P + 1):
            lp = _log_softmax(Tt[i, k - 1] / t_kd)
            lq = _log_softmax(S[i * block + k] / t_kd)
            p = np.exp(lp)
            kl_rows[i, k - 1] = np.sum(np.where(p > 0, p * (lp - lq), 0.0))
    l_kl = float(t_kd * t_kd / P * np.sum(kl_rows) / batch) if P else 0.0  # no position distilled: empty sum
    return {"loss": l_ce + alpha * l_kl, "ce": l_ce, "kl": l_kl, "ce_rows": ce, "kl_rows": kl_rows.reshape(-1)}
