"""Seeded synthetic workloads for the HyperDFlash block-drafting path.

This module only *draws* inputs: shapes, dtypes and random values.  It holds
none of the method's arithmetic, so both the CUDA path (tests, bench) and the
fp64 oracle (tests only) can consume the same tensors without sharing code.

Shapes follow the five workloads the paper's setting implies (DeepSeek-V4
style m=4 Hyper-Connection residual, Sec. 2.2; DFlash anchor-plus-mask block,
Sec. 2.1/2.3):

    tiny      m4 d256  T64   B8  L1  4x64   F1024  V1024   fp32, batch 1
    decode    m4 d2048 T2048 B16 L1  16x128 F8192  V32768  bf16, batch 1
    serve     m4 d4096 T~U[512,8192] B16 L1 32x128 F11008 V65536 bf16, batch 32
    large     m4 d7168 T16384 B16 L2 56x128 F18432 V129280 bf16, batch 8 (+log-softmax)
    sweep     reducer only, [N, 4, 7168] bf16, N = 1024 .. 1048576

Value recipe (one torch.Generator per call, drawn in a fixed order):
  * residual H ~ N(0, 1), stored in the workload dtype;
  * every projection weight ~ N(0, 0.02); the gate weight W_f ~ N(0, wf_std)
    (0.02 for the tiny workload, 0.1 elsewhere so the path gates are far
    from uniform); gate bias b ~ N(0, 0.5) in fp32;
  * RMSNorm weights ~ 1 + 0.1 N(0, 1) (not all-ones, so a dropped weight shows);
  * mask vector ~ N(0, 0.02); anchors ~ U[0, V).
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import torch

_TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}


@dataclass(frozen=True)
class DraftConfig:
    """One block-drafting workload (reducer + drafter + LM head + verify)."""

    name: str
    m: int              # Hyper-Connection paths per token
    d: int              # hidden width (target and drafter, Sec. 2.2 assumption)
    block: int          # B = anchor + (B-1) mask slots
    n_layers: int
    n_heads: int
    head_dim: int
    ffn: int            # SwiGLU hidden width
    vocab: int
    batch: int
    ctx_len: int        # T per sequence when fixed
    ctx_len_range: Optional[Sequence[int]] = None  # ragged: T_i ~ U{lo..hi}
    dtype: str = "bf16"
    wf_std: float = 0.1
    logsoftmax: bool = False
    mean_accept: Optional[int] = None   # target tokens give accept ~ U{0..2*mean}
    rope_theta: float = 10000.0
    norm_eps: float = 1e-6

    @property
    def torch_dtype(self) -> torch.dtype:
        return _TORCH_DTYPE[self.dtype]

    @property
    def rows(self) -> int:
        """M = batch * B block rows."""
        return self.batch * self.block


CONFIGS: Dict[str, DraftConfig] = {
    "tiny": DraftConfig("tiny", m=4, d=256, block=8, n_layers=1, n_heads=4,
                        head_dim=64, ffn=1024, vocab=1024, batch=1, ctx_len=64,
                        dtype="f32", wf_std=0.02),
    "decode": DraftConfig("decode", m=4, d=2048, block=16, n_layers=1,
                          n_heads=16, head_dim=128, ffn=8192, vocab=32768,
                          batch=1, ctx_len=2048),
    "serve": DraftConfig("serve", m=4, d=4096, block=16, n_layers=1,
                         n_heads=32, head_dim=128, ffn=11008, vocab=65536,
                         batch=32, ctx_len=8192, ctx_len_range=(512, 8192),
                         mean_accept=4),
    "large": DraftConfig("large", m=4, d=7168, block=16, n_layers=2,
                         n_heads=56, head_dim=128, ffn=18432, vocab=129280,
                         batch=8, ctx_len=16384, logsoftmax=True),
}

SWEEP_D = 7168
SWEEP_M = 4
SWEEP_N = [1024 * 4 ** k for k in range(6)]   # 1024 .. 1048576 tokens


def scaled(cfg: DraftConfig, **over) -> DraftConfig:
    """A copy of ``cfg`` with some fields replaced (small parity cases)."""
    return dataclasses.replace(cfg, **over)


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _randn(shape, std, dtype, g, device, chunk_elems: Optional[int] = None):
    """N(0, std^2) drawn in fp32 then cast; large tensors are drawn in row
    chunks of about chunk_elems values so the fp32 staging buffer stays small
    (same values on one device for a given seed).  Host chunks are kept small
    enough to be reused by the allocator; device chunks are large, so few
    kernels draw them."""
    if chunk_elems is None:
        chunk_elems = 1 << 22 if torch.device(device).type == "cpu" else 1 << 27
    out = torch.empty(shape, dtype=dtype, device=device)
    if out.numel() == 0:  # nothing to draw (e.g. a batch whose contexts are all empty)
        return out
    flat = out.view(shape[0], -1)
    chunk_rows = max(1, chunk_elems // max(1, flat.shape[1]))
    for r0 in range(0, shape[0], chunk_rows):
        r1 = min(shape[0], r0 + chunk_rows)
        t = torch.randn((r1 - r0, flat.shape[1]), generator=g, device=device,
                        dtype=torch.float32)
        if std != 1.0:
            t.mul_(std)
        flat[r0:r1].copy_(t)
    return out


def make_reduce_inputs(n_tokens: int, m: int, d: int, dtype: str = "bf16",
                       wf_std: float = 0.1, seed: int = 0,
                       device="cpu") -> Dict[str, torch.Tensor]:
    """Pre-collapse residual H [N, m, d], gate weight W_f [m, m*d], bias b [m]."""
    g = _gen(seed, device)
    td = _TORCH_DTYPE[dtype]
    H = _randn((n_tokens, m, d), 1.0, td, g, device)
    Wf = _randn((m, m * d), wf_std, td, g, device)
    b = torch.randn((m,), generator=g, device=device, dtype=torch.float32) * 0.5
    return {"H": H, "Wf": Wf, "b": b}


def context_lengths(cfg: DraftConfig, seed: int) -> List[int]:
    """T_i per sequence (fixed, or uniform in the ragged range)."""
    if cfg.ctx_len_range is None:
        return [cfg.ctx_len] * cfg.batch
    lo, hi = cfg.ctx_len_range
    g = _gen(seed + 7919, "cpu")
    return [int(v) for v in torch.randint(lo, hi + 1, (cfg.batch,), generator=g)]


def make_drafter_weights(cfg: DraftConfig, seed: int,
                         device="cpu") -> Dict[str, object]:
    """Random-init drafter weights, all [out, in] row-major."""
    g = _gen(seed, device)
    td = cfg.torch_dtype
    d, F, V = cfg.d, cfg.ffn, cfg.vocab

    def norm_w():
        return (1.0 + 0.1 * torch.randn((d,), generator=g, device=device)).to(td)

    w: Dict[str, object] = {}
    w["embed"] = _randn((V, d), 0.02, td, g, device)
    w["mask_vec"] = _randn((1, d), 0.02, td, g, device).view(d)
    w["ctx_norm"] = norm_w()
    w["final_norm"] = norm_w()
    w["lm_head"] = _randn((V, d), 0.02, td, g, device)
    layers = []
    for _ in range(cfg.n_layers):
        lw = {}
        lw["attn_norm"] = norm_w()
        for k in ("wq", "wk", "wv", "wo"):
            lw[k] = _randn((d, d), 0.02, td, g, device)
        lw["mlp_norm"] = norm_w()
        lw["wg"] = _randn((F, d), 0.02, td, g, device)
        lw["wu"] = _randn((F, d), 0.02, td, g, device)
        lw["wd"] = _randn((d, F), 0.02, td, g, device)
        layers.append(lw)
    w["layers"] = layers
    return w


def make_draft_inputs(cfg: DraftConfig, seed: int, device="cpu",
                      with_weights: bool = True) -> Dict[str, object]:
    """Everything one draft step consumes: the residual of every context token,
    gate parameters, ragged context offsets, anchors and drafter weights."""
    lens = context_lengths(cfg, seed)
    cu = [0]
    for t in lens:
        cu.append(cu[-1] + t)
    red = make_reduce_inputs(cu[-1], cfg.m, cfg.d, cfg.dtype, cfg.wf_std,
                             seed=seed, device=device)
    g = _gen(seed + 104729, "cpu")
    anchor = torch.randint(0, cfg.vocab, (cfg.batch,), generator=g,
                           dtype=torch.int32)
    out: Dict[str, object] = dict(red)
    out["ctx_lens"] = lens
    out["cu_ctx"] = torch.tensor(cu, dtype=torch.int32)
    out["anchor"] = anchor
    if with_weights:
        out["weights"] = make_drafter_weights(cfg, seed + 1, device=device)
    return out


def accept_plan(cfg: DraftConfig, seed: int) -> List[int]:
    """Desired accepted-prefix length per sequence for synthetic targets."""
    g = _gen(seed + 15485863, "cpu")
    nd = cfg.block - 1
    hi = nd if cfg.mean_accept is None else min(nd, 2 * cfg.mean_accept)
    return [int(v) for v in torch.randint(0, hi + 1, (cfg.batch,), generator=g)]


def make_targets(draft: torch.Tensor, accept: Sequence[int], vocab: int,
                 seed: int) -> torch.Tensor:
    """Target tokens [batch, nd] that agree with ``draft`` on exactly the first
    accept[i] slots: equal up to n, a guaranteed mismatch at n, uniform after."""
    draft = draft.to(torch.int64).cpu()
    batch, nd = draft.shape
    g = _gen(seed + 32452843, "cpu")
    tgt = torch.randint(0, vocab, (batch, nd), generator=g, dtype=torch.int64)
    for i in range(batch):
        n = int(accept[i])
        tgt[i, :n] = draft[i, :n]
        if n < nd:
            r = int(torch.randint(0, vocab - 1, (1,), generator=g))
            tgt[i, n] = (int(draft[i, n]) + 1 + r) % vocab
    return tgt.to(torch.int32)
