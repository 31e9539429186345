"""Thin ctypes binding of libhdf (include/hdf.h).

Argument marshalling only: every step runs in the library's CUDA kernels.
Tensors are torch CUDA tensors (the caller's device memory); calls are
asynchronous on the current torch stream.  If the library is missing the
import of a call raises -- there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Dict, List, Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libhdf.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "hdf.h")

HDF_F32, HDF_BF16 = 0, 1
STAGES_PER_LAYER = 8
_DT = {torch.float32: HDF_F32, torch.bfloat16: HDF_BF16}

c_vp = ctypes.c_void_p
c_i64 = ctypes.c_int64
c_int = ctypes.c_int
c_float = ctypes.c_float
c_size = ctypes.c_size_t


class HdfError(RuntimeError):
    def __init__(self, status: int, detail: str):
        super().__init__(f"hdf status {status}: {detail}")
        self.status = status


class LayerWeights(ctypes.Structure):
    _fields_ = [(n, c_vp) for n in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd")]


class DrafterWeights(ctypes.Structure):
    _fields_ = [("embed", c_vp), ("mask_vec", c_vp), ("ctx_norm", c_vp), ("final_norm", c_vp),
                ("rope_cos", c_vp), ("rope_sin", c_vp), ("rope_max_pos", c_i64),
                ("layers", ctypes.POINTER(LayerWeights))]


class DraftShape(ctypes.Structure):
    _fields_ = [("dtype", c_int), ("batch", c_int), ("block", c_int), ("d", c_int),
                ("n_heads", c_int), ("head_dim", c_int), ("ffn", c_int), ("vocab", c_int),
                ("n_layers", c_int), ("max_ctx", c_int), ("n_ctx", c_i64), ("norm_eps", c_float)]


class Trace(ctypes.Structure):
    _fields_ = [("events", ctypes.POINTER(c_vp)), ("n_events", c_int)]


class DraftWorkspaceLayout(ctypes.Structure):
    _fields_ = [(n, c_size) for n in ("c", "k_ctx", "v_ctx", "h", "x", "q", "k_blk", "v_blk", "o", "act", "total")]


class CtxCache(ctypes.Structure):
    _fields_ = [("k", c_vp), ("v", c_vp), ("len", c_vp), ("capacity", c_int)]


_SIGS = {
    "hdf_version": (c_int, []),
    "hdf_status_str": (ctypes.c_char_p, [c_int]),
    "hdf_last_error": (ctypes.c_char_p, []),
    "hdf_device_status": (c_int, [c_int]),
    "hdf_gated_reduce": (c_int, [c_vp, c_int, c_i64, c_int, c_int, c_vp, c_vp, c_float, c_float,
                                 c_float, c_vp, c_float, c_vp, c_vp, c_vp, c_vp]),
    "hdf_gated_reduce_backward_workspace_size": (c_size, [c_i64, c_int, c_int, c_int]),
    "hdf_gated_reduce_backward": (c_int, [c_vp, c_int, c_i64, c_int, c_int, c_vp, c_vp, c_float, c_float,
                                          c_vp, c_vp, c_vp, c_vp, c_size, c_vp]),
    "hdf_fc_reduce_workspace_size": (c_size, [c_i64, c_int, c_int, c_int, c_int]),
    "hdf_fc_reduce": (c_int, [c_vp, c_int, c_i64, c_int, c_int, c_int, c_vp, c_vp, c_vp, c_size, c_vp]),
    "hdf_draft_block_workspace_size": (c_size, [ctypes.POINTER(DraftShape)]),
    "hdf_draft_block": (c_int, [ctypes.POINTER(DrafterWeights), ctypes.POINTER(DraftShape), c_vp, c_vp,
                                c_vp, c_vp, c_vp, c_size, ctypes.POINTER(Trace), c_vp]),
    "hdf_draft_block_workspace_layout": (c_int, [ctypes.POINTER(DraftShape), ctypes.POINTER(DraftWorkspaceLayout)]),
    "hdf_ctx_append_workspace_size": (c_size, [ctypes.POINTER(DraftShape)]),
    "hdf_ctx_append": (c_int, [ctypes.POINTER(DrafterWeights), ctypes.POINTER(DraftShape), c_vp, c_vp,
                               ctypes.POINTER(CtxCache), c_vp, c_size, c_vp]),
    "hdf_draft_block_cached_workspace_size": (c_size, [ctypes.POINTER(DraftShape)]),
    "hdf_draft_block_cached": (c_int, [ctypes.POINTER(DrafterWeights), ctypes.POINTER(DraftShape),
                                       ctypes.POINTER(CtxCache), c_vp, c_vp, c_vp, c_size, ctypes.POINTER(Trace),
                                       c_vp]),
    "hdf_draft_round_workspace_size": (c_size, [ctypes.POINTER(DraftShape)]),
    "hdf_draft_round": (c_int, [ctypes.POINTER(DrafterWeights), ctypes.POINTER(DraftShape), c_vp, c_vp,
                                ctypes.POINTER(CtxCache), c_vp, c_vp, c_vp, c_size, c_vp]),
    "hdf_rope_table": (c_int, [ctypes.c_double, c_int, c_i64, c_vp, c_vp, c_vp]),
    "hdf_lm_head_workspace_size": (c_size, [c_i64, c_int, c_i64, c_int]),
    "hdf_lm_head_argmax": (c_int, [c_vp, c_int, c_i64, c_int, c_vp, c_i64, c_float, c_vp, c_vp, c_vp,
                                   c_vp, c_size, c_vp]),
    "hdf_accept_len": (c_int, [c_vp, c_i64, c_vp, c_i64, c_int, c_int, c_vp, c_vp]),
    "hdf_lm_head_argmax_static": (c_int, [c_vp, c_int, c_i64, c_int, c_vp, c_i64, c_float, c_vp, c_vp, c_vp,
                                          c_vp]),
    "hdf_gated_reduce_kernel": (c_int, [c_int, c_vp, c_int, c_i64, c_int, c_int, c_vp, c_vp, c_float, c_float,
                                        c_float, c_vp, c_float, c_vp, c_vp, c_vp, c_vp]),
    "hdf_accept_sample": (c_int, [c_vp, c_vp, c_vp, c_i64, c_vp, c_vp, c_int, c_int, c_i64, c_vp, c_vp, c_vp]),
    "hdf_kl_distill_workspace_size": (c_size, [c_i64, c_i64]),
    "hdf_kl_distill": (c_int, [c_vp, c_vp, c_i64, c_i64, c_float, c_vp, c_vp, c_vp, c_size, c_vp]),
    "hdf_draft_loss_workspace_size": (c_size, [c_int, c_int, c_i64]),
    "hdf_draft_loss": (c_int, [c_vp, c_vp, c_vp, c_int, c_int, c_int, c_i64, c_float, c_float, c_vp, c_vp, c_vp,
                               c_vp, c_size, c_vp]),
}

_lib = None


def load() -> ctypes.CDLL:
    """Load libhdf.so from the package directory (built by build())."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2606_26744_gb300.build` (no fallback exists)")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _lib = lib
    return _lib


def declared_functions() -> List[str]:
    """Names of every entry point declared in include/hdf.h."""
    txt = open(HEADER).read()
    return re.findall(r"^HDF_API\s+[\w\s\*]*?\b(hdf_\w+)\s*\(", txt, flags=re.M)


def _check(rc: int):
    if rc != 0:
        lib = load()
        raise HdfError(rc, lib.hdf_last_error().decode())


def _p(t: Optional[torch.Tensor]):
    return None if t is None else c_vp(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return c_vp(s.cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype not in _DT:
        raise TypeError(f"unsupported dtype {t.dtype}")
    return _DT[t.dtype]


def device_status(reset: bool = True) -> int:
    return load().hdf_device_status(1 if reset else 0)


# ----------------------------------------------------------------- reducer
REDUCE_KERNELS = {"auto": 0, "general": 1, "cluster": 2, "tile": 3}


def hdf_gated_reduce_backward(H: torch.Tensor, Wf: torch.Tensor, b: torch.Tensor, dy: torch.Tensor, *,
                              rms_eps: float = 1e-6, gate_scale: float = 1.0, dWf: Optional[torch.Tensor] = None,
                              db: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                              stream=None):
    """Gradient of Eq. 1 with respect to W_f and b for the upstream dy
    (H fixed): returns (dWf [m, m*d] fp32, db [m] fp32)."""
    N, m, d = H.shape
    lib = load()
    if dWf is None:
        dWf = torch.empty((m, m * d), dtype=torch.float32, device=H.device)
    if db is None:
        db = torch.empty(m, dtype=torch.float32, device=H.device)
    if ws is None:
        need = lib.hdf_gated_reduce_backward_workspace_size(N, m, d, _dtype(H))
        ws = torch.empty(max(need, 1), dtype=torch.uint8, device=H.device)
    _check(lib.hdf_gated_reduce_backward(_p(H), _dtype(H), N, m, d, _p(Wf), _p(b), rms_eps, gate_scale, _p(dy),
                                         _p(dWf), _p(db), _p(ws), ws.numel(), _stream(stream)))
    return dWf, db


def hdf_gated_reduce(H: torch.Tensor, Wf: Optional[torch.Tensor], b: Optional[torch.Tensor], *,
                     rms_eps: float = 1e-6, gate_scale: float = 1.0, gate_offset: float = 0.0,
                     path_norm_w: Optional[torch.Tensor] = None, path_norm_eps: float = 1e-6,
                     alpha_override: Optional[torch.Tensor] = None, y: Optional[torch.Tensor] = None,
                     alpha_out: Optional[torch.Tensor] = None, kernel: Optional[str] = None,
                     stream=None) -> torch.Tensor:
    """Eq. 1 reducer: H [N, m, d] -> y [N, d].  ``kernel`` ("general",
    "cluster", "tile", "auto") picks the kernel for this call through
    hdf_gated_reduce_kernel; None calls hdf_gated_reduce."""
    N, m, d = H.shape
    if y is None:
        y = torch.empty((N, d), dtype=H.dtype, device=H.device)
    args = (_p(H), _dtype(H), N, m, d, _p(Wf), _p(b), rms_eps, gate_scale, gate_offset, _p(path_norm_w),
            path_norm_eps, _p(alpha_override), _p(y), _p(alpha_out), _stream(stream))
    if kernel is None:
        _check(load().hdf_gated_reduce(*args))
    else:
        _check(load().hdf_gated_reduce_kernel(REDUCE_KERNELS[kernel], *args))
    return y


def hdf_fc_reduce(H: torch.Tensor, W_fc: torch.Tensor, y: Optional[torch.Tensor] = None,
                  stream=None) -> torch.Tensor:
    """Generic fc collapse y = vec(H) W_fc^T, H [N, m, d_in], W_fc [d_out, m*d_in]
    (the comparison path, and the fallback for unequal widths)."""
    N, m, d_in = H.shape
    d_out = W_fc.shape[0]
    if W_fc.shape[1] != m * d_in:
        raise ValueError(f"W_fc is {tuple(W_fc.shape)}, expected [d_out, {m * d_in}]")
    if y is None:
        y = torch.empty((N, d_out), dtype=H.dtype, device=H.device)
    lib = load()
    wsb = lib.hdf_fc_reduce_workspace_size(N, m, d_in, d_out, _dtype(H))
    ws = torch.empty(max(wsb, 1), dtype=torch.uint8, device=H.device)
    _check(lib.hdf_fc_reduce(_p(H), _dtype(H), N, m, d_in, d_out, _p(W_fc), _p(y), _p(ws), wsb, _stream(stream)))
    return y


def hdf_rope_table(theta: float, head_dim: int, max_pos: int, device, stream=None):
    cos = torch.empty((max_pos, head_dim // 2), dtype=torch.float32, device=device)
    sin = torch.empty_like(cos)
    _check(load().hdf_rope_table(theta, head_dim, max_pos, _p(cos), _p(sin), _stream(stream)))
    return cos, sin


# ----------------------------------------------------------------- drafter
class Drafter:
    """Device-resident drafter weights plus the ctypes structs that point at
    them.  ``weights`` follows workloads.make_drafter_weights (CUDA tensors)."""

    def __init__(self, weights: Dict, *, n_heads: int, head_dim: int, rope_theta: float = 10000.0,
                 rope_max_pos: int, norm_eps: float = 1e-6, stream=None):
        self.w = weights
        emb = weights["embed"]
        self.dtype = _dtype(emb)
        self.vocab, self.d = emb.shape
        self.n_heads, self.head_dim = n_heads, head_dim
        self.n_layers = len(weights["layers"])
        self.ffn = weights["layers"][0]["wg"].shape[0]
        self.norm_eps = norm_eps
        self.rope_cos, self.rope_sin = hdf_rope_table(rope_theta, head_dim, rope_max_pos, emb.device, stream)
        self._layers = (LayerWeights * self.n_layers)()
        for i, lw in enumerate(weights["layers"]):
            for k in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd"):
                setattr(self._layers[i], k, lw[k].data_ptr())
        self._w = DrafterWeights(emb.data_ptr(), weights["mask_vec"].data_ptr(), weights["ctx_norm"].data_ptr(),
                                 weights["final_norm"].data_ptr(), self.rope_cos.data_ptr(),
                                 self.rope_sin.data_ptr(), rope_max_pos,
                                 ctypes.cast(self._layers, ctypes.POINTER(LayerWeights)))

    def shape(self, batch: int, block: int, n_ctx: int, max_ctx: int) -> DraftShape:
        return DraftShape(self.dtype, batch, block, self.d, self.n_heads, self.head_dim, self.ffn, self.vocab,
                          self.n_layers, max_ctx, n_ctx, self.norm_eps)

    def workspace_size(self, batch: int, block: int, n_ctx: int, max_ctx: int) -> int:
        sh = self.shape(batch, block, n_ctx, max_ctx)
        return load().hdf_draft_block_workspace_size(ctypes.byref(sh))

    def workspace_views(self, ws: torch.Tensor, batch: int, block: int, n_ctx: int, max_ctx: int) -> Dict:
        """Views of the intermediates hdf_draft_block leaves in ``ws``
        (hdf_draft_block_workspace_layout): c, k_ctx, v_ctx [n_ctx, d];
        h [M, d] fp32; x, q, k_blk, v_blk, o [M, d]; act [M, F]."""
        sh = self.shape(batch, block, n_ctx, max_ctx)
        lay = DraftWorkspaceLayout()
        _check(load().hdf_draft_block_workspace_layout(ctypes.byref(sh), ctypes.byref(lay)))
        dt = self.w["embed"].dtype
        es = torch.empty((), dtype=dt).element_size()
        M = batch * block

        def view(off, rows, cols, dtype, esz):
            return ws[off:off + rows * cols * esz].view(dtype).view(rows, cols)
        out = {k: view(getattr(lay, k), n_ctx, self.d, dt, es) for k in ("c", "k_ctx", "v_ctx")}
        out["h"] = view(lay.h, M, self.d, torch.float32, 4)
        for k in ("x", "q", "k_blk", "v_blk", "o"):
            out[k] = view(getattr(lay, k), M, self.d, dt, es)
        out["act"] = view(lay.act, M, self.ffn, dt, es)
        return out

    def n_trace_events(self) -> int:
        return 3 + STAGES_PER_LAYER * self.n_layers

    def hdf_draft_block(self, ctx: torch.Tensor, cu_ctx: torch.Tensor, anchor: torch.Tensor, *, block: int,
                        max_ctx: int, h_out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                        events: Optional[Sequence] = None, stream=None) -> torch.Tensor:
        batch = anchor.shape[0]
        n_ctx = ctx.shape[0]
        sh = self.shape(batch, block, n_ctx, max_ctx)
        lib = load()
        need = lib.hdf_draft_block_workspace_size(ctypes.byref(sh))
        if ws is None:
            ws = torch.empty(max(need, 1), dtype=torch.uint8, device=ctx.device)
        if h_out is None:
            h_out = torch.empty((batch * block, self.d), dtype=ctx.dtype, device=ctx.device)
        tr = None
        if events is not None:
            arr = (c_vp * len(events))(*[e.cuda_event for e in events])
            tr = Trace(ctypes.cast(arr, ctypes.POINTER(c_vp)), len(events))
            self._keep = arr
        _check(lib.hdf_draft_block(ctypes.byref(self._w), ctypes.byref(sh), _p(ctx), _p(cu_ctx), _p(anchor),
                                   _p(h_out), _p(ws), ws.numel(), ctypes.byref(tr) if tr is not None else None,
                                   _stream(stream)))
        return h_out

    # ------------------------------------------------ incremental (cached) form
    def new_cache(self, batch: int, capacity: int, device, zero: bool = False) -> "ContextCache":
        """Per-layer K_c / V_c cache [n_layers, batch, capacity, d] and the
        device row counts (zero: an empty cache for every sequence)."""
        return ContextCache(self.n_layers, batch, capacity, self.d, self.w["embed"].dtype, device, zero)

    def append_workspace_size(self, batch: int, block: int, n_new: int) -> int:
        sh = self.shape(batch, block, n_new, 0)
        return load().hdf_ctx_append_workspace_size(ctypes.byref(sh))

    def cached_workspace_size(self, batch: int, block: int, max_ctx: int) -> int:
        sh = self.shape(batch, block, 0, max_ctx)
        return load().hdf_draft_block_cached_workspace_size(ctypes.byref(sh))

    def hdf_ctx_append(self, ctx_new: torch.Tensor, cu_new: torch.Tensor, cache: "ContextCache", *, block: int,
                       ws: Optional[torch.Tensor] = None, stream=None) -> None:
        batch = cu_new.shape[0] - 1
        sh = self.shape(batch, block, ctx_new.shape[0], 0)
        lib = load()
        if ws is None:
            ws = torch.empty(max(lib.hdf_ctx_append_workspace_size(ctypes.byref(sh)), 1), dtype=torch.uint8,
                             device=ctx_new.device)
        _check(lib.hdf_ctx_append(ctypes.byref(self._w), ctypes.byref(sh), _p(ctx_new), _p(cu_new),
                                  ctypes.byref(cache.c), _p(ws), ws.numel(), _stream(stream)))

    def hdf_draft_block_cached(self, cache: "ContextCache", anchor: torch.Tensor, *, block: int, max_ctx: int,
                               h_out: Optional[torch.Tensor] = None, ws: Optional[torch.Tensor] = None,
                               events: Optional[Sequence] = None, stream=None) -> torch.Tensor:
        batch = anchor.shape[0]
        sh = self.shape(batch, block, 0, max_ctx)
        lib = load()
        dev = anchor.device
        if ws is None:
            ws = torch.empty(max(lib.hdf_draft_block_cached_workspace_size(ctypes.byref(sh)), 1),
                             dtype=torch.uint8, device=dev)
        if h_out is None:
            h_out = torch.empty((batch * block, self.d), dtype=self.w["embed"].dtype, device=dev)
        tr = None
        if events is not None:
            arr = (c_vp * len(events))(*[e.cuda_event for e in events])
            tr = Trace(ctypes.cast(arr, ctypes.POINTER(c_vp)), len(events))
            self._keep = arr
        _check(lib.hdf_draft_block_cached(ctypes.byref(self._w), ctypes.byref(sh), ctypes.byref(cache.c),
                                          _p(anchor), _p(h_out), _p(ws), ws.numel(),
                                          ctypes.byref(tr) if tr is not None else None, _stream(stream)))
        return h_out


    def round_workspace_size(self, batch: int, block: int, n_new: int, max_ctx: int) -> int:
        sh = self.shape(batch, block, n_new, max_ctx)
        return load().hdf_draft_round_workspace_size(ctypes.byref(sh))

    def hdf_draft_round(self, ctx_new: torch.Tensor, cu_new: torch.Tensor, cache: "ContextCache",
                        anchor: torch.Tensor, *, block: int, max_ctx: int, h_out: Optional[torch.Tensor] = None,
                        ws: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        """hdf_ctx_append(ctx_new, cu_new) then hdf_draft_block_cached, in one
        call whose first block path runs beside the append."""
        batch = anchor.shape[0]
        sh = self.shape(batch, block, ctx_new.shape[0], max_ctx)
        lib = load()
        dev = anchor.device
        if ws is None:
            ws = torch.empty(max(lib.hdf_draft_round_workspace_size(ctypes.byref(sh)), 1), dtype=torch.uint8,
                             device=dev)
        if h_out is None:
            h_out = torch.empty((batch * block, self.d), dtype=self.w["embed"].dtype, device=dev)
        _check(lib.hdf_draft_round(ctypes.byref(self._w), ctypes.byref(sh), _p(ctx_new), _p(cu_new),
                                   ctypes.byref(cache.c), _p(anchor), _p(h_out), _p(ws), ws.numel(),
                                   _stream(stream)))
        return h_out


class ContextCache:
    """Device tensors of an hdf_ctx_cache: k, v [n_layers, batch, capacity, d]
    and len [batch] int32 (rows held per sequence)."""

    def __init__(self, n_layers: int, batch: int, capacity: int, d: int, dtype: torch.dtype, device,
                 zero: bool = False):
        alloc = torch.zeros if zero else torch.empty
        self.k = alloc((n_layers, batch, capacity, d), dtype=dtype, device=device)
        self.v = alloc((n_layers, batch, capacity, d), dtype=dtype, device=device)
        self.len = torch.zeros((batch,), dtype=torch.int32, device=device)
        self.capacity = capacity
        self.c = CtxCache(self.k.data_ptr(), self.v.data_ptr(), self.len.data_ptr(), capacity)


# ----------------------------------------------------------------- LM head
def lm_head_workspace_size(M: int, d: int, V: int, dtype: torch.dtype) -> int:
    return load().hdf_lm_head_workspace_size(M, d, V, _DT[dtype])


def hdf_lm_head_argmax(h: torch.Tensor, W_lm: torch.Tensor, *, inv_temp: float = 1.0,
                       logsoftmax: bool = False, tok: Optional[torch.Tensor] = None,
                       zmax: Optional[torch.Tensor] = None, ls: Optional[torch.Tensor] = None,
                       ws: Optional[torch.Tensor] = None, stream=None):
    M, d = h.shape
    V = W_lm.shape[0]
    dev = h.device
    if tok is None:
        tok = torch.empty((M,), dtype=torch.int32, device=dev)
    if zmax is None:
        zmax = torch.empty((M,), dtype=torch.float32, device=dev)
    if logsoftmax and ls is None:
        ls = torch.empty((M, V), dtype=torch.float32, device=dev)
    lib = load()
    need = lib.hdf_lm_head_workspace_size(M, d, V, _dtype(h))
    if ws is None:
        ws = torch.empty(max(need, 1), dtype=torch.uint8, device=dev)
    _check(lib.hdf_lm_head_argmax(_p(h), _dtype(h), M, d, _p(W_lm), V, inv_temp, _p(tok), _p(zmax),
                                  _p(ls) if logsoftmax else None, _p(ws), ws.numel(), _stream(stream)))
    return tok, zmax, (ls if logsoftmax else None)


def hdf_lm_head_argmax_static(h: torch.Tensor, W_lm: torch.Tensor, *, inv_temp: float = 1.0,
                              logsoftmax: bool = False, tok: Optional[torch.Tensor] = None,
                              zmax: Optional[torch.Tensor] = None, ls: Optional[torch.Tensor] = None,
                              stream=None):
    """LM head on the library's own scratch array: for callers that cannot
    give the library device memory for a workspace.  Outputs are still the
    caller's; calls that overlap on the GPU share the scratch and race."""
    M, d = h.shape
    V = W_lm.shape[0]
    dev = h.device
    if tok is None:
        tok = torch.empty((M,), dtype=torch.int32, device=dev)
    if zmax is None:
        zmax = torch.empty((M,), dtype=torch.float32, device=dev)
    if logsoftmax and ls is None:
        ls = torch.empty((M, V), dtype=torch.float32, device=dev)
    _check(load().hdf_lm_head_argmax_static(_p(h), _dtype(h), M, d, _p(W_lm), V, inv_temp, _p(tok), _p(zmax),
                                            _p(ls) if logsoftmax else None, _stream(stream)))
    return tok, zmax, (ls if logsoftmax else None)


# ------------------------------------------------------------------ verify
def hdf_accept_len(draft: torch.Tensor, target: torch.Tensor, *, n_draft: Optional[int] = None,
                   draft_stride: Optional[int] = None, batch: Optional[int] = None,
                   accept: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """draft/target int32; rows of n_draft entries at the given strides."""
    if batch is None:
        batch = target.shape[0]
    if n_draft is None:
        n_draft = target.shape[1]
    if draft_stride is None:
        draft_stride = draft.stride(0) if draft.dim() == 2 else n_draft
    if accept is None:
        accept = torch.empty((batch,), dtype=torch.int32, device=target.device)
    _check(load().hdf_accept_len(_p(draft), draft_stride, _p(target), target.stride(0), batch, n_draft,
                                 _p(accept), _stream(stream)))
    return accept


# ---------------------------------------------------------- KL distillation
def hdf_kl_distill(ls_teacher: torch.Tensor, ls_student: torch.Tensor, *, t_kd: float = 1.0,
                   kl_rows: Optional[torch.Tensor] = None, kl_mean: Optional[torch.Tensor] = None,
                   ws: Optional[torch.Tensor] = None, stream=None):
    """Eq. 2: per-row KL(p || q) of two [rows, V] fp32 log-softmax arrays at
    temperature t_kd, and t_kd^2 / rows * their sum."""
    rows, V = ls_teacher.shape
    dev = ls_teacher.device
    if kl_rows is None:
        kl_rows = torch.empty((rows,), dtype=torch.float32, device=dev)
    if kl_mean is None:
        kl_mean = torch.empty((1,), dtype=torch.float32, device=dev)
    lib = load()
    need = lib.hdf_kl_distill_workspace_size(rows, V)
    if ws is None:
        ws = torch.empty(max(need, 1), dtype=torch.uint8, device=dev)
    _check(lib.hdf_kl_distill(_p(ls_teacher), _p(ls_student), rows, V, t_kd, _p(kl_rows), _p(kl_mean), _p(ws),
                              ws.numel(), _stream(stream)))
    return kl_rows, kl_mean


# ------------------------------------------------ training objective, Eq. 3
def hdf_draft_loss(ls_teacher: Optional[torch.Tensor], ls_student: torch.Tensor, labels: torch.Tensor, *,
                   block: int, t_kd: float = 1.0, alpha: float = 0.1, ce_rows: Optional[torch.Tensor] = None,
                   kl_rows: Optional[torch.Tensor] = None, loss: Optional[torch.Tensor] = None,
                   ws: Optional[torch.Tensor] = None, stream=None):
    """Eq. 3, L = L_CE + alpha * L_KL: ls_teacher [batch, P, V] (or None for
    P = 0) and ls_student [batch * block, V] fp32 log-softmax rows at
    temperature 1, labels [batch, block - 1] int32 (< 0 = unsupervised).
    Returns (loss [3] = {L, L_CE, L_KL}, ce_rows [batch, block-1], kl_rows
    [batch, P])."""
    V = ls_student.shape[1]
    batch = ls_student.shape[0] // block
    P = 0 if ls_teacher is None else ls_teacher.shape[1]
    dev = ls_student.device
    if ce_rows is None:
        ce_rows = torch.empty((batch, block - 1), dtype=torch.float32, device=dev)
    if kl_rows is None:
        kl_rows = torch.empty((batch, max(P, 1)), dtype=torch.float32, device=dev)
    if loss is None:
        loss = torch.empty((3,), dtype=torch.float32, device=dev)
    lib = load()
    need = lib.hdf_draft_loss_workspace_size(batch, P, V)
    if ws is None:
        ws = torch.empty(max(need, 1), dtype=torch.uint8, device=dev)
    _check(lib.hdf_draft_loss(_p(ls_teacher) if P > 0 else None, _p(ls_student), _p(labels), batch, block, P, V,
                              t_kd, alpha, _p(ce_rows), _p(kl_rows) if P > 0 else None, _p(loss), _p(ws),
                              ws.numel(), _stream(stream)))
    return loss, ce_rows, kl_rows[:, :P]


# ------------------------------------------------------ T = 1 verification
def hdf_accept_sample(p_target: torch.Tensor, q_draft: torch.Tensor, draft: torch.Tensor, u: torch.Tensor,
                      r: torch.Tensor, *, accept: Optional[torch.Tensor] = None,
                      next_tok: Optional[torch.Tensor] = None, stream=None):
    """Speculative-sampling verification: p_target [batch, n+1, V], q_draft
    [batch, n, V] fp32 probabilities, draft [batch, n] int32 (row stride
    draft.stride(0)), u [batch, n] and r [batch] uint32 uniforms (int32
    tensors holding the same bits).  Returns (accept, next_tok) int32."""
    batch, n1, V = p_target.shape
    nd = n1 - 1
    dev = p_target.device
    if accept is None:
        accept = torch.empty((batch,), dtype=torch.int32, device=dev)
    if next_tok is None:
        next_tok = torch.empty((batch,), dtype=torch.int32, device=dev)
    _check(load().hdf_accept_sample(_p(p_target), _p(q_draft) if nd > 0 else None, _p(draft) if nd > 0 else None,
                                    draft.stride(0) if nd > 0 else 0, _p(u) if nd > 0 else None, _p(r), batch, nd,
                                    V, _p(accept), _p(next_tok), _stream(stream)))
    return accept, next_tok
