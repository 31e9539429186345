"""The C-ABI library loads without a GPU, exports every entry point that
include/hdf.h declares, and rejects bad arguments on the host before any
CUDA call (these calls return before touching the device)."""
import ctypes

import pytest

from paper_2606_26744_gb300 import build, hdf


@pytest.fixture(scope="module")
def lib():
    build.build()
    return hdf.load()


def test_every_declared_symbol_is_exported(lib):
    names = hdf.declared_functions()
    assert len(names) >= 13
    for n in ("hdf_gated_reduce", "hdf_draft_block", "hdf_lm_head_argmax", "hdf_accept_len"):
        assert n in names
    for n in names:
        assert hasattr(lib, n), n
    # the binding declares exactly the header's functions
    assert set(hdf._SIGS) == set(names)


def test_status_strings(lib):
    assert lib.hdf_version() == 102
    assert lib.hdf_status_str(0) == b"ok"
    assert b"aligned" in lib.hdf_status_str(4)


def _reduce(lib, **kw):
    a = dict(H=16, dtype=1, n=4, m=4, d=64, Wf=16, b=16, y=16)
    a.update(kw)
    p = lambda v: None if v is None else ctypes.c_void_p(v)
    return lib.hdf_gated_reduce(p(a["H"]), a["dtype"], a["n"], a["m"], a["d"], p(a["Wf"]), p(a["b"]),
                                1e-6, 1.0, 0.0, None, 1e-6, None, p(a["y"]), None, None)


def test_reduce_host_validation(lib):
    assert _reduce(lib, dtype=7) == 3                 # HDF_ERR_DTYPE
    assert _reduce(lib, m=5) == 7                     # HDF_ERR_UNSUPPORTED
    assert _reduce(lib, d=60) == 2                    # d % 8 for bf16
    assert _reduce(lib, n=-1) == 2
    assert _reduce(lib, n=0) == 0                     # empty: nothing launched
    assert _reduce(lib, H=None) == 1                  # HDF_ERR_INVALID_ARG
    assert _reduce(lib, Wf=None) == 1                 # gate weight required without override
    assert _reduce(lib, H=24) == 4                    # HDF_ERR_ALIGNMENT
    assert b"aligned" in lib.hdf_last_error()


def _reduce_bwd(lib, **kw):
    a = dict(H=16, dtype=1, n=4, m=4, d=64, Wf=16, b=16, dy=16, dWf=16, db=16, ws=256, ws_bytes=1 << 20)
    a.update(kw)
    p = lambda v: None if v is None else ctypes.c_void_p(v)
    return lib.hdf_gated_reduce_backward(p(a["H"]), a["dtype"], a["n"], a["m"], a["d"], p(a["Wf"]), p(a["b"]),
                                         1e-6, 1.0, p(a["dy"]), p(a["dWf"]), p(a["db"]), p(a["ws"]),
                                         a["ws_bytes"], None)


def test_reduce_backward_host_validation(lib):
    assert _reduce_bwd(lib, dtype=7) == 3             # HDF_ERR_DTYPE
    assert _reduce_bwd(lib, m=5) == 7                 # HDF_ERR_UNSUPPORTED
    assert _reduce_bwd(lib, d=60) == 2                # d % 8 for bf16
    assert _reduce_bwd(lib, n=-1) == 2
    assert _reduce_bwd(lib, dWf=None) == 1            # outputs required, even for n = 0
    assert _reduce_bwd(lib, n=0, db=None) == 1
    assert _reduce_bwd(lib, dy=None) == 1
    assert _reduce_bwd(lib, H=24) == 4                # HDF_ERR_ALIGNMENT
    assert _reduce_bwd(lib, dWf=40) == 4
    assert _reduce_bwd(lib, ws=None) == 5             # HDF_ERR_WORKSPACE
    assert _reduce_bwd(lib, ws=300) == 5              # not 256-byte aligned
    assert lib.hdf_gated_reduce_backward_workspace_size(4, 4, 64, 1) > 0
    assert lib.hdf_gated_reduce_backward_workspace_size(0, 4, 64, 1) == 0
    assert lib.hdf_gated_reduce_backward_workspace_size(4, 5, 64, 1) == 0   # unsupported m


def test_reduce_kernel_choice_is_validated_per_call(lib):
    v = ctypes.c_void_p
    args = (v(256), 1, 0, 4, 64, v(256), v(256), 1e-6, 1.0, 0.0, None, 1e-6, None, v(256), None, None)
    for kernel in (0, 1, 2, 3):                       # auto, general, cluster, tile: n_tokens = 0 is a no-op
        assert lib.hdf_gated_reduce_kernel(kernel, *args) == 0
    assert lib.hdf_gated_reduce_kernel(4, *args) == 1   # HDF_ERR_INVALID_ARG
    assert lib.hdf_gated_reduce_kernel(-1, *args) == 1


def test_accept_sample_host_validation(lib):
    v = ctypes.c_void_p
    assert lib.hdf_accept_sample(v(16), v(16), v(16), 3, v(16), v(16), 2, 7, 100, v(16), v(16), None) == 2  # stride
    assert lib.hdf_accept_sample(v(16), v(16), v(16), 7, v(16), v(16), 2, 7, 1 << 23, v(16), v(16), None) == 2
    assert lib.hdf_accept_sample(v(16), None, v(16), 7, v(16), v(16), 2, 7, 100, v(16), v(16), None) == 1
    assert lib.hdf_accept_sample(None, None, None, 0, None, None, 0, 7, 100, None, None, None) == 0  # empty


def test_kl_host_validation(lib):
    v = ctypes.c_void_p
    assert lib.hdf_kl_distill(v(16), v(16), 2, 100, 0.0, None, None, v(256), 4096, None) == 1   # t_kd <= 0
    assert lib.hdf_kl_distill(v(16), v(16), -1, 100, 1.0, None, None, v(256), 4096, None) == 2  # rows < 0
    assert lib.hdf_kl_distill(None, None, 0, 100, 1.0, None, None, None, 0, None) == 0         # empty
    assert lib.hdf_kl_distill(v(16), v(24), 2, 100, 1.0, None, None, v(256), 4096, None) == 4  # alignment
    assert lib.hdf_kl_distill(v(16), v(16), 2, 100, 1.0, None, None, None, 0, None) == 5       # workspace
    assert lib.hdf_kl_distill_workspace_size(2, 8193) == 256                                   # 2 x 2 partials


def test_draft_loss_host_validation(lib):
    v = ctypes.c_void_p
    ws = v(256)

    def call(lt=16, ls=16, lab=16, batch=2, block=16, P=2, V=1000, t=1.0, a=0.1, loss=16, w=ws, wb=1 << 20):
        p = lambda x: None if x is None else (x if isinstance(x, ctypes.c_void_p) else v(x))
        return lib.hdf_draft_loss(p(lt), p(ls), p(lab), batch, block, P, V, t, a, None, None, p(loss), p(w), wb,
                                  None)
    assert call(block=1) == 2                    # block < 2
    assert call(P=16) == 2                       # P > block - 1
    assert call(V=0) == 2
    assert call(t=0.0) == 1                      # t_kd <= 0
    assert call(a=float("nan")) == 1
    assert call(batch=0, lt=None, ls=None, lab=None, loss=None, w=None, wb=0) == 0   # empty batch
    assert call(lt=None) == 1                    # teacher needed when P > 0
    assert call(lt=None, P=0, ls=24, w=None, wb=0) == 4   # ... not when P == 0 (the next check fires)
    assert call(lab=None) == 1
    assert call(ls=24) == 4                      # alignment
    assert call(w=None, wb=0) == 5               # workspace
    assert call(w=v(300)) == 5                   # not 256-byte aligned
    assert lib.hdf_draft_loss_workspace_size(2, 2, 8193) == 256       # 4 rows x 2 chunks x 5 floats
    assert lib.hdf_draft_loss_workspace_size(2, 0, 8193) == 0


def test_fc_reduce_host_validation(lib):
    v = ctypes.c_void_p
    assert lib.hdf_fc_reduce(v(16), 1, 4, 4, 64, 100, v(16), v(16), None, 0, None) == 2     # d_out % 128
    assert lib.hdf_fc_reduce(v(16), 1, 4, 3, 7, 128, v(16), v(16), None, 0, None) == 2      # row stride
    assert lib.hdf_fc_reduce(v(16), 9, 4, 4, 64, 128, v(16), v(16), None, 0, None) == 3     # dtype
    assert lib.hdf_fc_reduce(None, 1, 0, 4, 7168, 4096, None, None, None, 0, None) == 0     # empty
    assert lib.hdf_fc_reduce(None, 1, 4, 4, 7168, 4096, v(16), v(16), None, 0, None) == 1
    assert lib.hdf_fc_reduce(v(24), 1, 4, 4, 7168, 4096, v(16), v(16), None, 0, None) == 4


def test_lm_head_and_accept_host_validation(lib):
    v = ctypes.c_void_p
    assert lib.hdf_lm_head_argmax(v(16), 9, 4, 64, v(16), 100, 1.0, v(16), None, None, v(256), 1 << 20, None) == 3
    assert lib.hdf_lm_head_argmax(v(16), 1, 4, 64, v(16), 100, 0.0, v(16), None, None, v(256), 1 << 20, None) == 1
    assert lib.hdf_lm_head_argmax(v(16), 1, 4, 60, v(16), 100, 1.0, v(16), None, None, v(256), 1 << 20, None) == 2
    assert lib.hdf_accept_len(v(16), 3, v(16), 7, 2, 7, v(16), None) == 2   # stride < n_draft
    assert lib.hdf_accept_len(None, 7, v(16), 7, 2, 7, v(16), None) == 1
    assert lib.hdf_accept_len(None, 7, None, 7, 0, 7, None, None) == 0      # empty batch
    assert lib.hdf_accept_len(v(16), 48, v(16), 48, 2, 48, v(16), None) == 7  # n_draft above 47


def test_draft_block_host_validation(lib):
    sh = hdf.DraftShape(1, 1, 16, 2048, 16, 128, 8192, 32768, 1, 2048, 2048, 1e-6)
    w = hdf.DrafterWeights()
    bad = hdf.DraftShape(1, 1, 40, 2048, 16, 128, 8192, 32768, 1, 2048, 2048, 1e-6)   # block > 16
    assert lib.hdf_draft_block(ctypes.byref(w), ctypes.byref(bad), None, None, None, None, None, 0, None, None) == 2
    bad2 = hdf.DraftShape(1, 1, 16, 2000, 16, 125, 8192, 32768, 1, 2048, 2048, 1e-6)  # d % 128
    assert lib.hdf_draft_block(ctypes.byref(w), ctypes.byref(bad2), None, None, None, None, None, 0, None, None) == 2
    assert lib.hdf_draft_block(None, ctypes.byref(sh), None, None, None, None, None, 0, None, None) == 1
    assert lib.hdf_draft_block_workspace_size(ctypes.byref(bad)) == 0


def _fake_weights(n_layers, rope_max_pos):
    """Drafter weights whose pointers are aligned but never dereferenced
    (every call below returns during host validation)."""
    layers = (hdf.LayerWeights * n_layers)()
    for i in range(n_layers):
        for k in ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd"):
            setattr(layers[i], k, 4096)
    w = hdf.DrafterWeights(4096, 4096, 4096, 4096, 4096, 4096, rope_max_pos,
                           ctypes.cast(layers, ctypes.POINTER(hdf.LayerWeights)))
    return w, layers


def test_ctx_cache_host_validation(lib):
    v = ctypes.c_void_p
    w, _keep = _fake_weights(2, 4096 + 16)
    sh = hdf.DraftShape(1, 4, 16, 2048, 16, 128, 8192, 32768, 2, 4096, 20, 1e-6)   # 20 new rows
    good = hdf.CtxCache(4096, 8192, 256, 4096)
    ws = v(1 << 20)
    # append: no cache, zero capacity, misaligned k, rope table too short, workspace too small
    assert lib.hdf_ctx_append(ctypes.byref(w), ctypes.byref(sh), v(4096), v(256), None, ws, 1 << 20, None) == 1
    bad = hdf.CtxCache(4096, 8192, 256, 0)
    assert lib.hdf_ctx_append(ctypes.byref(w), ctypes.byref(sh), v(4096), v(256), ctypes.byref(bad), ws, 1 << 20,
                              None) == 2
    bad = hdf.CtxCache(4100, 8192, 256, 4096)
    assert lib.hdf_ctx_append(ctypes.byref(w), ctypes.byref(sh), v(4096), v(256), ctypes.byref(bad), ws, 1 << 20,
                              None) == 4
    huge = hdf.CtxCache(4096, 8192, 256, 1 << 30)   # batch * capacity >= 2^31 rows
    assert lib.hdf_ctx_append(ctypes.byref(w), ctypes.byref(sh), v(4096), v(256), ctypes.byref(huge), ws, 1 << 20,
                              None) == 2
    w_short, _k2 = _fake_weights(2, 1000)
    assert lib.hdf_ctx_append(ctypes.byref(w_short), ctypes.byref(sh), v(4096), v(256), ctypes.byref(good), ws,
                              1 << 20, None) == 2
    need = lib.hdf_ctx_append_workspace_size(ctypes.byref(sh))
    assert need == ((20 * 2048 * 2 + 255) // 256) * 256
    assert lib.hdf_ctx_append(ctypes.byref(w), ctypes.byref(sh), v(4096), v(256), ctypes.byref(good), ws, need - 1,
                              None) == 5
    assert lib.hdf_ctx_append(ctypes.byref(w), ctypes.byref(sh), None, v(256), ctypes.byref(good), ws, need,
                              None) == 1
    # nothing to append: returns before any launch
    empty = hdf.DraftShape(1, 4, 16, 2048, 16, 128, 8192, 32768, 2, 4096, 0, 1e-6)
    assert lib.hdf_ctx_append(ctypes.byref(w), ctypes.byref(empty), None, None, ctypes.byref(good), None, 0,
                              None) == 0
    # cached block forward: max_ctx above the capacity, no workspace, empty batch
    small = hdf.CtxCache(4096, 8192, 256, 1024)
    assert lib.hdf_draft_block_cached(ctypes.byref(w), ctypes.byref(sh), ctypes.byref(small), v(256), v(4096), ws,
                                      1 << 20, None, None) == 2
    assert lib.hdf_draft_block_cached(ctypes.byref(w), ctypes.byref(sh), ctypes.byref(good), v(256), v(4096), None,
                                      0, None, None) == 5
    assert lib.hdf_draft_block_cached(ctypes.byref(w), ctypes.byref(sh), None, v(256), v(4096), ws, 1 << 20,
                                      None, None) == 1
    nob = hdf.DraftShape(1, 0, 16, 2048, 16, 128, 8192, 32768, 2, 4096, 0, 1e-6)
    assert lib.hdf_draft_block_cached(ctypes.byref(w), ctypes.byref(nob), ctypes.byref(good), None, None, None, 0,
                                      None, None) == 0
    # the cached form needs no context buffers in its workspace
    cold = hdf.DraftShape(1, 4, 16, 2048, 16, 128, 8192, 32768, 2, 4096, 4 * 4096, 1e-6)
    assert (lib.hdf_draft_block_cached_workspace_size(ctypes.byref(cold)) + 3 * 4 * 4096 * 2048 * 2
            <= lib.hdf_draft_block_workspace_size(ctypes.byref(cold)))


def test_draft_round_host_validation(lib):
    v = ctypes.c_void_p
    w, _keep = _fake_weights(2, 4096 + 16)
    sh = hdf.DraftShape(1, 4, 16, 2048, 16, 128, 8192, 32768, 2, 4096, 20, 1e-6)   # 20 new rows
    good = hdf.CtxCache(4096, 8192, 256, 4096)
    ws = v(1 << 24)
    need = lib.hdf_draft_round_workspace_size(ctypes.byref(sh))
    # the append's normed rows, then the cached block's workspace
    assert need == lib.hdf_ctx_append_workspace_size(ctypes.byref(sh)) + \
        lib.hdf_draft_block_cached_workspace_size(ctypes.byref(sh))
    args = lambda **k: [k.get("w", ctypes.byref(w)), k.get("sh", ctypes.byref(sh)), k.get("ctx", v(4096)),
                        k.get("cu", v(256)), k.get("cache", ctypes.byref(good)), k.get("anchor", v(256)),
                        k.get("h", v(4096)), k.get("ws", ws), k.get("nb", need), None]
    assert lib.hdf_draft_round(*args(cache=None)) == 1
    assert lib.hdf_draft_round(*args(ctx=None)) == 1
    assert lib.hdf_draft_round(*args(anchor=None)) == 1
    assert lib.hdf_draft_round(*args(ctx=v(4100))) == 4
    assert lib.hdf_draft_round(*args(h=v(4100))) == 4
    assert lib.hdf_draft_round(*args(nb=need - 1)) == 5
    assert lib.hdf_draft_round(*args(ws=v(1 << 24 | 128))) == 5
    small = hdf.CtxCache(4096, 8192, 256, 1024)   # max_ctx 4096 above the capacity
    assert lib.hdf_draft_round(*args(cache=ctypes.byref(small))) == 2
    w_short, _k2 = _fake_weights(2, 1000)
    assert lib.hdf_draft_round(*args(w=ctypes.byref(w_short))) == 2
    # nothing to append and no block: returns before any launch
    none = hdf.DraftShape(1, 0, 16, 2048, 16, 128, 8192, 32768, 2, 4096, 0, 1e-6)
    assert lib.hdf_draft_round(*args(sh=ctypes.byref(none), ctx=None, cu=None, anchor=None, h=None, ws=None,
                                     nb=0)) == 0
