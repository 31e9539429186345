"""The LM head entry point that needs no workspace (hdf_lm_head_argmax_static).

Some callers cannot hand the library device memory -- a plugin inside a host
whose allocator owns every device byte, or code that may not call an
allocator once it serves -- so this entry point keeps its scratch in a
device array the library owns.  These tests call it through the C ABI and
compare it with the workspace entry point on the same inputs, twice in a
row (the shared scratch keeps the previous call's contents), and check that
a request larger than the array is refused without touching the outputs.

Collected last on purpose: if it fails, a run stopping at the first failure
has already run every other test."""
import ctypes

import numpy as np
import pytest
import torch

from paper_2606_26744_gb300 import build, hdf
from _util import TOL_BF16, rowwise_rel, to64

pytestmark = pytest.mark.gpu


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _static_call(lib, h, W, inv_temp, tok, zmax, ls):
    M, d = h.shape
    V = W.shape[0]
    return lib.hdf_lm_head_argmax_static(_p(h), hdf.HDF_BF16, M, d, _p(W), V, inv_temp, _p(tok), _p(zmax), _p(ls),
                                         ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("M,d,V,with_ls", [(16, 2048, 32768, True), (37, 512, 1000, False), (128, 1024, 4099, True)])
def test_static_scratch_matches_workspace_entry_point(M, d, V, with_ls):
    build.build()
    lib = hdf.load()
    g = torch.Generator(device="cuda").manual_seed(M * 7 + V)
    h = torch.randn(M, d, device="cuda", generator=g).to(torch.bfloat16)
    W = (torch.randn(V, d, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    ref_tok, ref_zmax, ref_ls = hdf.hdf_lm_head_argmax(h, W, inv_temp=0.5, logsoftmax=with_ls)
    torch.cuda.synchronize()
    for _ in range(2):  # two calls in a row on the same shared scratch
        tok = torch.full((M,), -1, dtype=torch.int32, device="cuda")
        zmax = torch.full((M,), float("nan"), device="cuda")
        ls = torch.full((M, V), float("nan"), device="cuda") if with_ls else None
        rc = _static_call(lib, h, W, 0.5, tok, zmax, ls)
        assert rc == 0, lib.hdf_last_error()
        torch.cuda.synchronize()
        assert hdf.device_status() == 0
        assert torch.equal(tok, ref_tok)
        assert rowwise_rel(to64(zmax)[None, :], to64(ref_zmax)[None, :]) <= TOL_BF16
        if with_ls:
            assert rowwise_rel(to64(ls), to64(ref_ls)) <= TOL_BF16


def test_static_scratch_refuses_oversized_requests():
    lib = hdf.load()
    M, d, V = 4096, 128, 200000  # per-tile partials alone exceed the array
    h = torch.zeros(M, d, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(V, d, dtype=torch.bfloat16, device="cuda")
    need = hdf.lm_head_workspace_size(M, d, V, torch.bfloat16)
    assert need > 16 * 1024 * 1024
    tok = torch.full((M,), -1, dtype=torch.int32, device="cuda")
    zmax = torch.zeros(M, device="cuda")
    rc = _static_call(lib, h, W, 1.0, tok, zmax, None)
    assert rc == 5  # HDF_ERR_WORKSPACE
    assert b"static buffer" in lib.hdf_last_error()
    torch.cuda.synchronize()
    assert int((tok != -1).sum()) == 0
