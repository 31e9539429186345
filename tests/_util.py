"""Shared helpers for the parity tests (comparison metrics only)."""
import numpy as np
import torch

# Tolerances of the parity contract: row-normwise relative error
#   max_i |a_i - b_i| / max_i |b_i|   per row, maximum over rows.
TOL_BF16 = 2e-2      # bf16 outputs, fp32 accumulation
TOL_F32_REDUCE = 1e-5  # fp32 reducer path
TOL_F32_TF32 = 2e-2  # fp32 storage with tf32 tensor-core GEMMs
# reducer gradient (fp32 throughout): the dots behind dg have relative error
# ~sqrt(length)*2^-24 (< 1e-5 at m*d = 28672), which moves sigmoid' by at
# most that relative amount; the token sums add ~sqrt(N)*2^-24 normwise.
TOL_F32_REDUCE_BWD = 1e-4
TIE_BAND = 1e-3      # argmax positions whose oracle top-2 gap is below this are reported apart


def to64(t) -> np.ndarray:
    if isinstance(t, np.ndarray):
        return t.astype(np.float64)
    return t.detach().float().cpu().double().numpy()


def rowwise_rel(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    a2 = a.reshape(a.shape[0], -1) if a.ndim > 1 else a.reshape(1, -1)
    b2 = b.reshape(b.shape[0], -1) if b.ndim > 1 else b.reshape(1, -1)
    num = np.abs(a2 - b2).max(axis=1)
    den = np.maximum(np.abs(b2).max(axis=1), 1e-30)
    return float((num / den).max()) if num.size else 0.0


def exact_fraction(a, b) -> float:
    a = np.asarray(a)
    b = np.asarray(b)
    return float(np.mean(a == b)) if a.size else 1.0


def check_tokens(tok_gpu, z_oracle, band=TIE_BAND):
    """Draft tokens must equal the oracle argmax bit-exactly, except rows whose
    oracle top-2 gap is below ``band``; there the GPU token must be one of the
    oracle's near-maximal entries.  Returns the number of such tie rows."""
    tok_gpu = np.asarray(tok_gpu).astype(np.int64)
    z = np.asarray(z_oracle, np.float64)
    ref = np.argmax(z, axis=1)
    part = np.partition(z, -2, axis=1)
    gap = part[:, -1] - part[:, -2]
    ties = gap < band
    bad = (tok_gpu != ref) & ~ties
    assert not bad.any(), f"token mismatch outside the tie band at rows {np.nonzero(bad)[0][:10]}"
    rows = np.arange(z.shape[0])
    zmax = z.max(axis=1)
    assert np.all(z[rows, tok_gpu] >= zmax - band), "tie-band token not near the maximum"
    return int(ties.sum())
