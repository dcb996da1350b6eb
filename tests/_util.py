"""Shared helpers of the GPU parity tests."""
import numpy as np

# Tolerances of the attention outputs against the fp64 oracle (bf16 inputs,
# fp32 accumulation): max |dO| <= 2e-2, mean |dO| <= 2e-3, |dLSE| <= 1e-3.
MAX_ABS = 2e-2
MEAN_ABS = 2e-3
LSE_ABS = 1e-3


def compare(out, lse, o_ref, lse_ref, what=""):
    """out/lse: device or host torch tensors [rows, Hq, d] / [rows, Hq];
    o_ref/lse_ref: float64 numpy arrays of the same shape."""
    o = out.float().cpu().numpy().astype(np.float64)
    l = lse.float().cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(o)), f"{what}: non-finite output"
    d = np.abs(o - o_ref)
    dl = np.abs(l - lse_ref)
    rel = np.linalg.norm(o - o_ref) / max(np.linalg.norm(o_ref), 1e-30)
    stats = dict(max=float(d.max()), mean=float(d.mean()), lse=float(dl.max()), rel=float(rel))
    assert d.max() <= MAX_ABS, f"{what}: max |dO| {stats}"
    assert d.mean() <= MEAN_ABS, f"{what}: mean |dO| {stats}"
    assert dl.max() <= LSE_ABS, f"{what}: max |dLSE| {stats}"
    assert rel <= 2e-2, f"{what}: relative {stats}"
    return stats


def stack_decode_ref(ref, positions):
    o = np.stack([ref[i][0] for i in positions])
    l = np.stack([ref[i][1] for i in positions])
    return o, l
