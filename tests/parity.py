"""Comparison rules between the CUDA path and the oracle.

fp32 model: the tokens must be identical in every slot.
bf16 model: per head row, max |logit_gpu - logit_oracle| <= 3e-2 * (max - min
of the oracle's logits), and every token that differs must be explained by
that logit error: the noise lies within the first-order CDF perturbation of
the bin boundary between the two tokens (inverse-CDF map), or the two
logits are within the error of each other (argmax map).
"""
import numpy as np

LOGIT_TOL = 3e-2     # relative to the oracle row's logit range


def logit_check(gpu, ref):
    """Returns the worst (max |d| / range) over rows; rows are the last axis."""
    g = np.asarray(gpu, np.float64).reshape(-1, gpu.shape[-1])
    r = np.asarray(ref, np.float64).reshape(-1, ref.shape[-1])
    rng = r.max(1) - r.min(1)
    return float((np.abs(g - r).max(1) / rng).max())


def icdf_mismatch_explained(gpu_lg, ref_lg, z, t_gpu, t_ref) -> bool:
    """z within the CDF perturbation of the boundary F(min(t_gpu, t_ref))."""
    l = np.asarray(ref_lg, np.float64)
    dl = np.asarray(gpu_lg, np.float64) - l
    p = np.exp(l - l.max())
    p /= p.sum()
    F = np.cumsum(p)
    dbar = float((p * dl).sum())
    delta = float((p * np.abs(dl - dbar)).sum())
    delta = 2.0 * delta + 1e-5          # second-order slack + fp32 decision rounding
    v = min(int(t_gpu), int(t_ref))
    return abs(float(z) - float(F[v])) <= delta


def argmax_mismatch_explained(gpu_lg, ref_lg, t_gpu, t_ref) -> bool:
    l = np.asarray(ref_lg, np.float64)
    dl = np.abs(np.asarray(gpu_lg, np.float64) - l)
    gap = l[int(t_ref)] - l[int(t_gpu)]
    return gap <= dl[int(t_ref)] + dl[int(t_gpu)] + 1e-6


def compare_tokens(gpu_tok, ref_tok, gpu_lg, ref_lg, z, map_kind="icdf"):
    """Returns (n_slots, n_mismatch, n_unexplained)."""
    gt = np.asarray(gpu_tok).reshape(-1)
    rt = np.asarray(ref_tok).reshape(-1)
    V = gpu_lg.shape[-1]
    gl = np.asarray(gpu_lg).reshape(-1, V)
    rl = np.asarray(ref_lg).reshape(-1, V)
    zz = np.asarray(z).reshape(-1)
    mism = np.nonzero(gt != rt)[0]
    bad = 0
    for i in mism:
        if map_kind == "icdf":
            ok = icdf_mismatch_explained(gl[i], rl[i], zz[i], gt[i], rt[i])
        else:
            ok = argmax_mismatch_explained(gl[i], rl[i], gt[i], rt[i])
        bad += 0 if ok else 1
    return len(gt), len(mism), bad
