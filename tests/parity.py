"""Comparison rules between the CUDA path and the oracle.

fp32 model: the tokens must be identical in every slot.

bf16 model, per head row:
- logits: max |logit_gpu - logit_oracle| <= 3e-2 * (max - min of the oracle's
  logits);
- tokens: every token that differs must be explained by that logit error.
  For the inverse-CDF map, the noise must lie within the first-order CDF
  perturbation delta of *every* bin boundary between the two tokens:
  F(lo), ..., F(hi - 1), where F(v) is the softmax mass of ids <= v.
  For the argmax map, the two logits must be within the error of each other.

A slot is *decidable* when its noise is farther than delta from every CDF
boundary. In such a slot no logit error within the bound can change the
token, so the two sides must agree there. The agreement rate over decidable
slots is the ">= 99.9 %" criterion; the raw agreement over all slots is
recorded beside it. AGREEMENT collects both per test, and conftest.py prints
them at the end of the run.
"""
import numpy as np

LOGIT_TOL = 3e-2     # relative to the oracle row's logit range

# test name -> [slots, mismatches, unexplained, decidable, decidable mismatches]
AGREEMENT = {}


def logit_check(gpu, ref):
    """Returns the worst (max |d| / range) over rows; rows are the last axis."""
    g = np.asarray(gpu, np.float64).reshape(-1, gpu.shape[-1])
    r = np.asarray(ref, np.float64).reshape(-1, ref.shape[-1])
    rng = r.max(1) - r.min(1)
    return float((np.abs(g - r).max(1) / rng).max())


def _cdf_delta(gpu_lg, ref_lg):
    """(F, delta): the oracle's CDF over ids and the first-order bound on how far
    the GPU's logit error moves any point of it."""
    l = np.asarray(ref_lg, np.float64)
    dl = np.asarray(gpu_lg, np.float64) - l
    p = np.exp(l - l.max())
    p /= p.sum()
    F = np.cumsum(p)
    dbar = float((p * dl).sum())
    delta = float((p * np.abs(dl - dbar)).sum())
    # second-order slack, plus the fp32 rounding of the decision itself
    return F, 2.0 * delta + 1e-5


def icdf_mismatch_explained(gpu_lg, ref_lg, z, t_gpu, t_ref) -> bool:
    """z within delta of every CDF boundary between the two tokens' bins."""
    F, delta = _cdf_delta(gpu_lg, ref_lg)
    lo, hi = sorted((int(t_gpu), int(t_ref)))
    bounds = F[lo:hi]                 # F(lo) .. F(hi - 1): the boundaries crossed
    return bool(np.all(np.abs(float(z) - bounds) <= delta))


def icdf_decidable(gpu_lg, ref_lg, z) -> bool:
    """No CDF boundary lies within delta of z."""
    F, delta = _cdf_delta(gpu_lg, ref_lg)
    return bool(np.min(np.abs(F[:-1] - float(z))) > delta) if len(F) > 1 else True


def argmax_mismatch_explained(gpu_lg, ref_lg, t_gpu, t_ref) -> bool:
    l = np.asarray(ref_lg, np.float64)
    dl = np.abs(np.asarray(gpu_lg, np.float64) - l)
    gap = l[int(t_ref)] - l[int(t_gpu)]
    return gap <= dl[int(t_ref)] + dl[int(t_gpu)] + 1e-6


def argmax_decidable(gpu_lg, ref_lg) -> bool:
    """The oracle's top-2 gap exceeds twice the row's logit error."""
    l = np.asarray(ref_lg, np.float64)
    err = float(np.abs(np.asarray(gpu_lg, np.float64) - l).max())
    top2 = np.sort(l)[-2:]
    return bool(top2[1] - top2[0] > 2.0 * err + 1e-6)


def compare_tokens(gpu_tok, ref_tok, gpu_lg, ref_lg, z, map_kind="icdf", stats=None):
    """Returns (n_slots, n_mismatch, n_unexplained). With ``stats`` (a list of
    5 ints) it also accumulates [slots, mismatches, unexplained, decidable
    slots, mismatches among the decidable slots]."""
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
    if stats is not None:
        dec = dec_mism = 0
        for i in range(len(gt)):
            d = icdf_decidable(gl[i], rl[i], zz[i]) if map_kind == "icdf" else \
                argmax_decidable(gl[i], rl[i])
            if d:
                dec += 1
                dec_mism += int(gt[i] != rt[i])
        for j, v in enumerate((len(gt), len(mism), bad, dec, dec_mism)):
            stats[j] += v
    return len(gt), len(mism), bad


def record(name, stats):
    """Keep one test's agreement counts for the end-of-run summary."""
    AGREEMENT[name] = list(stats)
