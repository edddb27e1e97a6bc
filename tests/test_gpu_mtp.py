"""The standard MTP variant (Sec. 3.3: one noise-conditioning token, k
independent heads) against the oracle, through the C ABI (needs a GB300).

fp32 model: tokens identical and logits within 1e-4.  bf16: logits within
LOGIT_TOL and every differing token explained (tests/parity.py).
"""
import numpy as np
import pytest

import oracle
from synth import LM1B_MTP, TINY_MTP, make_prompts, make_weights

from parity import LOGIT_TOL, compare_tokens, logit_check

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def kf():
    import __graft_entry__ as g
    g.build()
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_10820_gb300 import kforcing
    return kforcing


def _steps(kf, cfg, w, prompts, ks, seed, flags=0, check=None):
    B = len(prompts)
    dec = kf.Decoder(cfg, w, max_batch=B, max_k=cfg.mtp_k, flags=flags)
    dec.prefill(prompts)
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, w))
    ref.prefill(prompts)
    rng = np.random.default_rng(seed)
    toks = []
    for k in ks:
        z = rng.random((B, max(k, 1)), dtype=np.float32)
        gt = dec.step(k, z)
        gl = dec.logits(max(k, 1))
        rt, rl = ref.step(k, z, want_logits=True)
        check(k, z, gt, rt, gl, rl)
        for b in range(B):
            ref.seqs[b]["pending"] = [int(t) for t in gt[b]]
        assert list(dec.lengths()) == [ref.cached_len(b) for b in range(B)]
        toks.append(gt.copy())
    dec.close()
    return toks


def test_mtp_fp32_tokens_identical(kf):
    cfg = TINY_MTP
    w = make_weights(cfg)
    prompts = make_prompts([9, 14, 5], cfg.vocab)

    def check(k, z, gt, rt, gl, rl):
        assert np.array_equal(gt, rt.astype(np.int32)), (k, gt, rt)
        assert np.abs(gl - rl).max() < 1e-4

    a = _steps(kf, cfg, w, prompts, [3, 3, 0, 3, 3], 41, check=check)
    b = _steps(kf, cfg, w, prompts, [3, 3, 0, 3, 3], 41, flags=kf.KF_FLAG_NO_GRAPH, check=check)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)


def test_mtp_bf16_lm1b(kf):
    cfg = LM1B_MTP
    w = make_weights(cfg)
    prompts = make_prompts([32] * 5, cfg.vocab)
    stats = {"worst": 0.0, "bad": 0}

    def check(k, z, gt, rt, gl, rl):
        stats["worst"] = max(stats["worst"], logit_check(gl, rl))
        stats["bad"] += compare_tokens(gt, rt, gl, rl, z)[2]

    _steps(kf, cfg, w, prompts, [4, 4, 4, 0, 4], 42, check=check)
    assert stats["worst"] <= LOGIT_TOL and stats["bad"] == 0


def test_mtp_rejects_other_k(kf):
    cfg = TINY_MTP
    w = make_weights(cfg)
    dec = kf.Decoder(cfg, w, max_batch=2, max_k=4)
    dec.prefill(make_prompts([6, 6], cfg.vocab))
    with pytest.raises(kf.KfError) as e:
        dec.step(2, np.full((2, 2), 0.5, np.float32))
    assert e.value.code == kf.KF_E_ARG
    dec.step(3, np.full((2, 3), 0.5, np.float32))
    dec.close()
