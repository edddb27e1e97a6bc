"""Self-checks of the oracle's KV-cached decode (Alg. 1) on the tiny model.

(a) cached steps equal cache-free whole-sequence recomputation;
(b) causal invariance: later noise never changes earlier slots;
(c) the AR step (k = 0) equals textbook AR sampling by recomputation;
(d) the noise -> token map on the model's logits follows the softmax
    (chi-square over many noise draws);
plus k-prefix invariance (any k <= k_train, Sec. 3.4) and the fixed stride.
"""
import numpy as np
import pytest

import oracle
from synth import TINY, make_noise, make_prompts, make_weights


@pytest.fixture(scope="module")
def tiny():
    cfg = TINY
    return oracle.OracleModel(cfg, make_weights(cfg)), cfg


def _prompts(cfg, B=2, n=12):
    return make_prompts([n] * B, cfg.vocab)


def test_cached_equals_recompute(tiny):
    m, cfg = tiny
    prompts = _prompts(cfg)
    dec = oracle.OracleDecoder(m, map_dtype=np.float64)
    dec.prefill(prompts)
    seqs = [list(p) for p in prompts]
    ks = [2, 2, 3, 0, 1, 2]
    noise = make_noise(len(ks), 2, 3)
    for s, k in enumerate(ks):
        z = noise[s]
        toks, lg = dec.step(k, z, want_logits=True)
        for b in range(2):
            ref = oracle.full_forward_logits(m, seqs[b], z[b], k)
            np.testing.assert_allclose(lg[b, :max(k, 1)], ref, rtol=1e-10, atol=1e-10)
            # the committed sequence is the prompt plus every emitted token
            seqs[b] = seqs[b] + [int(t) for t in toks[b, :max(k, 1)]]
    for b in range(2):
        full = dec.seqs[b]["committed"] + dec.seqs[b]["pending"]
        assert full == seqs[b]


def test_causal_noise_invariance(tiny):
    m, cfg = tiny
    toks = _prompts(cfg, 1, 9)[0]
    z = np.array([0.2, 0.5, 0.7, 0.9], np.float32)
    base = oracle.full_forward_logits(m, toks, z, 4)
    for j in range(4):
        z2 = z.copy()
        z2[j] = np.float32(0.05)
        pert = oracle.full_forward_logits(m, toks, z2, 4)
        np.testing.assert_array_equal(base[:j], pert[:j])
        assert np.abs(base[j] - pert[j]).max() > 1e-6


def test_k_prefix_invariance(tiny):
    m, cfg = tiny
    prompts = _prompts(cfg)
    z = make_noise(1, 2, 4)[0]
    d4 = oracle.OracleDecoder(m)
    d4.prefill(prompts)
    t4, l4 = d4.step(4, z, want_logits=True)
    d2 = oracle.OracleDecoder(m)
    d2.prefill(prompts)
    t2, l2 = d2.step(2, z[:, :2], want_logits=True)
    np.testing.assert_allclose(l2, l4[:, :2], rtol=1e-12, atol=1e-12)
    assert (t2 == t4[:, :2]).all()


def test_ar_step_equals_textbook_sampler(tiny):
    m, cfg = tiny
    prompts = _prompts(cfg, 2, 10)
    T = 6
    zs = make_noise(T, 2, 1)[:, :, 0]
    dec = oracle.OracleDecoder(m)
    dec.prefill(prompts)
    got = np.stack([dec.step(0, zs[t][:, None])[:, 0] for t in range(T)], 1)
    for b in range(2):
        want = oracle.ar_sample(m, prompts[b], zs[:, b])
        assert list(got[b]) == want


def test_gstar_with_model_equals_ar_steps(tiny):
    """G* (App. B) driven by the model as AR oracle equals k AR steps."""
    m, cfg = tiny
    prompt = list(_prompts(cfg, 1, 8)[0])
    z = [0.3, 0.8, 0.55]

    def nxt(tokens):
        return oracle.full_forward_logits(m, tokens)[0]

    g = oracle.gstar(nxt, prompt, z, np.float32)
    assert g == oracle.ar_sample(m, prompt, z)


def test_admit_one_pending_equals_prefill(tiny):
    """Admitting a prompt with one pending token reproduces its prefill state."""
    m, cfg = tiny
    p1, p2, q = (list(x) for x in _prompts(cfg, 3, 9))
    a = oracle.OracleDecoder(m)
    a.prefill([p1, p2])
    b = oracle.OracleDecoder(m)
    b.prefill([p1, q])
    b.admit(1, p2, 1)
    sa, sb = a.seqs[1], b.seqs[1]
    assert sa["committed"] == sb["committed"] and sa["pending"] == sb["pending"]
    for (ka, va), (kb, vb) in zip(sa["cache"], sb["cache"]):
        np.testing.assert_array_equal(ka, kb)
        np.testing.assert_array_equal(va, vb)


def test_admit_pending_tail_equals_cache_free_forward(tiny):
    """A sequence admitted with P pending tokens, stepped once with k noise
    slots, gives the tokens of the cache-free forward over the whole prompt
    plus the noise rows (Alg. 1's first step)."""
    m, cfg = tiny
    p1, p2 = (list(x) for x in _prompts(cfg, 2, 11))
    dec = oracle.OracleDecoder(m)
    dec.prefill([p1, p1])
    k, P = 3, 4
    dec.admit(0, p2, P)
    z = np.array([[0.21, 0.67, 0.93], [0.5, 0.5, 0.5]], np.float32)
    toks = dec.step(k, z)
    lg = oracle.full_forward_logits(m, p2, z[0], k)
    want = [oracle.token_map(cfg, lg[j], z[0, j], np.float32) for j in range(k)]
    assert [int(t) for t in toks[0]] == want


def test_mtp_with_one_head_equals_fully_causal_k1():
    """Standard MTP with k = 1, its head equal to the shared head, is the
    fully causal step with one noise token (both are one noise row decoded
    by the same head)."""
    from synth import TINY
    cfg1 = TINY.replace(mtp_k=1)
    w1 = make_weights(cfg1)
    w0 = {n: a for n, a in w1.items() if n != "w_mtp"}
    w1["w_mtp"] = w1["w_head"][None].copy()
    prompts = make_prompts([7, 10], cfg1.vocab)
    a = oracle.OracleDecoder(oracle.OracleModel(cfg1, w1))
    b = oracle.OracleDecoder(oracle.OracleModel(TINY, w0))
    a.prefill(prompts)
    b.prefill(prompts)
    for z in ([[0.3], [0.9]], [[0.05], [0.61]]):
        z = np.array(z, np.float32)
        ta, la = a.step(1, z, want_logits=True)
        tb, lb = b.step(1, z, want_logits=True)
        np.testing.assert_array_equal(ta, tb)
        np.testing.assert_allclose(la, lb, rtol=0, atol=1e-12)


def test_mtp_step_equals_cache_free_forward():
    """An MTP step after prefill gives the heads' maps of the cache-free
    forward over the whole prompt plus the one noise token."""
    from synth import TINY_MTP as cfg
    w = make_weights(cfg)
    m = oracle.OracleModel(cfg, w)
    p = list(make_prompts([9], cfg.vocab)[0])
    dec = oracle.OracleDecoder(m)
    dec.prefill([p])
    z = np.array([[0.14, 0.52, 0.97]], np.float32)
    toks = dec.step(3, z)
    n = len(p)
    h = np.concatenate([m.token_rows(p, np.arange(n)), m.noise_rows(z[0], np.array([n]))], 0)
    o, _ = m.forward(h, np.arange(n + 1), m.empty_cache())
    lg = m.logits_mtp(o[n])
    want = [oracle.token_map(cfg, lg[j], z[0, j], np.float32) for j in range(3)]
    assert [int(t) for t in toks[0]] == want


def test_map_histogram_matches_softmax(tiny):
    from scipy import stats
    m, cfg = tiny
    toks = _prompts(cfg, 1, 12)[0]
    lg = oracle.full_forward_logits(m, toks)[0]
    p = np.exp(lg - lg.max())
    p /= p.sum()
    rng = np.random.default_rng(11)
    zs = rng.random(60_000)
    hist = np.bincount([oracle.icdf_token(lg, z, np.float64) for z in zs],
                       minlength=cfg.vocab)
    # pool ids into 50 bins of equal expected mass to keep expected counts large
    order = np.arange(cfg.vocab)
    edges = np.searchsorted(np.cumsum(p[order]), np.linspace(0, 1, 51)[1:-1])
    obs = np.add.reduceat(hist, np.r_[0, edges])
    exp = np.add.reduceat(p, np.r_[0, edges]) * len(zs)
    chi = stats.chisquare(obs, exp)
    assert chi.pvalue > 1e-3, chi


def test_fixed_stride(tiny):
    m, cfg = tiny
    dec = oracle.OracleDecoder(m)
    dec.prefill(make_prompts([5, 9], cfg.vocab))
    assert [dec.cached_len(b) for b in range(2)] == [4, 8]
    P = 1
    for k in (2, 3, 0, 2):
        before = [dec.cached_len(b) for b in range(2)]
        dec.step(k, make_noise(1, 2, 3)[0])
        assert [dec.cached_len(b) for b in range(2)] == [x + P for x in before]
        P = max(k, 1) if k > 0 else 1


def test_learned_vs_rope_models_run():
    from synth import TINY
    for pos in ("learned", "rope"):
        cfg = TINY.replace(pos=pos)
        m = oracle.OracleModel(cfg, make_weights(cfg))
        dec = oracle.OracleDecoder(m)
        dec.prefill(make_prompts([6], cfg.vocab))
        t = dec.step(2, make_noise(1, 1, 2)[0])
        assert t.shape == (1, 2) and (0 <= t).all() and (t < cfg.vocab).all()
