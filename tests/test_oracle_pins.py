"""Pins of the CPU oracle's primitives against the paper and closed forms.

Each ``check_*`` helper is a pin; ``test_planted_*`` plants a plausible
mistake in the oracle (on the CPU) and shows that the pin catches it.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import ops

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
IDS = {"A": 0, "B": 1, "C": 2}
NAMES = "ABC"


def _num(x):
    return float(Fraction(x)) if isinstance(x, str) else float(x)


def _load_gstar():
    with open(os.path.join(GOLDEN, "gstar_example.json")) as f:
        return json.load(f)


def check_gstar_worked_example(icdf=None):
    """App. B worked example: G* partitions [0,1]^2 into three regions of
    probability 1/3 with half-open bins (z1 = 1/3 exactly gives B)."""
    icdf = icdf or ops.icdf_from_weights
    g = _load_gstar()
    table = {k: np.array([v[c] for c in NAMES], np.float64)
             for k, v in g["ar_table"].items()}

    def draw(z):
        out = []
        for zj in z:
            ctx = "sos" if not out else NAMES[out[-1]]
            out.append(icdf(table[ctx], zj))
        return out

    for pt in g["points"]:
        z = [_num(v) for v in pt["z"]]
        assert draw(z) == [IDS[c] for c in pt["out"]], (pt, draw(z))
    # region probabilities, integrated on a midpoint grid (exact for these
    # axis-aligned regions whose edges fall on grid-cell boundaries)
    n = 120
    grid = (np.arange(n) + 0.5) / n
    counts = {}
    for z1 in grid:
        for z2 in grid:
            key = "".join(NAMES[t] for t in draw([z1, z2]))
            counts[key] = counts.get(key, 0) + 1
    tot = sum(counts.values())
    for key, p in g["probabilities"].items():
        assert abs(counts[key] / tot - float(Fraction(p))) < 1e-9, counts


def check_icdf_bins():
    """Bins are [F(v-1), F(v)): equal weights over 4 ids, z = v/4 exactly."""
    w = np.ones(4)
    assert [ops.icdf_from_weights(w, z) for z in (0.0, 0.2499, 0.25, 0.5, 0.75, 0.9999)] \
        == [0, 0, 1, 2, 3, 3]
    # zero-weight ids are never chosen, even on their boundary
    w = np.array([0.0, 1.0, 0.0, 1.0])
    assert [ops.icdf_from_weights(w, z) for z in (0.0, 0.5, 0.99)] == [1, 3, 3]


def check_icdf_chi_square(icdf_token=None):
    """F^{-1}(z) with z ~ U(0,1) is distributed as the softmax (App. B
    'Correctness'): a chi-square test over 1e5 draws on V = 16."""
    from scipy import stats
    icdf_token = icdf_token or ops.icdf_token
    rng = np.random.default_rng(7)
    logits = rng.normal(0, 1.5, 16)
    p = np.exp(logits - logits.max())
    p /= p.sum()
    zs = rng.random(100_000)
    hist = np.bincount([icdf_token(logits, z, np.float64) for z in zs], minlength=16)
    chi = stats.chisquare(hist, p * len(zs))
    assert chi.pvalue > 1e-3, chi


def test_gstar_worked_example():
    check_gstar_worked_example()


def test_gstar_function_on_example():
    """The same example through oracle.gstar at the logit level."""
    g = _load_gstar()
    with np.errstate(divide="ignore"):
        table = {k: np.log(np.array([v[c] for c in NAMES], np.float64))
                 for k, v in g["ar_table"].items()}

    def nxt(tokens):
        return table["sos"] if not tokens else table[NAMES[tokens[-1]]]

    for z, want in [((0.1, 0.9), "AB"), ((0.5, 0.2), "BA"), ((0.7, 0.75), "BC")]:
        with np.errstate(divide="ignore"):
            got = oracle.gstar(nxt, [], z)
        assert "".join(NAMES[t] for t in got) == want


def test_icdf_bins():
    check_icdf_bins()


def test_icdf_chi_square():
    check_icdf_chi_square()


def test_icdf_bruteforce_small():
    """Against a pure-Python scan over random small weight vectors."""
    rng = np.random.default_rng(3)
    for _ in range(300):
        V = int(rng.integers(1, 9))
        w = rng.random(V) * (rng.random(V) > 0.3)
        if w.sum() == 0:
            w[rng.integers(V)] = 1.0
        z = float(rng.random())
        acc, want = 0.0, None
        S = float(np.sum(w))
        for v in range(V):
            acc += w[v]
            if acc > z * S:
                want = v
                break
        if want is None:
            want = max(v for v in range(V) if w[v] > 0)
        assert ops.icdf_from_weights(w, z) == want


def test_icdf_fallback_at_top():
    """If rounding leaves no prefix above z*S, the largest nonzero id wins."""
    w = np.array([0.3, 0.7, 0.0], np.float32)
    assert ops.icdf_from_weights(w, np.float32(1.0)) == 1


def test_argmax_lowest_tie():
    assert ops.argmax_token(np.array([1.0, 3.0, 3.0, 2.0])) == 1


def check_rmsnorm(rmsnorm=None):
    rmsnorm = rmsnorm or ops.rmsnorm
    x = np.array([3.0, 4.0])
    np.testing.assert_allclose(rmsnorm(x, np.ones(2), 0.0),
                               x / np.sqrt(12.5), rtol=1e-15)
    g = np.array([2.0, -1.0])
    np.testing.assert_allclose(rmsnorm(x, g, 0.0), g * x / np.sqrt(12.5), rtol=1e-15)
    y = np.random.default_rng(0).normal(size=(5, 16))
    np.testing.assert_allclose(rmsnorm(7.5 * y, np.ones(16), 0.0),
                               rmsnorm(y, np.ones(16), 0.0), rtol=1e-13)


def test_rmsnorm_closed_form():
    check_rmsnorm()


def test_gelu_tanh_values():
    # tanh-form GELU at 1 (known constant) and its odd-part identity
    assert abs(ops.gelu_tanh(np.array(1.0)) - 0.8411919906082768) < 1e-15
    assert ops.gelu_tanh(np.array(0.0)) == 0.0
    x = np.linspace(-6, 6, 101)
    np.testing.assert_allclose(ops.gelu_tanh(x) - ops.gelu_tanh(-x), x, atol=1e-14)
    assert abs(ops.gelu_tanh(np.array(20.0)) - 20.0) < 1e-12


def check_rope(apply_rope=None):
    apply_rope = apply_rope or ops.apply_rope
    # head_dim 2: (1, 0) at position 1 rotates by +1 radian
    x = np.array([[[1.0, 0.0]]])
    np.testing.assert_allclose(apply_rope(x, np.array([1]), 1e4)[0, 0],
                               [np.cos(1.0), np.sin(1.0)], rtol=1e-15)
    rng = np.random.default_rng(1)
    q = rng.normal(size=(1, 1, 64))
    k = rng.normal(size=(1, 1, 64))
    # position 0 is the identity
    np.testing.assert_allclose(apply_rope(q, np.array([0]), 1e4), q, rtol=0, atol=0)
    # the score depends only on the offset m - n
    def score(m, n):
        return float(np.sum(apply_rope(q, np.array([m]), 1e4) * apply_rope(k, np.array([n]), 1e4)))
    for m, n, s in [(5, 2, 11), (40, 39, 100), (3, 17, 64)]:
        assert abs(score(m, n) - score(m + s, n + s)) < 1e-10
    # the pair (i, i + 32) rotates with frequency theta^(-2i/64)
    i = 5
    e = np.zeros((1, 1, 64))
    e[0, 0, i] = 1.0
    r = apply_rope(e, np.array([3]), 1e4)[0, 0]
    ang = 3 * 1e4 ** (-2 * i / 64)
    assert abs(r[i] - np.cos(ang)) < 1e-14 and abs(r[i + 32] - np.sin(ang)) < 1e-14


def test_rope():
    check_rope()


def check_attention(attn=None):
    attn = attn or ops.causal_attention
    rng = np.random.default_rng(2)
    m, H, hd = 7, 2, 4
    k = rng.normal(size=(m, H, hd))
    v = rng.normal(size=(m, H, hd))
    kp = np.arange(m)
    qp = np.array([0, 3, 6])
    # zero queries: uniform weights over the visible keys -> prefix means
    out = attn(np.zeros((3, H, hd)), k, v, qp, kp)
    for i, p in enumerate(qp):
        np.testing.assert_allclose(out[i], v[: p + 1].mean(axis=0), rtol=1e-13)
    # keys after a query's position do not affect it
    q = rng.normal(size=(3, H, hd))
    base = attn(q, k, v, qp, kp)
    k2, v2 = k.copy(), v.copy()
    k2[4:] += 5.0
    v2[4:] -= 3.0
    pert = attn(q, k2, v2, qp, kp)
    np.testing.assert_array_equal(base[:2], pert[:2])
    # one strongly matching key takes all the weight
    kk = np.zeros((3, 1, 2))
    kk[1, 0] = [50.0, 0.0]
    vv = np.arange(6.0).reshape(3, 1, 2)
    o = attn(np.array([[[50.0, 0.0]]]), kk, vv, np.array([2]), np.arange(3))
    np.testing.assert_allclose(o[0, 0], vv[1, 0], atol=1e-12)


def test_attention_special_cases():
    check_attention()


def test_sinusoid_closed_form():
    s = ops.sinusoid(np.array([0.0, 0.25]), 8, 1000.0)
    np.testing.assert_allclose(s[0], [1, 1, 1, 1, 0, 0, 0, 0], atol=0)
    freqs = np.exp(-np.log(1e4) * np.arange(4) / 4)
    np.testing.assert_allclose(s[1, :4], np.cos(250.0 * freqs), rtol=1e-14)
    np.testing.assert_allclose(s[1, 4:], np.sin(250.0 * freqs), rtol=1e-14)


def _tiny_model(**kw):
    from synth import TINY, make_weights
    cfg = TINY.replace(**kw)
    return oracle.OracleModel(cfg, make_weights(cfg)), cfg


def check_layer_closed_forms(model_cls=None):
    """Degenerate weights whose decoder layer has a closed form (Table 4
    layer structure: pre-norm attention and MLP, each with a residual)."""
    model_cls = model_cls or oracle.OracleModel
    from synth import TINY, make_weights
    cfg = TINY.replace(n_layer=1, pos="rope")
    w = make_weights(cfg)
    d, H, hd = cfg.d_model, cfg.n_head, cfg.d_model // cfg.n_head
    rng = np.random.default_rng(4)
    h = rng.normal(size=(6, d))
    pos = np.arange(6)
    # (1) all projections zero: the layer is the identity (both residuals)
    w0 = dict(w)
    for name in ("wqkv", "wo", "w_up", "w_down"):
        w0[name] = np.zeros_like(w[name])
    m = model_cls(cfg, w0)
    out, _, _ = m.layer(0, h, pos, *m.empty_cache()[0])
    np.testing.assert_array_equal(out, h)
    # (2) Wq = Wk = 0, Wv = Wo = I, MLP off: h + causal prefix mean of
    #     rmsnorm(h) (uniform attention over positions <= p)
    w1 = dict(w0)
    wqkv = np.zeros((1, 3 * d, d))
    wqkv[0, 2 * d:, :] = np.eye(d)
    w1["wqkv"] = wqkv
    w1["wo"] = np.eye(d)[None]
    m = model_cls(cfg, w1)
    out, _, _ = m.layer(0, h, pos, *m.empty_cache()[0])
    a = h / np.sqrt(np.mean(h * h, axis=1, keepdims=True) + cfg.rms_eps)
    want = h + np.cumsum(a, axis=0) / np.arange(1, 7)[:, None]
    np.testing.assert_allclose(out, want, rtol=1e-12, atol=1e-12)
    # (3) attention off, W_up = I-like, W_down = I-like: h + gelu(rmsnorm(h))
    w2 = dict(w0)
    up = np.zeros((1, cfg.d_ff, d))
    up[0, :d, :] = np.eye(d)
    dn = np.zeros((1, d, cfg.d_ff))
    dn[0, :, :d] = np.eye(d)
    w2["w_up"], w2["w_down"] = up, dn
    m = model_cls(cfg, w2)
    out, _, _ = m.layer(0, h, pos, *m.empty_cache()[0])
    np.testing.assert_allclose(out, h + ops.gelu_tanh(a), rtol=1e-12, atol=1e-12)
    assert H * hd == d


def test_layer_closed_forms():
    check_layer_closed_forms()


# ---------------------------------------------------------- planted mistakes

def _fails(fn, *args):
    try:
        fn(*args)
    except AssertionError:
        return True
    return False


def test_planted_icdf_ge_instead_of_gt():
    def bad(w, z):
        w = np.asarray(w, np.float64)
        p = np.cumsum(w)
        return int(np.argmax(p >= z * p[-1]))
    assert _fails(check_gstar_worked_example, bad)


def test_planted_icdf_reversed_order():
    def bad(w, z):
        w = np.asarray(w, np.float64)[::-1]
        return len(w) - 1 - ops.icdf_from_weights(w, z)
    assert _fails(check_gstar_worked_example, bad)


def test_planted_icdf_wrong_temperature():
    def bad(logits, z, dtype=np.float64):
        l = np.asarray(logits, dtype)
        return ops.icdf_from_weights(np.exp(2.0 * (l - l.max())), z)
    assert _fails(check_icdf_chi_square, bad)


def test_planted_rope_sign():
    def bad(x, pos, theta):
        hd = x.shape[-1]
        half = hd // 2
        ang = ops.rope_angles(pos, hd, theta)[:, None, :]
        c, s = np.cos(ang), np.sin(ang)
        x1, x2 = x[..., :half], x[..., half:]
        return np.concatenate([x1 * c + x2 * s, x2 * c + x1 * s], axis=-1)
    assert _fails(check_rope, bad)


def test_planted_mask_off_by_one():
    def bad(q, k, v, qp, kp):
        hd = q.shape[-1]
        sc = np.einsum("nhd,mhd->hnm", q, k) / np.sqrt(hd)
        mask = np.asarray(kp)[None, :] >= np.asarray(qp)[:, None]
        mask[:, 0] = False
        sc = np.where(mask[None], -np.inf, sc)
        p = np.exp(sc - sc.max(-1, keepdims=True))
        p /= p.sum(-1, keepdims=True)
        return np.einsum("hnm,mhd->nhd", p, v)
    assert _fails(check_attention, bad)


def test_planted_rmsnorm_mean_abs():
    def bad(x, g, eps):
        return x / (np.mean(np.abs(x), axis=-1, keepdims=True) + eps) * g
    assert _fails(check_rmsnorm, bad)


def test_planted_dropped_residual():
    class Bad(oracle.OracleModel):
        def layer(self, li, h, pos, ck, cv):
            out, k, v = super().layer(li, h, pos, ck, cv)
            return out - h + 0.0 * h, k, v   # attention + MLP without the skip
    assert _fails(check_layer_closed_forms, Bad)
