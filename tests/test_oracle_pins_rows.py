"""Pins of the oracle's input rows, noise encoder and head.

They cover the noise encoder (Table 4), the noise rows and their positions
(Alg. 1: h = [h_x; h_z]), the token rows with learned positions, and the
head: final RMSNorm, untied LM head, then division by tau (Sec. 3.4).

Each ``check_*`` is a pin against degenerate weights whose output has a
closed form. Each ``test_planted_*`` plants a plausible mistake in the oracle,
on the CPU, and shows that the pin fails on it.
"""
import numpy as np

import oracle
from oracle import ops
from synth import TINY, make_weights


def _fails(fn, *args):
    try:
        fn(*args)
    except AssertionError:
        return True
    return False


# ------------------------------------------------------------ noise encoder

def check_noise_encoder(enc=None):
    """NoiseEnc(s) = W2 gelu(W1 s + b1) + b2 (Table 4: a two-layer MLP with GELU
    on the sinusoidal features). With W1 = [I; 0] and W2 = [I 0] the first d
    hidden units pass through and the result is gelu(s + b1[:d]) + b2 exactly.
    A W2 that reads the second block of hidden units shows that the hidden
    width is W1's row count (4d), not d."""
    enc = enc or ops.noise_encoder
    rng = np.random.default_rng(11)
    n, d, h = 5, 16, 64
    s = rng.normal(size=(n, d))
    w1 = np.zeros((h, d))
    w1[:d] = np.eye(d)
    w2 = np.zeros((d, h))
    w2[:, :d] = np.eye(d)
    zero_h, zero_d = np.zeros(h), np.zeros(d)
    # 1. pass-through: gelu(s) with zero biases
    np.testing.assert_allclose(enc(s, w1, zero_h, w2, zero_d), ops.gelu_tanh(s), rtol=0, atol=1e-15)
    # 2. b1 enters before the GELU, b2 after it
    b1 = rng.normal(size=h)
    b2 = rng.normal(size=d)
    np.testing.assert_allclose(enc(s, w1, b1, w2, b2), ops.gelu_tanh(s + b1[:d]) + b2,
                               rtol=0, atol=1e-14)
    # 3. the second block of d hidden units, reached through rows d..2d-1 of W1
    w1b = np.zeros((h, d))
    w1b[d:2 * d] = 2.0 * np.eye(d)
    w2b = np.zeros((d, h))
    w2b[:, d:2 * d] = np.eye(d)
    np.testing.assert_allclose(enc(s, w1b, zero_h, w2b, zero_d), ops.gelu_tanh(2.0 * s),
                               rtol=0, atol=1e-15)
    # 4. a negative input is bent by the GELU (gelu(-3) is about -0.004, not -3)
    neg = np.full((1, d), -3.0)
    out = enc(neg, w1, zero_h, w2, zero_d)
    assert np.all(np.abs(out) < 0.01), out


def test_noise_encoder_closed_forms():
    check_noise_encoder()


def test_planted_noise_encoder_gelu_after_w2():
    def bad(feat, w1, b1, w2, b2):
        return ops.gelu_tanh((feat @ w1.T + b1) @ w2.T + b2)
    assert _fails(check_noise_encoder, bad)


def test_planted_noise_encoder_swapped_bias():
    def bad(feat, w1, b1, w2, b2):
        return ops.gelu_tanh(feat @ w1.T + np.resize(b2, b1.shape)) @ w2.T + b1[: w2.shape[0]]
    assert _fails(check_noise_encoder, bad)


def test_planted_noise_encoder_no_gelu():
    def bad(feat, w1, b1, w2, b2):
        return (feat @ w1.T + b1) @ w2.T + b2
    assert _fails(check_noise_encoder, bad)


# ------------------------------------------------------------ probe models

def _probe_weights(cfg, tok_onehot=False):
    """Degenerate weights for a learned-position model with V = d = max_len.
    - Every decoder projection is zero, so each layer is the identity.
    - NoiseEnc is zero, so a noise row is its learned position alone.
    - pos_emb is 3 I, so a row at position p carries 3 e_p.
    - tok_emb is zero, or 5 I with tok_onehot, so token t adds 5 e_t.
    - final_norm is 1 and w_head is I.
    The head row's logits are then rmsnorm(row) / tau, and the argmax map
    returns the row's position, or its token with tok_onehot."""
    w = make_weights(cfg)
    for name in ("wqkv", "wo", "w_up", "w_down", "ne_w1", "ne_b1", "ne_w2", "ne_b2"):
        w[name] = np.zeros_like(w[name])
    d = cfg.d_model
    w["pos_emb"] = 3.0 * np.eye(cfg.max_len, d)
    w["tok_emb"] = 5.0 * np.eye(cfg.vocab, d) if tok_onehot else np.zeros((cfg.vocab, d))
    w["w_head"] = np.eye(cfg.vocab, d)
    w["final_norm"] = np.ones(d)
    return w


PROBE = TINY.replace(n_layer=2, d_model=64, n_head=2, d_ff=128, vocab=64, max_len=64,
                     pos="learned", map="argmax")


def check_noise_slot_positions(model_cls=None, decoder_cls=None):
    """Alg. 1, h = [h_x; h_z]: the P pending tokens sit at c..c+P-1 and noise
    slot j at c+P+j. The probe model's argmax token is the head row's position.
    So a k-step returns c+P .. c+P+k-1, and an AR step returns c+P-1, the last
    pending row. The cached length then advances by P (App. C.1)."""
    model_cls = model_cls or oracle.OracleModel
    decoder_cls = decoder_cls or oracle.OracleDecoder
    cfg = PROBE
    m = model_cls(cfg, _probe_weights(cfg))
    dec = decoder_cls(m)
    prompts = [np.arange(1, 6), np.arange(1, 12), np.arange(1, 2)]   # lengths 5, 11, 1
    dec.prefill(prompts)
    c = np.array([4, 10, 0])
    P = 1
    for k in (3, 3, 2, 0, 4, 1):
        z = np.full((3, max(k, 1)), 0.5, np.float32)
        toks = dec.step(k, z)
        if k > 0:
            want = c[:, None] + P + np.arange(k)[None, :]
        else:
            want = (c + P - 1)[:, None]
        assert np.array_equal(toks, want), (k, toks, want)
        c = c + P
        P = max(k, 1)
        assert [dec.cached_len(b) for b in range(3)] == list(c)


def test_noise_slot_positions():
    check_noise_slot_positions()


def test_planted_noise_slot_position_off_by_one():
    class Bad(oracle.OracleModel):
        def noise_rows(self, z, pos):
            return super().noise_rows(z, np.asarray(pos) - 1)
    assert _fails(check_noise_slot_positions, Bad)


def test_planted_noise_slot_position_one_late():
    class Bad(oracle.OracleModel):
        def noise_rows(self, z, pos):
            return super().noise_rows(z, np.asarray(pos) + 1)
    assert _fails(check_noise_slot_positions, Bad)


def check_token_rows(model_cls=None):
    """Token rows are E[x] + P[pos] in the learned-position model (the tiny
    configuration). The learned-position table is indexed by the row's own
    position, and the embedding by the token id."""
    model_cls = model_cls or oracle.OracleModel
    cfg = PROBE
    w = _probe_weights(cfg, tok_onehot=True)
    m = model_cls(cfg, w)
    toks = np.array([7, 0, 63, 7])
    pos = np.array([0, 5, 9, 63])
    h = m.token_rows(toks, pos)
    want = np.zeros((4, cfg.d_model))
    for i, (t, p) in enumerate(zip(toks, pos)):
        want[i, t] += 5.0
        want[i, p] += 3.0
    np.testing.assert_array_equal(h, want)
    # through the decoder: the AR step's head row is the last pending token
    # at position c; the bigger component, 5 e_token, wins the argmax
    dec = oracle.OracleDecoder(m)
    dec.prefill([np.array([3, 9, 40])])
    assert dec.step(0, np.zeros((1, 1), np.float32))[0, 0] == 40


def test_token_rows():
    check_token_rows()


def test_planted_token_rows_position_off_by_one():
    class Bad(oracle.OracleModel):
        def token_rows(self, tokens, pos):
            return super().token_rows(tokens, np.minimum(np.asarray(pos) + 1, self.cfg.max_len - 1))
    assert _fails(check_token_rows, Bad)


# ------------------------------------------------------------ head

def check_logits(model_cls=None):
    """Head(o) = RMSNorm_final(o) . W_head^T / tau (Table 4, Sec. 3.4).
    - tau = 2 halves the tau = 1 logits exactly, since halving is exact in
      binary floating point.
    - A row of +-1 has mean square 1. With W_head = [I; 2I] the logits are
      exactly g * o / sqrt(1 + eps) and twice that, because the norm comes
      before the head.
    - Scaling the row by any c > 0 leaves the logits unchanged, up to eps."""
    model_cls = model_cls or oracle.OracleModel
    d = 32
    cfg = TINY.replace(d_model=d, n_head=2, d_ff=64, vocab=2 * d, max_len=8, rms_eps=1e-6)
    w = make_weights(cfg)
    rng = np.random.default_rng(5)
    g = 1.0 + 0.5 * rng.random(d)
    w["final_norm"] = g
    w["w_head"] = np.concatenate([np.eye(d), 2.0 * np.eye(d)], 0)
    o = np.where(rng.random((3, d)) < 0.5, -1.0, 1.0)
    m1 = model_cls(cfg, w)
    m2 = model_cls(cfg.replace(tau=2.0), w)
    l1 = m1.logits(o)
    np.testing.assert_array_equal(m2.logits(o), l1 / 2.0)
    base = g * o / np.sqrt(1.0 + cfg.rms_eps)
    np.testing.assert_allclose(l1, np.concatenate([base, 2.0 * base], 1), rtol=1e-15, atol=0)
    np.testing.assert_allclose(m1.logits(7.5 * o), l1, rtol=1e-6)
    # a general row: the logits of c o equal those of o up to eps's share
    x = rng.normal(size=(2, d))
    np.testing.assert_allclose(m1.logits(100.0 * x), m1.logits(x), rtol=1e-5)


def test_logits_closed_forms():
    check_logits()


def test_planted_logits_tau_multiplied():
    class Bad(oracle.OracleModel):
        def logits(self, h_rows):
            o = ops.rmsnorm(h_rows, self.w["final_norm"], self.cfg.rms_eps)
            return (o @ self.w["w_head"].T) * self.cfg.tau
    assert _fails(check_logits, Bad)


def test_planted_logits_no_final_norm():
    class Bad(oracle.OracleModel):
        def logits(self, h_rows):
            return (h_rows * self.w["final_norm"]) @ self.w["w_head"].T / self.cfg.tau
    assert _fails(check_logits, Bad)


def test_planted_logits_norm_after_head():
    class Bad(oracle.OracleModel):
        def logits(self, h_rows):
            lg = ops.rmsnorm(h_rows @ self.w["w_head"].T, 1.0, self.cfg.rms_eps)
            return lg / self.cfg.tau
    assert _fails(check_logits, Bad)


# ------------------------------------------------------------ noise rows

def check_noise_rows(model_cls=None):
    """Noise rows are NoiseEnc(s(z, tau)), plus the learned position in the
    tiny model (Table 4; Alg. 1 h_z = NoiseEnc(z)). With the pass-through
    encoder of check_noise_encoder they equal gelu(s(z) + s(tau)) + P[pos]."""
    model_cls = model_cls or oracle.OracleModel
    d = 32
    cfg = TINY.replace(d_model=d, n_head=2, d_ff=64, vocab=64, max_len=16, noise_hidden=4 * d,
                       tau=0.7)
    w = make_weights(cfg)
    h = cfg.ne_hidden
    w1 = np.zeros((h, d))
    w1[:d] = np.eye(d)
    w2 = np.zeros((d, h))
    w2[:, :d] = np.eye(d)
    w.update(ne_w1=w1, ne_b1=np.zeros(h), ne_w2=w2, ne_b2=np.zeros(d))
    w["pos_emb"] = np.eye(cfg.max_len, d) * 0.25
    m = model_cls(cfg, w)
    z = np.array([0.0, 0.3, 0.999], np.float32)
    pos = np.array([3, 4, 9])
    got = m.noise_rows(z, pos)
    zz = z.astype(np.float64)
    s = ops.sinusoid(zz, d, cfg.noise_scale) + ops.sinusoid(np.full(3, cfg.tau), d, cfg.noise_scale)
    want = ops.gelu_tanh(s) + w["pos_emb"][pos]
    np.testing.assert_allclose(got, want, rtol=0, atol=1e-14)
    # z = 0 at tau: the z half of the features is [1..1 | 0..0]
    s0 = ops.sinusoid(np.zeros(1), d, cfg.noise_scale)
    np.testing.assert_array_equal(s0[0], np.r_[np.ones(d // 2), np.zeros(d // 2)])


def test_noise_rows_closed_form():
    check_noise_rows()


def test_planted_noise_rows_tau_dropped():
    class Bad(oracle.OracleModel):
        def noise_rows(self, z, pos):
            cfg = self.cfg
            feat = ops.sinusoid(np.asarray(z, np.float64), cfg.d_model, cfg.noise_scale)
            h = ops.noise_encoder(feat, self.w["ne_w1"], self.w["ne_b1"], self.w["ne_w2"], self.w["ne_b2"])
            return h + self.w["pos_emb"][np.asarray(pos)]
    assert _fails(check_noise_rows, Bad)
