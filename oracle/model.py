"""The push-forward causal Transformer and its KV-cached k-token decode step.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).  Plain, slow,
per-sequence numpy; fp64 unless asked otherwise.

Model (Table 4 backbone, Sec. 3.3 fully causal PFLM, Fig. 2b):
  rows h: token rows E[x] (+ learned position), noise rows NoiseEnc(z)
  (+ learned position); L pre-norm decoder layers
  [RMSNorm -> QKV -> RoPE -> causal attention -> O + residual ->
   RMSNorm -> MLP(GELU) + residual]; final RMSNorm; untied LM head / tau.

Decode (Alg. 1, App. C.1): per sequence, P pending committed tokens at
positions c..c+P-1 and k noise slots at c+P..c+P+k-1; one forward pass over
those rows against the cache; keep the P context rows' KV, drop the noise
rows' KV; the k noise rows' logits go through the noise -> token map; the k
tokens become the next step's pending rows.  k = 0 is the AR teacher step:
one token per sequence from the last pending row's logits with noise z.
"""
from __future__ import annotations

import numpy as np

from . import ops


class OracleModel:
    """Forward pass of one sequence's rows against its KV cache."""

    def __init__(self, cfg, weights: dict, dtype=np.float64):
        self.cfg = cfg
        self.dtype = dtype
        self.w = {k: np.asarray(v, dtype) for k, v in weights.items()}
        self.H = cfg.n_head
        self.hd = cfg.d_model // cfg.n_head

    # -- input rows (Alg. 1: h_x = Embed(x), h_z = NoiseEnc(z), h = [h_x; h_z])
    def token_rows(self, tokens, pos) -> np.ndarray:
        h = self.w["tok_emb"][np.asarray(tokens, np.int64)]
        if self.cfg.pos == "learned":
            h = h + self.w["pos_emb"][np.asarray(pos, np.int64)]
        return h

    def noise_rows(self, z, pos) -> np.ndarray:
        """Fully causal: one row per noise value.  Standard MTP (cfg.mtp_k > 0,
        Sec. 3.3): the k values are one noise-conditioning token; reading: its
        features are the k values' sinusoidal features concatenated."""
        cfg = self.cfg
        z = np.asarray(z, np.float32).astype(self.dtype)
        feat = ops.noise_features(z, cfg.tau, cfg.d_model, cfg.noise_scale)
        if cfg.mtp_k:
            feat = feat.reshape(1, -1)
        h = ops.noise_encoder(feat, self.w["ne_w1"], self.w["ne_b1"],
                              self.w["ne_w2"], self.w["ne_b2"])
        if cfg.pos == "learned":
            h = h + self.w["pos_emb"][np.asarray(pos, np.int64)]
        return h

    # -- one decoder layer (Table 4), rows of a single sequence
    def layer(self, li: int, h, pos, cache_k, cache_v):
        """Returns (h_out, k_rows, v_rows).  cache_k/v hold positions
        0 .. pos[0]-1 as [c, H, hd]; the rows sit at positions ``pos``."""
        cfg, w, H, hd = self.cfg, self.w, self.H, self.hd
        d = cfg.d_model
        n = h.shape[0]
        a = ops.rmsnorm(h, w["attn_norm"][li], cfg.rms_eps)
        qkv = a @ w["wqkv"][li].T
        q = qkv[:, :d].reshape(n, H, hd)
        k = qkv[:, d:2 * d].reshape(n, H, hd)
        v = qkv[:, 2 * d:].reshape(n, H, hd)
        if cfg.pos == "rope":
            q = ops.apply_rope(q, pos, cfg.rope_theta)
            k = ops.apply_rope(k, pos, cfg.rope_theta)
        keys = np.concatenate([cache_k, k], axis=0)
        vals = np.concatenate([cache_v, v], axis=0)
        k_pos = np.arange(keys.shape[0])
        att = ops.causal_attention(q, keys, vals, np.asarray(pos), k_pos)
        h = h + att.reshape(n, d) @ w["wo"][li].T
        m = ops.rmsnorm(h, w["mlp_norm"][li], cfg.rms_eps)
        h = h + ops.gelu_tanh(m @ w["w_up"][li].T) @ w["w_down"][li].T
        return h, k, v

    def forward(self, h, pos, cache):
        """TF(h, C) of Alg. 1 for one sequence.  ``cache`` is a list of
        (K, V) per layer.  Returns (final hidden rows, per-layer new (K, V))."""
        new = []
        for li in range(self.cfg.n_layer):
            ck, cv = cache[li]
            h, k, v = self.layer(li, h, pos, ck, cv)
            new.append((k, v))
        return h, new

    def logits(self, h_rows) -> np.ndarray:
        """Head(o): final RMSNorm, untied LM head, divided by tau."""
        o = ops.rmsnorm(h_rows, self.w["final_norm"], self.cfg.rms_eps)
        return (o @ self.w["w_head"].T) / self.cfg.tau

    def logits_mtp(self, h_row) -> np.ndarray:
        """The k independent MTP heads on the noise token's final hidden
        state (Sec. 3.3): [k, V], head j = final RMSNorm then w_mtp[j], / tau."""
        o = ops.rmsnorm(np.asarray(h_row).reshape(1, -1), self.w["final_norm"], self.cfg.rms_eps)
        return np.stack([(o @ wj.T)[0] for wj in self.w["w_mtp"]]) / self.cfg.tau

    def empty_cache(self):
        z = np.zeros((0, self.H, self.hd), self.dtype)
        return [(z, z) for _ in range(self.cfg.n_layer)]


def token_map(cfg, logits_row, z, map_dtype):
    if cfg.map == "argmax":
        return ops.argmax_token(logits_row)
    return ops.icdf_token(logits_row, z, map_dtype)


class OracleDecoder:
    """KV-cached inference of Alg. 1 over a batch, one sequence at a time.

    ``map_dtype`` is the precision of the noise -> token decision. By default
    it is the precision in which the CUDA path takes it: fp32 for bf16
    models, whose logits carry bf16 rounding far above fp32's, and fp64 for
    fp32 models, so the decision adds no rounding of its own beyond the
    fp32 logits. A test may ask for another.
    """

    def __init__(self, model: OracleModel, map_dtype=None):
        self.m = model
        if map_dtype is None:
            map_dtype = np.float64 if model.cfg.dtype == "fp32" else np.float32
        self.map_dtype = map_dtype
        self.seqs = []

    def prefill(self, prompts):
        """Cache the KV of every prompt token but the last; the last becomes
        the one pending token (equivalent to Alg. 1's first step over the
        whole prompt plus noise, because attention is causal)."""
        self.seqs = []
        for p in prompts:
            p = [int(t) for t in p]
            assert len(p) >= 1
            cache = self.m.empty_cache()
            if len(p) > 1:
                pos = np.arange(len(p) - 1)
                h = self.m.token_rows(p[:-1], pos)
                _, new = self.m.forward(h, pos, cache)
                cache = [(k, v) for (k, v) in new]
            self.seqs.append({"committed": p[:-1], "pending": p[-1:],
                              "cache": cache})

    def admit(self, b: int, prompt, n_pending: int):
        """Replace sequence b by a new prompt at a step boundary, its last
        n_pending tokens pending (continuous batching, App. C.1: every
        sequence of the batch keeps the same stride).  With n_pending = 1
        this is prefill of that prompt alone."""
        p = [int(t) for t in prompt]
        assert 1 <= n_pending <= len(p)
        n = len(p) - n_pending
        cache = self.m.empty_cache()
        if n > 0:
            pos = np.arange(n)
            h = self.m.token_rows(p[:n], pos)
            _, new = self.m.forward(h, pos, cache)
            cache = [(k, v) for (k, v) in new]
        self.seqs[b] = {"committed": p[:n], "pending": p[n:], "cache": cache}

    def cached_len(self, b: int) -> int:
        return len(self.seqs[b]["committed"])

    def step(self, k: int, z: np.ndarray, want_logits: bool = False):
        """One decode step (Alg. 1 loop body).  z: [B, max(k, 1)] fp32.
        Returns tokens [B, max(k, 1)] (and logits [B, max(k, 1), V])."""
        cfg = self.m.cfg
        nb = len(self.seqs)
        nout = max(k, 1)
        toks = np.zeros((nb, nout), np.int64)
        lg_all = np.zeros((nb, nout, cfg.vocab), self.m.dtype) if want_logits else None
        for b, s in enumerate(self.seqs):
            c = len(s["committed"])
            P = len(s["pending"])
            pos_x = np.arange(c, c + P)
            h = self.m.token_rows(s["pending"], pos_x)
            mtp = cfg.mtp_k > 0 and k > 0
            if mtp:
                assert k == cfg.mtp_k
                pos_z = np.array([c + P])
                h = np.concatenate([h, self.m.noise_rows(z[b, :k], pos_z)], 0)
                pos = np.concatenate([pos_x, pos_z])
            elif k > 0:
                pos_z = np.arange(c + P, c + P + k)
                h = np.concatenate([h, self.m.noise_rows(z[b, :k], pos_z)], 0)
                pos = np.concatenate([pos_x, pos_z])
            else:
                pos = pos_x
            assert pos[-1] < cfg.max_len
            o, new = self.m.forward(h, pos, s["cache"])
            # C <- [C; C_x]: keep the P context rows' KV, discard the noise KV
            s["cache"] = [(np.concatenate([ck, nk[:P]]), np.concatenate([cv, nv[:P]]))
                          for (ck, cv), (nk, nv) in zip(s["cache"], new)]
            if mtp:
                lg = self.m.logits_mtp(o[P])
            else:
                head_rows = o[P:] if k > 0 else o[P - 1:P]
                lg = self.m.logits(head_rows)
            for j in range(nout):
                toks[b, j] = token_map(cfg, lg[j], z[b, j], self.map_dtype)
            if want_logits:
                lg_all[b] = lg
            s["committed"] = s["committed"] + list(s["pending"])
            s["pending"] = [int(t) for t in toks[b]]
        return (toks, lg_all) if want_logits else toks


# ------------------------------------------------ cache-free definitions

def full_forward_logits(model: OracleModel, tokens, z=None, k: int = 0):
    """Logits of one whole-sequence forward pass with no cache: rows are the
    token rows at positions 0..n-1 followed by k noise rows.  Returns the k
    noise rows' logits, or (k = 0) the last token row's logits."""
    n = len(tokens)
    pos = np.arange(n)
    h = model.token_rows(tokens, pos)
    if k > 0:
        pz = np.arange(n, n + k)
        h = np.concatenate([h, model.noise_rows(np.asarray(z)[:k], pz)], 0)
        pos = np.concatenate([pos, pz])
    o, _ = model.forward(h, pos, model.empty_cache())
    return model.logits(o[n:] if k > 0 else o[n - 1:n])


def ar_sample(model: OracleModel, prompt, zs, map_dtype=None):
    """Textbook AR sampling by full recomputation: each new token is
    F^{-1}(z_t) of the next-token softmax of the whole current sequence
    (Eq. 1 with k = 1)."""
    if map_dtype is None:
        map_dtype = np.float64 if model.cfg.dtype == "fp32" else np.float32
    seq = [int(t) for t in prompt]
    out = []
    for zt in zs:
        lg = full_forward_logits(model, seq)[0]
        t = token_map(model.cfg, lg, zt, map_dtype)
        out.append(t)
        seq.append(t)
    return out
