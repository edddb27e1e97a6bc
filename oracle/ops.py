"""Primitive operations of the push-forward causal Transformer, written plainly.

TEST INFRASTRUCTURE ONLY.  This is the CPU oracle: only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s ``cpu_baseline`` / reference
leg may import it.  It shares no code with the CUDA path.

Every function computes in the floating type of its inputs (fp64 unless a
caller passes fp32).  Readings of points the paper leaves open are marked
"reading:".
"""
from __future__ import annotations

import numpy as np


# ---------------------------------------------------------------- backbone

def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm, the backbone's pre-norm (Table 4): x / sqrt(mean(x^2) + eps) * g.

    reading: eps = 1e-6, gain initialised to 1.
    """
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def gelu_tanh(x: np.ndarray) -> np.ndarray:
    """GELU of the MLPs (Table 4 names GELU for the noise-encoder MLP).

    reading: the tanh form 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))
    for both the backbone MLP and the noise encoder.
    """
    x = np.asarray(x)
    c = x.dtype.type(np.sqrt(2.0 / np.pi))      # a constant of x's own type
    return 0.5 * x * (1.0 + np.tanh(c * (x + 0.044715 * x * x * x)))


def rope_angles(pos: np.ndarray, head_dim: int, theta: float,
                dtype=np.float64) -> np.ndarray:
    """Rotary angles (Table 4: RoPE with d_rot = 64 = head_dim).

    angle[p, i] = p * theta^(-2 i / head_dim), i = 0 .. head_dim/2 - 1.
    """
    half = head_dim // 2
    i = np.arange(half, dtype=np.float64)
    inv = theta ** (-2.0 * i / head_dim)
    return (np.asarray(pos, np.float64)[:, None] * inv[None, :]).astype(dtype)


def apply_rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotate pairs (i, i + head_dim/2) of x[n, H, head_dim] by rope_angles.

    reading: the rotate-half pairing, theta = 1e4.
    """
    hd = x.shape[-1]
    half = hd // 2
    ang = rope_angles(pos, hd, theta, x.dtype)[:, None, :]   # [n, 1, half]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                     q_pos: np.ndarray, k_pos: np.ndarray) -> np.ndarray:
    """Softmax attention of q[n, H, hd] over keys k, v [m, H, hd].

    A query at position p sees exactly the keys at positions <= p: this is
    the fully causal layout of Sec. 3.3, where noise slot j attends to the
    context and to noise slots 1..j (and Alg. 1 reuses it with a KV cache).
    Scale 1/sqrt(hd).
    """
    hd = q.shape[-1]
    scores = np.einsum("nhd,mhd->hnm", q, k) / q.dtype.type(np.sqrt(hd))
    mask = np.asarray(k_pos)[None, :] > np.asarray(q_pos)[:, None]    # [n, m]
    scores = np.where(mask[None, :, :], -np.inf, scores)
    scores = scores - scores.max(axis=-1, keepdims=True)
    p = np.exp(scores)
    p = p / p.sum(axis=-1, keepdims=True)
    return np.einsum("hnm,mhd->nhd", p, v)


# ---------------------------------------------------------- noise encoder

def sinusoid(u: np.ndarray, d: int, scale: float) -> np.ndarray:
    """Sinusoidal encoding of scalars u (Table 4: noise & temperature
    embedding is a sinusoidal positional encoding of width d).

    reading: argument scale * u, frequencies exp(-ln(1e4) i / (d/2)) for
    i = 0 .. d/2 - 1, output [cos | sin].
    """
    u = np.asarray(u)
    half = d // 2
    i = np.arange(half, dtype=np.float64)
    freq = np.exp(-np.log(1e4) * i / half).astype(u.dtype)
    arg = (scale * u)[:, None] * freq[None, :]
    return np.concatenate([np.cos(arg), np.sin(arg)], axis=-1)


def noise_features(z: np.ndarray, tau: float, d: int,
                   scale: float) -> np.ndarray:
    """Input features of NoiseEnc for noise values z at temperature tau.

    reading: the temperature's encoding is added to the noise's encoding
    (Sec. 3.4 conditions the noise encoder on tau; the combination is not
    stated).
    """
    z = np.asarray(z)
    t = np.full_like(z, tau)
    return sinusoid(z, d, scale) + sinusoid(t, d, scale)


def noise_encoder(feat: np.ndarray, w1, b1, w2, b2) -> np.ndarray:
    """Two-layer MLP with GELU on the sinusoidal features (Table 4; Alg. 1
    h_z = NoiseEnc(z)).  reading: hidden width 4d, with biases."""
    return gelu_tanh(feat @ w1.T + b1) @ w2.T + b2


# ------------------------------------------------- noise -> token maps

def icdf_from_weights(w: np.ndarray, z) -> int:
    """Inverse-CDF map on unnormalised, nonnegative weights w over the vocab
    in id order (App. B, Eq. cdf / icdf): the least index v whose prefix sum
    exceeds z * S, S = sum of w.

    reading: the strict '>' of App. B (the main text's Eq. 1 writes '>='),
    giving half-open bins [F(v-1), F(v)) as in the worked example where
    z1 in [0, 1/3) gives A.  Sums are taken sequentially in id order in the
    dtype of w.  If rounding leaves no prefix above z * S (z near 1), the
    answer is the largest v with w[v] > 0.
    """
    w = np.asarray(w)
    prefix = np.cumsum(w, dtype=w.dtype)
    s = prefix[-1]
    t = w.dtype.type(z) * s
    hit = prefix > t
    if hit.any():
        return int(np.argmax(hit))
    nz = np.nonzero(w > 0)[0]
    return int(nz[-1])


def icdf_token(logits: np.ndarray, z, dtype=np.float32) -> int:
    """F^{-1}(z) of the softmax of logits (Eq. 1 with App. B's convention).

    The decision is taken in ``dtype``: logits are cast, the maximum m is
    subtracted, w = exp(l - m) and the prefix sums are formed in that type.
    """
    l = np.asarray(logits).astype(dtype)
    w = np.exp(l - l.max())
    return icdf_from_weights(w, dtype(z))


def argmax_token(logits: np.ndarray) -> int:
    """Greedy map of the learned PFLM's shared head (Sec. 3.2; Alg. 1
    applies arg max to Head(o_{-k:})).  Ties go to the lowest id."""
    return int(np.argmax(np.asarray(logits)))


def gstar(next_logits, context: list, z, dtype=np.float64) -> list:
    """Closed-form push-forward map G* (App. B, Eq. sequential-icdf):
    k sequential inverse-CDF draws, the j-th one from the AR distribution
    conditioned on the context and the j-1 tokens already drawn.

    ``next_logits(tokens) -> logits`` is the AR oracle.
    """
    out = []
    for zj in z:
        out.append(icdf_token(next_logits(list(context) + out), zj, dtype))
    return out
