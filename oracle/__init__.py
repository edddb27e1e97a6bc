"""CPU oracle for the K-Forcing joint next-k-token decode step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s ``cpu_baseline`` leg and ``--impl reference`` arm may import
or run anything in this package; the product path (the CUDA library and
its Python binding) never does, and fails loudly when the CUDA extension is
missing instead of falling back here.  It shares no code with the CUDA path:
the only module both sides use is ``synth`` (seeded inputs, no arithmetic of
the method).

Contents
  ops.py    primitive operations: RMSNorm, GELU, RoPE, causal attention,
            sinusoidal noise features, NoiseEnc, the inverse-CDF and argmax
            noise -> token maps, and the closed-form map G* (App. B).
  model.py  the push-forward causal Transformer (Sec. 3.3, Table 4) and the
            KV-cached decode of Alg. 1 (App. C.1), plus cache-free
            definitions (whole-sequence forward, textbook AR sampling).
  train_attention.py  the SingleForward / DoubleForward training masks
            (App. C.2) and dense masked attention over them.

Pins (``tests/test_oracle_*.py``, run with ``-m "not gpu"``) tie each part
to something other than itself: the worked example of App. B, a chi-square
test of the inverse-CDF map against the softmax, closed forms of the
primitives, degenerate weights whose layer output has a closed form,
cache-free recomputation, causal invariance, k-prefix invariance and the
textbook AR sampler.

Parity unpinned: the values a *trained* push-forward model would produce
(no checkpoint exists here), and the readings marked "reading:" in ops.py
(noise-encoder widths and feature scale, GELU form, eps, no biases in the
backbone), which the paper leaves open.
"""
from .ops import (apply_rope, argmax_token, causal_attention, gelu_tanh,  # noqa: F401
                  gstar, icdf_from_weights, icdf_token, noise_encoder,
                  noise_features, rmsnorm, rope_angles, sinusoid)
from .model import (OracleDecoder, OracleModel, ar_sample,  # noqa: F401
                    full_forward_logits, token_map)
