"""The measurement arithmetic of bench.py (algorithmic bytes and flops of a
decode call, from which every roofline fraction is computed) against the
ceilings derived independently from the model shapes (12·L·d² weights,
the LM head V·d, NoiseEnc 8d², KV 2·L·d per token; 2 flops per weight per
row, 4·L·d per visible key).

The byte counts here add the K/V writes of the k noise rows, which the
decode step performs (all P + k rows are appended, Alg. 1) and which the
closed-form ceiling omits: B·k·2·L·d·2 B.
"""
import numpy as np
import pytest

import bench
from synth import LM1B, LM1B_MTP, OWT


def _kv_token(cfg):
    return 2 * cfg.n_layer * cfg.d_model * 2


@pytest.mark.parametrize("cfg,B,P,k,ctx,mb,gflop", [
    (LM1B, 64, 1, 0, 80, 408, 14),     # AR step
    (LM1B, 64, 4, 4, 80, 424, 103),    # k = 4 steady state
    (OWT, 256, 4, 4, 768, 7542, 495),
    (OWT, 1, 4, 4, 768, 285, 1.9),
])
def test_step_costs_match_closed_form(cfg, B, P, k, ctx, mb, gflop):
    byt, fl = bench.step_bytes_flops(cfg, B, P, k, np.full(B, ctx))
    noise_kv = B * k * _kv_token(cfg)
    assert abs((byt - noise_kv) / 1e6 - mb) / mb < 0.01, (byt / 1e6, mb)
    assert abs(fl / 1e9 - gflop) / gflop < 0.03, (fl / 1e9, gflop)


def test_kind_costs_add_up_to_the_step():
    """Per-launch costs of the dense kinds times the layer count equal the
    step's weight bytes and projection flops; activations are not counted
    (the method does not need them in HBM)."""
    cfg, B, P, k = LM1B, 64, 4, 4
    ctx = np.full(B, 80)
    c = bench.kind_costs(cfg, B, P, k, ctx)
    d, F, L = cfg.d_model, cfg.d_ff, cfg.n_layer
    R = B * (P + k)
    w_layer = (4 * d * d + 2 * d * F) * 2
    wb = sum(c[n]["bytes"] for n in ("gemm_qkv", "gemm_o", "gemm_up", "gemm_down"))
    assert wb == w_layer
    # attention: the K and V of every key each sequence's rows see, per layer
    assert c["attention"]["bytes"] == B * (80 + P + k) * 2 * d * 2
    # the LM head reads its weights once per call
    assert c["gemm_head"]["bytes"] == cfg.vocab * d * 2
    fl = sum(c[n]["flops"] for n in ("gemm_qkv", "gemm_o", "gemm_up", "gemm_down"))
    assert fl == 2.0 * R * (4 * d * d + 2 * d * F)
    _, step_fl = bench.step_bytes_flops(cfg, B, P, k, ctx)
    attn = L * c["attention"]["flops"]
    head = c["gemm_head"]["flops"]
    noise = 2.0 * B * k * cfg.ne_hidden * 2 * d
    assert abs(L * fl + attn + head + noise - step_fl) / step_fl < 1e-12


def test_mtp_head_bytes_read_k_matrices():
    """The standard-MTP variant reads k untied head matrices once per call."""
    cfg = LM1B_MTP
    k = cfg.mtp_k
    c = bench.kind_costs(cfg, 64, k, k, np.full(64, 80))
    assert c["gemm_head"]["bytes"] >= k * cfg.vocab * cfg.d_model * 2
