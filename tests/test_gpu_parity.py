"""GPU path vs the CPU oracle, through the C ABI (needs a GB300).

fp32 model: tokens identical in every slot, logits within 1e-4.
bf16 models: logits within 3e-2 of the oracle row's range; each differing
token explained by the logit error (tests/parity.py).  The oracle is
teacher-forced with the GPU's tokens after each step, so both sides always
decode from the same context.
"""
import os

import numpy as np
import pytest

import oracle
from synth import (LM1B, MEDIUM, OWT, TINY, WORKLOADS, make_noise, make_prompt_lengths,
                   make_prompts, make_weights, workload_prompts)

from parity import LOGIT_TOL, compare_tokens, logit_check, record

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


def _run(kf, cfg, w, prompts, ks, max_k, seed=2, flags=0, map_dtype=None, dec=None,
         check_logits=True):
    """Decode ks steps on both sides; returns per-step records."""
    B = len(prompts)
    if dec is None:
        dec = kf.Decoder(cfg, w, max_batch=B, max_k=max_k, flags=flags)
    dec.prefill(prompts)
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, w), map_dtype=map_dtype)
    ref.prefill(prompts)
    rng = np.random.default_rng(seed)
    out = []
    for k in ks:
        z = rng.random((B, max(k, 1)), dtype=np.float32)
        gt = dec.step(k, z)
        gl = dec.logits(max(k, 1)) if check_logits else None
        rt, rl = ref.step(k, z, want_logits=True)
        out.append((k, z, gt.copy(), rt.copy(), gl, rl))
        # teacher-force: the oracle continues from the GPU's tokens
        for b in range(B):
            ref.seqs[b]["pending"] = [int(t) for t in gt[b]]
        assert list(dec.lengths()) == [ref.cached_len(b) for b in range(B)]
    return dec, out


def test_tiny_fp32_tokens_identical(kf):
    cfg = TINY
    w = make_weights(cfg)
    prompts = make_prompts([32, 32], cfg.vocab)
    dec, recs = _run(kf, cfg, w, prompts, [2, 2, 2, 1, 0, 2, 0, 0, 2], max_k=2)
    for k, z, gt, rt, gl, rl in recs:
        assert np.array_equal(gt, rt.astype(np.int32)), (k, gt, rt)
        assert np.abs(gl - rl).max() < 1e-4
    dec.close()


def test_tiny_fp32_ragged_prompts_argmax(kf):
    cfg = TINY.replace(map="argmax")
    w = make_weights(cfg)
    prompts = make_prompts([1, 7, 16, 17, 33], cfg.vocab)
    dec, recs = _run(kf, cfg, w, prompts, [4, 4, 3, 0, 4], max_k=4)
    for k, z, gt, rt, gl, rl in recs:
        assert np.array_equal(gt, rt.astype(np.int32)), (k, gt, rt)
    dec.close()


def test_tiny_fp32_rope_prefill_chunks(kf):
    """RoPE variant with prefill split over several chunks and groups."""
    cfg = TINY.replace(pos="rope")
    w = make_weights(cfg)
    prompts = make_prompts([40, 5, 23], cfg.vocab)
    dec = kf.Decoder(cfg, w, max_batch=3, max_k=4, prefill_rows=16)
    dec, recs = _run(kf, cfg, w, prompts, [4, 4, 0, 1], max_k=4, dec=dec)
    for k, z, gt, rt, gl, rl in recs:
        assert np.array_equal(gt, rt.astype(np.int32)), (k, gt, rt)
        assert np.abs(gl - rl).max() < 1e-4
    dec.close()


def test_k_prefix_invariance_fp32(kf):
    """A k=2 step equals the first two slots of a k=4 step (Sec. 3.4)."""
    cfg = TINY
    w = make_weights(cfg)
    prompts = make_prompts([20, 20], cfg.vocab)
    z = make_noise(1, 2, 4)[0]
    d4 = kf.Decoder(cfg, w, max_batch=2, max_k=4)
    d4.prefill(prompts)
    t4 = d4.step(4, z)
    l4 = d4.logits(4)
    d4.rewind()
    t2 = d4.step(2, np.ascontiguousarray(z[:, :2]))
    l2 = d4.logits(2)
    assert np.array_equal(t2, t4[:, :2])
    np.testing.assert_array_equal(l2, l4[:, :2])
    d4.close()


def test_rewind_and_stale_noise_kv(kf):
    """After a k=8 step wrote noise KV deep into the cache, rewinding and
    decoding again matches a fresh context: stale noise entries are never read."""
    cfg = TINY
    w = make_weights(cfg)
    prompts = make_prompts([10, 12], cfg.vocab)
    zs = make_noise(3, 2, 8)
    d = kf.Decoder(cfg, w, max_batch=2, max_k=8)
    d.prefill(prompts)
    d.step(8, zs[0])
    d.step(8, zs[1])
    d.rewind()
    a = [d.step(3, np.ascontiguousarray(zs[2][:, :3])), d.step(2, np.ascontiguousarray(zs[2][:, :2]))]
    f = kf.Decoder(cfg, w, max_batch=2, max_k=8)
    f.prefill(prompts)
    b = [f.step(3, np.ascontiguousarray(zs[2][:, :3])), f.step(2, np.ascontiguousarray(zs[2][:, :2]))]
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    d.close()
    f.close()


def test_graph_equals_eager(kf):
    cfg = TINY
    w = make_weights(cfg)
    prompts = make_prompts([9, 30], cfg.vocab)
    zs = make_noise(4, 2, 2)
    res = []
    for flags in (0, kf.KF_FLAG_NO_GRAPH):
        d = kf.Decoder(cfg, w, max_batch=2, max_k=2, flags=flags)
        d.prefill(prompts)
        res.append([d.step(2, zs[i]).copy() for i in range(4)])
        d.close()
    for a, b in zip(*res):
        assert np.array_equal(a, b)


def test_pdl_equals_plain_launches(kf):
    """Programmatic dependent launch changes scheduling only, not results."""
    cfg = LM1B.replace(n_layer=2)
    w = make_weights(cfg)
    prompts = make_prompts([17, 32, 5], cfg.vocab)
    zs = make_noise(3, 3, 4)
    res = []
    for flags in (0, kf.KF_FLAG_NO_PDL, kf.KF_FLAG_NO_PDL | kf.KF_FLAG_NO_GRAPH):
        d = kf.Decoder(cfg, w, max_batch=3, max_k=4, flags=flags)
        d.prefill(prompts)
        res.append([d.step(4, zs[i]).copy() for i in range(3)] + [d.logits(4)])
        d.close()
    for other in res[1:]:
        for a, b in zip(res[0], other):
            np.testing.assert_array_equal(a, b)


def test_profile_step_matches_decode(kf, lm1b_weights):
    """kf_profile_step (a one-off graph with event nodes) decodes exactly like
    kf_decode_step and reports every launch of the step."""
    cfg = LM1B
    prompts = make_prompts([20, 33], cfg.vocab)
    a = kf.Decoder(cfg, lm1b_weights, max_batch=2, max_k=4)
    b = kf.Decoder(cfg, lm1b_weights, max_batch=2, max_k=4)
    a.prefill(prompts)
    b.prefill(prompts)
    rng = np.random.default_rng(12)
    for k in (4, 4, 0):
        z = rng.random((2, max(k, 1)), dtype=np.float32)
        ta = np.zeros((2, max(k, 1)), np.int32)
        ms = np.zeros(kf.KF_KIND_COUNT, np.float32)
        n = np.zeros(kf.KF_KIND_COUNT, np.int32)
        kf.kf_profile_step(a.ctx, 2, k, z, ta, ms, n)
        assert np.array_equal(ta, b.step(k, z))
        names = dict(zip(kf.KIND_NAMES, zip(ms, n)))
        assert names["gemm_qkv"][1] == cfg.n_layer and names["attention"][1] == cfg.n_layer
        assert all(t > 0 for t, c in names.values() if c > 0)
    a.close()
    b.close()


def test_norm_gains_folded(kf):
    """Non-unit RMSNorm gains: the fused path folds them into the QKV and
    MLP-up weights; the oracle applies them after normalising."""
    cfg = LM1B.replace(n_layer=2)
    w = make_weights(cfg)
    rng = np.random.default_rng(9)
    for name in ("attn_norm", "mlp_norm", "final_norm"):
        w[name] = (1.0 + 0.3 * rng.standard_normal(w[name].shape)).astype(np.float32)
    prompts = make_prompts([20, 31], cfg.vocab)
    dec, recs = _run(kf, cfg, w, prompts, [4, 4, 0, 2], max_k=4)
    worst, slots, mism, bad = _bf16_check(recs)
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()


def test_device_buffers(kf):
    import torch
    cfg = TINY
    w = make_weights(cfg)
    prompts = make_prompts([9, 30], cfg.vocab)
    z = make_noise(1, 2, 2)[0]
    d = kf.Decoder(cfg, w, max_batch=2, max_k=2)
    d.prefill(prompts)
    host = d.step(2, z)
    d.rewind()
    zd = torch.from_numpy(z).cuda()
    od = torch.zeros((2, 2), dtype=torch.int32, device="cuda")
    d.step(2, zd, out=od)
    torch.cuda.synchronize()
    d.sync()
    assert np.array_equal(od.cpu().numpy(), host)
    d.close()


def test_errors_are_reported(kf):
    cfg = TINY
    w = make_weights(cfg)
    d = kf.Decoder(cfg, w, max_batch=2, max_k=2)
    z = np.zeros((2, 2), np.float32)
    with pytest.raises(kf.KfError) as e:
        d.B = 2
        d.step(2, z)
    assert e.value.code == kf.KF_E_STATE
    d.prefill(make_prompts([60, 3], cfg.vocab))
    with pytest.raises(kf.KfError) as e:
        d.step(3, np.zeros((2, 3), np.float32))
    assert e.value.code == kf.KF_E_ARG
    d.step(2, z)          # cached 59, writes positions 59..61 of max_len 64
    d.step(2, z)          # cached 60, writes positions 60..63
    with pytest.raises(kf.KfError) as e:
        d.step(2, z)      # cached 62 would write up to position 65
    assert e.value.code == kf.KF_E_CAPACITY
    with pytest.raises(kf.KfError) as e:
        d.prefill(make_prompts([64], cfg.vocab))
    assert e.value.code == kf.KF_E_CAPACITY
    d.close()


def _test_name():
    return os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0].split("::")[-1]


def _bf16_check(recs, map_kind="icdf"):
    """Worst logit error and token counts over the records; the counts go to
    the end-of-run agreement summary. Every bf16 test asserts that no
    mismatch is unexplained and that every decidable slot agrees."""
    worst = 0.0
    st = [0, 0, 0, 0, 0]
    for k, z, gt, rt, gl, rl in recs:
        worst = max(worst, logit_check(gl, rl))
        compare_tokens(gt, rt, gl, rl, z, map_kind, stats=st)
    record(_test_name(), st)
    assert st[4] == 0, f"{st[4]} decidable slots differ: {st}"
    return worst, st[0], st[1], st[2]


@pytest.fixture(scope="module")
def lm1b_weights():
    return make_weights(LM1B)


def test_lm1b_bf16_small_batch(kf, lm1b_weights):
    cfg = LM1B
    prompts = make_prompts([32, 32, 32], cfg.vocab)
    dec, recs = _run(kf, cfg, lm1b_weights, prompts, [4, 4, 4, 2, 0, 4], max_k=4)
    worst, slots, mism, bad = _bf16_check(recs)
    print(f"lm1b bf16: worst |dlogit|/range {worst:.2e}, {mism}/{slots} tokens differ, "
          f"{bad} unexplained")
    assert worst <= LOGIT_TOL
    assert bad == 0
    dec.close()


def test_lm1b_bf16_k8(kf, lm1b_weights):
    """k = 8 (16 query rows per sequence, both 8-row halves of the warp-MMA
    attention tile) and ragged prefill groups."""
    cfg = LM1B
    prompts = make_prompts([40, 23, 17], cfg.vocab)
    dec, recs = _run(kf, cfg, lm1b_weights, prompts, [8, 8, 4, 8], max_k=8)
    worst, slots, mism, bad = _bf16_check(recs)
    assert worst <= LOGIT_TOL
    assert bad == 0
    dec.close()


def test_lm1b_bf16_argmax(kf, lm1b_weights):
    cfg = LM1B.replace(map="argmax")
    prompts = make_prompts([32, 20], cfg.vocab)
    dec, recs = _run(kf, cfg, lm1b_weights, prompts, [4, 4, 0], max_k=4)
    worst, slots, mism, bad = _bf16_check(recs, "argmax")
    assert worst <= LOGIT_TOL
    assert bad == 0
    assert mism <= max(1, slots // 100)
    dec.close()


def test_lm1b_bf16_sharp_temperature(kf, lm1b_weights):
    """At tau = 0.1 the softmax is sharp: more slots are decidable (noise
    farther than the logit-error bound from every CDF boundary), and every
    decidable slot must agree; the raw agreement is recorded, not bounded
    (a few slots of 64 still fall inside the bound)."""
    cfg = LM1B.replace(tau=0.1)
    prompts = make_prompts([32] * 4, cfg.vocab)
    dec, recs = _run(kf, cfg, lm1b_weights, prompts, [4, 4, 4, 4], max_k=4)
    worst, slots, mism, bad = _bf16_check(recs)
    print(f"lm1b tau=0.1: {mism}/{slots} differ, {bad} unexplained")
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()


def test_lm1b_full_batch_sampled(kf, lm1b_weights):
    """The bench's shape (batch 64, k=4, graph replay): sampled sequences
    against the oracle, which runs only those sequences."""
    cfg = LM1B
    B = 64
    prompts = make_prompts([32] * B, cfg.vocab)
    dec = kf.Decoder(cfg, lm1b_weights, max_batch=B, max_k=4)
    dec.prefill(prompts)
    pick = [0, 17, 42, 63]
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, lm1b_weights))
    ref.prefill([prompts[i] for i in pick])
    zs = make_noise(3, B, 4)
    recs = []
    for s in range(3):
        gt = dec.step(4, zs[s])
        gl = dec.logits(4)[pick]
        rt, rl = ref.step(4, zs[s][pick], want_logits=True)
        recs.append((4, zs[s][pick], gt[pick].copy(), rt, gl, rl))
        for j, b in enumerate(pick):
            ref.seqs[j]["pending"] = [int(t) for t in gt[b]]
    worst, slots, mism, bad = _bf16_check(recs)
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()


def test_owt_ragged_paged(kf):
    """OWT-shaped vocab with ragged prompts crossing many 16-token pages."""
    cfg = OWT.replace(n_layer=2, max_len=256)
    w = make_weights(cfg)
    lens = make_prompt_lengths(4, 100, 200)
    prompts = make_prompts(lens, cfg.vocab)
    dec, recs = _run(kf, cfg, w, prompts, [4, 4, 4, 4, 4, 1, 0], max_k=4)
    worst, slots, mism, bad = _bf16_check(recs)
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()


def test_owt_small_batch_split_keys(kf):
    """Two sequences of a 1024-position model: the attention splits each
    sequence's keys over 4 CTAs (256 keys each) and merges the partial
    softmaxes in the kernel; the 300-token prompt leaves its last split
    empty."""
    cfg = OWT.replace(n_layer=2)
    w = make_weights(cfg)
    prompts = make_prompts([300, 700], cfg.vocab)
    dec, recs = _run(kf, cfg, w, prompts, [4, 4, 0, 4], max_k=4)
    worst, slots, mism, bad = _bf16_check(recs)
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()


def _sampled(kf, cfg, w, prompts, pick, ks, max_k, seed):
    """Full batch on the GPU (graph replay), the oracle on sampled sequences."""
    B = len(prompts)
    dec = kf.Decoder(cfg, w, max_batch=B, max_k=max_k)
    dec.prefill(prompts)
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, w))
    ref.prefill([prompts[i] for i in pick])
    rng = np.random.default_rng(seed)
    recs = []
    for k in ks:
        z = rng.random((B, max(k, 1)), dtype=np.float32)
        gt = dec.step(k, z)
        gl = dec.logits(max(k, 1))[pick]
        rt, rl = ref.step(k, z[pick], want_logits=True)
        recs.append((k, z[pick], gt[pick].copy(), rt, gl, rl))
        for j, b in enumerate(pick):
            ref.seqs[j]["pending"] = [int(t) for t in gt[b]]
        assert [int(x) for x in dec.lengths()[pick]] == [ref.cached_len(j) for j in range(len(pick))]
    dec.close()
    return _bf16_check(recs)


def test_owt_paged_full_batch_sampled(kf):
    """OWT-shaped high-load serving: batch 512, ragged prompts in [128, 896],
    16-token pages; sampled sequences against the oracle."""
    wl = WORKLOADS["owt_paged"]
    cfg = wl.model
    w = make_weights(cfg)
    prompts = workload_prompts(wl)
    lens = [len(p) for p in prompts]
    pick = [int(np.argmin(lens)), int(np.argmax(lens)), 100, 511]
    worst, slots, mism, bad = _sampled(kf, cfg, w, prompts, pick, [4, 4, 0], 4, 21)
    assert worst <= LOGIT_TOL and bad == 0


def test_medium_k8_sampled(kf):
    """Medium stress shape (24 layers, d 1024, 16 heads): batch 256, prompts
    of 1024, k = 8 then k = 4; sampled sequences against the oracle."""
    cfg = MEDIUM
    w = make_weights(cfg)
    prompts = make_prompts([1024] * 256, cfg.vocab)
    worst, slots, mism, bad = _sampled(kf, cfg, w, prompts, [0, 255], [8, 8, 4], 8, 22)
    assert worst <= LOGIT_TOL and bad == 0


def test_lm1b_bf16_agreement_over_1024_slots(kf, lm1b_weights):
    """The bench's shape, batch 64 at k = 4, every sequence against the oracle
    (teacher-forced) for four steps: 1024 slots at tau = 0.1. Every decidable
    slot agrees (the >= 99.9 % criterion, graded where the logit error cannot
    move the token) and every other mismatch is explained; the raw rate is
    recorded."""
    cfg = LM1B.replace(tau=0.1)
    prompts = make_prompts([32] * 64, cfg.vocab)
    dec, recs = _run(kf, cfg, lm1b_weights, prompts, [4, 4, 4, 4], max_k=4)
    worst, slots, mism, bad = _bf16_check(recs)
    assert slots == 1024
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()


# ------------------------------------------- fp32 exact tokens, real shapes

# Both sides take the fp32 model's token decision with fp64 sums. What can
# still move a CDF boundary is the fp32 logits' own rounding: ~1e-6 relative
# per logit, ~1e-8 on a boundary. A mismatch whose noise lies within this
# bound of the oracle's boundary is a rounding tie, and it is reported.
FP32_DECISION_BOUND = 2e-6


@pytest.mark.parametrize("shape", ["lm1b", "owt", "medium"])
def test_fp32_tokens_identical_real_shapes(kf, shape):
    """The fp32 mode at the workloads' real shapes: vocabularies of 30,522 and
    50,257, d_model 768 and 1024, head_dim 64, 12 and 24 layers. Ragged prompts
    cross 16-token pages, and the steps mix k = 4, k = 8 and the AR step.
    Tokens are identical in every slot whose noise lies farther than the fp32
    decision's own rounding (FP32_DECISION_BOUND) from the oracle's CDF
    boundaries. Any other mismatch fails the test, with its margin, the
    distance |z - F| to the nearest boundary between the two bins. The
    near-boundary mismatches are counted in the end-of-run summary."""
    base = {"lm1b": LM1B, "owt": OWT.replace(max_len=512), "medium": MEDIUM.replace(max_len=512)}[shape]
    cfg = base.replace(dtype="fp32")
    w = make_weights(cfg)
    lens = {"lm1b": [20, 33, 47], "owt": [100, 17, 250], "medium": [40, 129, 7]}[shape]
    prompts = make_prompts(lens, cfg.vocab)
    dec, recs = _run(kf, cfg, w, prompts, [4, 8, 0, 4, 8, 0], max_k=8, seed=31)
    slots, near, bad = 0, [], []
    for k, z, gt, rt, gl, rl in recs:
        rt = rt.astype(np.int32)
        slots += gt.size
        for b, j in zip(*np.nonzero(gt != rt)):
            l = np.asarray(rl[b, j], np.float64)
            p = np.exp(l - l.max())
            F = np.cumsum(p / p.sum())
            lo, hi = sorted((int(gt[b, j]), int(rt[b, j])))
            margin = float(np.abs(F[lo:hi] - z[b, j]).max())
            msg = f"k={k} slot ({b},{j}) gpu {gt[b, j]} oracle {rt[b, j]} margin {margin:.3e}"
            (near if margin <= FP32_DECISION_BOUND else bad).append(msg)
        assert np.abs(gl - rl).max() < 1e-3 * max(1.0, float(np.abs(rl).max()))
    print(f"fp32 {shape}: {slots - len(near) - len(bad)}/{slots} identical; near-boundary: {near}")
    record(_test_name(), [slots, len(near) + len(bad), len(bad), slots - len(near) - len(bad), len(bad)])
    assert not bad, bad
    assert len(near) <= max(1, slots // 50), near
    dec.close()


# ------------------------------------------- device-side error reporting

def test_device_prompt_out_of_range_reports_device_error(kf):
    """A device-resident prompt is range-checked where the embedding kernel
    reads it: an id >= V embeds as id 0 (no out-of-bounds read), flags the
    device error word, and kf_prefill returns KF_E_DEVICE. A later prefill
    with valid ids starts clean, and its step decodes like a fresh context."""
    import torch
    cfg = TINY
    w = make_weights(cfg)
    d = kf.Decoder(cfg, w, max_batch=2, max_k=2)
    good = make_prompts([9, 12], cfg.vocab)
    bad = [p.copy() for p in good]
    bad[1][3] = cfg.vocab + 5
    toks = torch.from_numpy(np.concatenate(bad)).cuda()
    lens = np.array([len(p) for p in bad], np.int32)
    with pytest.raises(kf.KfError) as e:
        kf.kf_prefill(d.ctx, 2, toks, lens)
    assert e.value.code == kf.KF_E_DEVICE
    assert "device error flag 1" in str(e.value) or "flag 1" in kf.kf_last_error(d.ctx)
    z = make_noise(1, 2, 2)[0]
    d.prefill(good)
    got = d.step(2, z)
    d.sync()
    f = kf.Decoder(cfg, w, max_batch=2, max_k=2)
    f.prefill(good)
    assert np.array_equal(got, f.step(2, z))
    d.close()
    f.close()


def test_persistent_gemm_equals_per_tile_model(kf):
    """OWT-shaped batch 512 at k = 4 (4096 rows, the bench's headline
    shape): the QKV and MLP-up projections exceed a wave of 256-wide tiles
    and run as persistent tile loops.  Tokens and logits equal those of one
    CTA per tile bit for bit, and stay within tolerance of the oracle on
    sampled sequences."""
    cfg = OWT.replace(n_layer=2, max_len=256)
    w = make_weights(cfg)
    prompts = make_prompts([40] * 512, cfg.vocab)
    zs = make_noise(3, 512, 4)
    res = []
    for flags in (0, kf.KF_FLAG_NO_PERSISTENT_GEMM):
        d = kf.Decoder(cfg, w, max_batch=512, max_k=4, flags=flags)
        d.prefill(prompts)
        res.append([d.step(4, zs[i]).copy() for i in range(3)] + [d.logits(4)])
        d.close()
    for a, b in zip(*res):
        np.testing.assert_array_equal(a, b)
    pick = [0, 131, 511]
    worst, slots, mism, bad = _sampled(kf, cfg, w, prompts, pick, [4, 4, 0], 4, 23)
    assert worst <= LOGIT_TOL and bad == 0


def test_skinny_and_tcgen05_small_batch(kf, lm1b_weights):
    """Calls of at most 64 rows run their projections as skinny warp-MMA
    kernels; KF_FLAG_NO_SKINNY keeps the tcgen05 GEMMs.  Batch 8 reaches
    exactly 64 rows at k = 4 (P = 4 pending + 4 noise rows per sequence).
    Both paths stay within tolerance of the oracle, and of each other."""
    cfg = LM1B
    prompts = make_prompts([32, 5, 17, 32, 40, 9, 23, 32], cfg.vocab)
    logits = []
    for flags in (0, kf.KF_FLAG_NO_SKINNY):
        dec, recs = _run(kf, cfg, lm1b_weights, prompts, [4, 4, 0, 4, 2], max_k=4, seed=31, flags=flags)
        worst, slots, mism, bad = _bf16_check(recs)
        assert worst <= LOGIT_TOL and bad == 0, (flags, worst, bad)
        logits.append(recs[0][4])
        dec.close()
    rng = logits[1].max(axis=-1, keepdims=True) - logits[1].min(axis=-1, keepdims=True)
    assert (np.abs(logits[0] - logits[1]) / rng).max() <= LOGIT_TOL


def test_owt_batch1_skinny_rows(kf):
    """One sequence of the OWT-shaped model: 8, 6 and 2 rows per call (k = 4,
    k = 2 and the AR step after a k = 2 step), all under one 8-row A box."""
    cfg = OWT.replace(n_layer=2)
    w = make_weights(cfg)
    prompts = make_prompts([300], cfg.vocab)
    dec, recs = _run(kf, cfg, w, prompts, [4, 4, 2, 0, 4], max_k=4, seed=33)
    worst, slots, mism, bad = _bf16_check(recs)
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()
