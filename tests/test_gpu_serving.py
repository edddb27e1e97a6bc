"""The serving entry points around the decode step, through the C ABI (needs
a GB300): the k-pass teacher G* (kf_teacher_step) and continuous batching
(kf_admit: replace a sequence at a step boundary, pages recycled).

fp32 model: tokens identical to the oracle.  bf16: logits within LOGIT_TOL
and every differing token explained (tests/parity.py).
"""
import numpy as np
import pytest

import oracle
from synth import LM1B, TINY, make_prompts, make_weights

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


def _ar_steps(dec, z):
    """k separate AR calls (kf_decode_step with k = 0) on the columns of z."""
    return np.stack([dec.step(0, np.ascontiguousarray(z[:, j:j + 1]))[:, 0] for j in range(z.shape[1])], 1)


def test_teacher_step_equals_ar_calls_and_oracle_fp32(kf):
    cfg = TINY
    w = make_weights(cfg)
    prompts = make_prompts([9, 14, 5], cfg.vocab)
    rng = np.random.default_rng(31)
    a = kf.Decoder(cfg, w, max_batch=3, max_k=4)
    b = kf.Decoder(cfg, w, max_batch=3, max_k=4)
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, w))
    for d in (a, b):
        d.prefill(prompts)
    ref.prefill(prompts)
    # a joint step first, so the teacher starts from P = 4 pending tokens
    z0 = rng.random((3, 4), dtype=np.float32)
    t0 = a.step(4, z0)
    assert np.array_equal(t0, b.step(4, z0))
    assert np.array_equal(t0, ref.step(4, z0).astype(np.int32))
    for k in (3, 4, 1):
        z = rng.random((3, k), dtype=np.float32)
        got = a.teacher_step(k, z)
        want = _ar_steps(b, z)
        assert np.array_equal(got, want), (k, got, want)
        ref_t = np.stack([ref.step(0, z[:, j:j + 1])[:, 0] for j in range(k)], 1)
        assert np.array_equal(got, ref_t.astype(np.int32)), (k, got, ref_t)
        assert list(a.lengths()) == list(b.lengths()) == [ref.cached_len(i) for i in range(3)]
    # the joint step continues from the teacher's state (one pending token)
    z = rng.random((3, 2), dtype=np.float32)
    assert np.array_equal(a.step(2, z), ref.step(2, z).astype(np.int32))
    a.close()
    b.close()


def test_teacher_step_bf16_graph_and_host_buffers(kf):
    import torch
    cfg = LM1B
    w = make_weights(cfg)
    prompts = make_prompts([32] * 8, cfg.vocab)
    rng = np.random.default_rng(32)
    a = kf.Decoder(cfg, w, max_batch=8, max_k=4)
    b = kf.Decoder(cfg, w, max_batch=8, max_k=4, flags=kf.KF_FLAG_NO_GRAPH)
    for d in (a, b):
        d.prefill(prompts)
    for k in (4, 4, 2):
        z = rng.random((8, k), dtype=np.float32)
        got = a.teacher_step(k, z)
        want = _ar_steps(b, z)
        assert np.array_equal(got, want), k
    # device buffers
    z = torch.rand((8, 3), device="cuda")
    out = torch.zeros((8, 3), dtype=torch.int32, device="cuda")
    kf.kf_teacher_step(a.ctx, 8, 3, z, out)
    want = _ar_steps(b, z.cpu().numpy())
    assert np.array_equal(out.cpu().numpy(), want)
    a.close()
    b.close()


def test_admit_matches_oracle_fp32(kf):
    """Replace a sequence mid-generation; every sequence keeps decoding like
    the oracle's, the admitted one from its prompt."""
    cfg = TINY
    w = make_weights(cfg)
    prompts = make_prompts([9, 14, 5], cfg.vocab)
    new = make_prompts([7, 12, 3], cfg.vocab)
    rng = np.random.default_rng(33)
    dec = kf.Decoder(cfg, w, max_batch=3, max_k=3)
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, w))
    dec.prefill(prompts)
    ref.prefill(prompts)
    plan = [("step", 2), ("admit", [1], [0]), ("step", 2), ("admit", [0, 2], [1, 0]), ("step", 0),
            ("admit", [2], [2]), ("step", 3), ("step", 3)]
    for item in plan:
        if item[0] == "admit":
            _, slots, which = item
            P = len(ref.seqs[0]["pending"])
            ps = [new[i] for i in which]
            if min(len(p) for p in ps) < P:
                with pytest.raises(kf.KfError):
                    dec.admit(slots, ps)
                continue
            dec.admit(slots, ps)              # several slots in one call
            for slot, p in zip(slots, ps):
                ref.admit(slot, p, P)
        else:
            k = item[1]
            z = rng.random((3, max(k, 1)), dtype=np.float32)
            got = dec.step(k, z)
            want = ref.step(k, z).astype(np.int32)
            assert np.array_equal(got, want), (item, got, want)
        assert list(dec.lengths()) == [ref.cached_len(b) for b in range(3)]
    dec.close()


def test_admit_bf16_sampled(kf):
    cfg = LM1B
    w = make_weights(cfg)
    prompts = make_prompts([32] * 6, cfg.vocab)
    newp = make_prompts([20, 41], cfg.vocab)
    rng = np.random.default_rng(34)
    dec = kf.Decoder(cfg, w, max_batch=6, max_k=4)
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, w))
    dec.prefill(prompts)
    ref.prefill(prompts)
    worst, bad = 0.0, 0
    for i, k in enumerate([4, 4, 4, 4, 0, 4]):
        if i == 2:
            dec.admit(3, newp[0])
            ref.admit(3, newp[0], 4)
        if i == 3:
            dec.admit(0, newp[1])
            ref.admit(0, newp[1], 4)
        z = rng.random((6, max(k, 1)), dtype=np.float32)
        gt = dec.step(k, z)
        gl = dec.logits(max(k, 1))
        rt, rl = ref.step(k, z, want_logits=True)
        worst = max(worst, logit_check(gl, rl))
        _, _, u = compare_tokens(gt, rt, gl, rl, z)
        bad += u
        for b in range(6):
            ref.seqs[b]["pending"] = [int(t) for t in gt[b]]
        assert list(dec.lengths()) == [ref.cached_len(b) for b in range(6)]
    assert worst <= LOGIT_TOL and bad == 0
    dec.close()


def test_admit_recycles_pages(kf):
    """A pool with exactly the pages of two full-length sequences: admissions
    only succeed because the replaced sequence's pages return to the pool."""
    cfg = TINY                                    # max_len 64: 4 pages per sequence
    w = make_weights(cfg)
    dec = kf.Decoder(cfg, w, max_batch=2, max_k=2, n_pages=8)
    ref = oracle.OracleDecoder(oracle.OracleModel(cfg, w))
    prompts = make_prompts([40, 45], cfg.vocab)
    dec.prefill(prompts)
    ref.prefill(prompts)
    rng = np.random.default_rng(35)

    def run(n):
        for _ in range(n):
            z = rng.random((2, 2), dtype=np.float32)
            assert np.array_equal(dec.step(2, z), ref.step(2, z).astype(np.int32))

    run(5)                                        # both sequences now hold 4 pages: pool empty
    for rnd in range(3):
        p = make_prompts([30 + 5 * rnd], cfg.vocab)[0]
        slot = rnd % 2
        dec.admit(slot, p)
        ref.admit(slot, p, 2)
        run(3)
    dec.close()


def test_admit_and_teacher_errors(kf):
    cfg = TINY
    w = make_weights(cfg)
    dec = kf.Decoder(cfg, w, max_batch=2, max_k=2)
    with pytest.raises(kf.KfError) as e:
        dec.admit(0, [1, 2, 3])
    assert e.value.code == kf.KF_E_STATE
    dec.prefill(make_prompts([6, 6], cfg.vocab))
    for slot, toks, code in [(2, [1, 2], kf.KF_E_ARG), (-1, [1, 2], kf.KF_E_ARG),
                             (0, [cfg.vocab], kf.KF_E_ARG)]:
        with pytest.raises(kf.KfError) as e:
            dec.admit(slot, toks)
        assert e.value.code == code
    with pytest.raises(kf.KfError) as e:
        dec.admit([1, 1], [[1, 2], [3, 4]])                # a slot listed twice
    assert e.value.code == kf.KF_E_ARG
    dec.step(2, np.full((2, 2), 0.5, np.float32))        # P = 2 now
    with pytest.raises(kf.KfError) as e:
        dec.admit(1, [5])                                 # shorter than P
    assert e.value.code == kf.KF_E_ARG
    with pytest.raises(kf.KfError) as e:
        dec.teacher_step(3, np.full((2, 3), 0.5, np.float32))   # k > max_k
    assert e.value.code == kf.KF_E_ARG
    dec.admit(1, [5, 6, 7])
    with pytest.raises(kf.KfError) as e:
        dec.rewind()
    assert e.value.code == kf.KF_E_STATE
    dec.close()
