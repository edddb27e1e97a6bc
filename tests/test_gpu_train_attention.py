"""kf_op_train_attention (SingleForward / DoubleForward, App. C.2) against the
oracle's dense masked attention in fp64, through the C ABI (needs a GB300).

Tolerance: the output rows are convex combinations of V rows; the kernel
rounds the probabilities to bf16 for the P.V product (relative error <= 2^-9
each, the row sums use the rounded values), so |out - ref| <= 2^-8 max|V| up
to fp32 accumulation: the test allows 8e-3 max|V|.
"""
import ctypes

import numpy as np
import pytest

from oracle import train_attention as ta

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2606_10820_gb300 import kforcing as kf
    lib = kf.load_library()
    lib.kf_op_train_attention.argtypes = [ctypes.c_int32] * 7 + [ctypes.c_void_p] * 4 + \
        [ctypes.c_int32, ctypes.c_void_p]
    lib.kf_op_train_attention.restype = ctypes.c_int
    return torch, lib


def _run(torch, lib, blocks, B, H, N, k, q_begin=None, q_end=None, dense=0, seed=0):
    T = N + blocks * N * k
    q_begin = 0 if q_begin is None else q_begin
    q_end = T if q_end is None else q_end
    g = torch.Generator(device="cuda").manual_seed(seed)
    q, kk, v = ((torch.randn(B, T, H, 64, device="cuda", generator=g)).to(torch.bfloat16) for _ in range(3))
    out = torch.full((B, q_end - q_begin, H, 64), float("nan"), device="cuda")
    rc = lib.kf_op_train_attention(blocks, B, H, N, k, q_begin, q_end, q.data_ptr(), kk.data_ptr(),
                                   v.data_ptr(), out.data_ptr(), dense, None)
    assert rc == 0, rc
    torch.cuda.synchronize()
    return [x.float().cpu().numpy() for x in (q, kk, v)] + [out.cpu().numpy()]


def _check(q, kk, v, out, blocks, N, k, q_begin, q_end):
    mask = ta.mask_full(N, k, blocks)[q_begin:q_end]
    for b in range(q.shape[0]):
        ref = ta.masked_attention(q[b, q_begin:q_end], kk[b], v[b], mask)
        err = np.abs(out[b] - ref).max()
        assert err <= 8e-3 * np.abs(v[b]).max(), (b, err)


CASES = [
    (1, 2, 3, 5, 3), (1, 1, 2, 33, 4), (1, 1, 1, 130, 1), (1, 1, 2, 1, 8), (1, 1, 2, 70, 8),
    (2, 2, 2, 9, 2), (2, 1, 3, 20, 4), (2, 1, 2, 7, 5), (2, 1, 1, 40, 3),
]


# flags: 1 every key tile (dense mask), 2 the warp-level MMA kernel instead of tcgen05
@pytest.mark.parametrize("blocks,B,H,N,k", CASES)
@pytest.mark.parametrize("dense", [0, 1, 2, 3])
def test_train_attention_matches_dense_oracle(env, blocks, B, H, N, k, dense):
    torch, lib = env
    q, kk, v, out = _run(torch, lib, blocks, B, H, N, k, dense=dense, seed=N * 31 + k)
    assert np.isfinite(out).all()
    _check(q, kk, v, out, blocks, N, k, 0, N + blocks * N * k)


def test_double_future2_only_rows(env):
    """DoubleForward with KV reuse: only the Future-2 queries."""
    torch, lib = env
    blocks, B, H, N, k = 2, 2, 2, 37, 4
    qb, qe = N + N * k, N + 2 * N * k
    q, kk, v, out = _run(torch, lib, blocks, B, H, N, k, qb, qe, seed=5)
    _check(q, kk, v, out, blocks, N, k, qb, qe)


@pytest.mark.parametrize("flags", [0, 2])
def test_long_sequence_sampled_rows(env, flags):
    """N = 512, k = 4 (T = 2560): rows sampled across the blocks."""
    torch, lib = env
    blocks, B, H, N, k = 1, 1, 2, 512, 4
    q, kk, v, out = _run(torch, lib, blocks, B, H, N, k, dense=flags, seed=9)
    mask = ta.mask_single(N, k)
    rows = np.array([0, 1, 127, 128, 511, N, N + 3, N + 4 * 200 + 2, N + 4 * 511 + 3])
    ref = ta.masked_attention(q[0, rows], kk[0], v[0], mask[rows])
    assert np.abs(out[0, rows] - ref).max() <= 8e-3 * np.abs(v[0]).max()


def test_kernels_agree_double_forward(env):
    """DoubleForward N = 300, k = 4 (T = 2700, ragged 128-row tiles): the
    tcgen05 kernel and the warp-level MMA kernel within the tolerance of each
    other on every row, and the oracle on sampled rows."""
    torch, lib = env
    blocks, B, H, N, k = 2, 2, 3, 300, 4
    q, kk, v, out = _run(torch, lib, blocks, B, H, N, k, dense=0, seed=11)
    out2 = _run(torch, lib, blocks, B, H, N, k, dense=2, seed=11)[3]
    assert np.isfinite(out).all()
    assert np.abs(out - out2).max() <= 8e-3 * np.abs(v).max()
    mask = ta.mask_full(N, k, blocks)
    rows = np.array([0, 127, 128, 299, N, N + 517, N + N * k - 1, N + N * k, N + N * k + 3 * 77 + 2,
                     N + 2 * N * k - 1])
    for b in range(B):
        ref = ta.masked_attention(q[b, rows], kk[b], v[b], mask[rows])
        assert np.abs(out[b, rows] - ref).max() <= 8e-3 * np.abs(v[b]).max()


def test_argument_errors(env):
    torch, lib = env
    buf = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(64, device="cuda")
    p = buf.data_ptr()
    for args in [(3, 1, 1, 4, 2, 0, 12), (1, 1, 1, 4, 2, 0, 13), (1, 1, 1, 4, 2, 5, 5),
                 (1, 0, 1, 4, 2, 0, 12), (2, 1, 1, 4, 0, 0, 4)]:
        assert lib.kf_op_train_attention(*args, p, p, p, out.data_ptr(), 0, None) == -1, args
    # an unknown flag
    assert lib.kf_op_train_attention(1, 1, 1, 4, 2, 0, 12, p, p, p, out.data_ptr(), 4, None) == -1


@pytest.mark.parametrize("blocks,B,H,N,k", [(1, 4, 12, 128, 4), (1, 4, 12, 256, 4), (2, 2, 12, 256, 4)])
def test_many_items_per_cta(env, blocks, B, H, N, k):
    """More (query tile, head, sequence) items than SMs, so each persistent
    CTA carries its tiles, buffers and row sums across several items: every
    row against the warp-level MMA kernel, sampled rows against the oracle."""
    torch, lib = env
    T = N + blocks * N * k
    q, kk, v, out = _run(torch, lib, blocks, B, H, N, k, dense=0, seed=N + B)
    out2 = _run(torch, lib, blocks, B, H, N, k, dense=2, seed=N + B)[3]
    assert np.isfinite(out).all()
    assert np.abs(out - out2).max() <= 8e-3 * np.abs(v).max()
    mask = ta.mask_full(N, k, blocks)
    rows = np.array([0, 127, N - 1, N, N + 5, N + N * k // 2 + 1, N + N * k - 1, T - 1])
    for b in range(B):
        ref = ta.masked_attention(q[b, rows], kk[b], v[b], mask[rows])
        assert np.abs(out[b, rows] - ref).max() <= 8e-3 * np.abs(v[b]).max()


def test_future2_rows_many_items(env):
    """DoubleForward's Future-2 rows only (q_begin > 0) over more items than
    SMs: every row against the warp-level MMA kernel, sampled rows against
    the oracle."""
    torch, lib = env
    blocks, B, H, N, k = 2, 2, 12, 256, 4
    qb, qe = N + N * k, N + 2 * N * k
    q, kk, v, out = _run(torch, lib, blocks, B, H, N, k, qb, qe, seed=13)
    out2 = _run(torch, lib, blocks, B, H, N, k, qb, qe, dense=2, seed=13)[3]
    assert np.isfinite(out).all()
    assert np.abs(out - out2).max() <= 8e-3 * np.abs(v).max()
    mask = ta.mask_full(N, k, blocks)[qb:qe]
    rel = np.array([0, 1, 127, 128, 511, 777, qe - qb - 1])
    for b in range(B):
        ref = ta.masked_attention(q[b, qb + rel], kk[b], v[b], mask[rel])
        assert np.abs(out[b, rel] - ref).max() <= 8e-3 * np.abs(v[b]).max()
