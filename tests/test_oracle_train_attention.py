"""Pins of the training-time attention oracle (App. C.2) to the paper's
closed-form mask sizes and to the inference-time causal attention (Sec. 3.3),
which the decode oracle pins separately."""
import numpy as np
import pytest

from oracle import causal_attention
from oracle import train_attention as ta

GRID = [(1, 1), (1, 4), (2, 3), (5, 1), (5, 2), (7, 4), (16, 8), (33, 3)]


@pytest.mark.parametrize("N,k", GRID)
def test_single_mask_size_is_the_closed_form(N, k):
    # |M_S| = N(N+1)/2 + kN(N+1)/2 + N k(k+1)/2
    want = N * (N + 1) // 2 + k * N * (N + 1) // 2 + N * k * (k + 1) // 2
    assert int(ta.mask_single(N, k).sum()) == want


@pytest.mark.parametrize("N,k", GRID)
def test_double_mask_future2_size_is_the_closed_form(N, k):
    # Future-2 queries: |M_D| = kN(N+1)/2 + N k^2 + N k(k+1)/2
    want = k * N * (N + 1) // 2 + N * k * k + N * k * (k + 1) // 2
    md = ta.mask_double(N, k)
    assert int(md[N * k:].sum()) == want
    # Future-1 rows are M_S's noise rows
    np.testing.assert_array_equal(md[:N * k, :N + N * k], ta.mask_single(N, k)[N:])
    assert not md[:N * k, N + N * k:].any()


def _qkv(n, H=2, hd=8, seed=0):
    rng = np.random.default_rng(seed)
    return [rng.standard_normal((n, H, hd)) for _ in range(3)]


@pytest.mark.parametrize("N,k", [(5, 3), (9, 4), (6, 1)])
def test_single_noise_rows_equal_inference_attention(N, k):
    """Group t of SingleForward attends exactly like the k noise rows of a
    decode step whose cache holds x_1..x_t (positions t+1.. for the noise)."""
    T = N + N * k
    q, kk, v = _qkv(T, seed=N * 10 + k)
    out = ta.masked_attention(q, kk, v, ta.mask_single(N, k))
    # context rows: plain causal attention
    pos = np.arange(N)
    np.testing.assert_allclose(out[:N], causal_attention(q[:N], kk[:N], v[:N], pos, pos), atol=1e-12)
    for t in range(N):
        g = slice(N + t * k, N + (t + 1) * k)
        keys = np.concatenate([kk[:t + 1], kk[g]])
        vals = np.concatenate([v[:t + 1], v[g]])
        k_pos = np.concatenate([np.arange(t + 1), t + 1 + np.arange(k)])
        want = causal_attention(q[g], keys, vals, t + 1 + np.arange(k), k_pos)
        np.testing.assert_allclose(out[g], want, atol=1e-12)


@pytest.mark.parametrize("N,k", [(5, 3), (4, 2)])
def test_double_future2_rows_equal_two_sequential_passes(N, k):
    """A Future-2 token sees its window's Future-1 tokens as extended context:
    causal attention over [x_1..x_t ; Future-1 window ; Future-2 window]."""
    T = N + 2 * N * k
    q, kk, v = _qkv(T, seed=N + 7 * k)
    md = ta.mask_double(N, k)
    out = ta.masked_attention(q[N:], kk, v, md)
    for t in range(N):
        f1 = slice(N + t * k, N + (t + 1) * k)
        f2 = slice(N + N * k + t * k, N + N * k + (t + 1) * k)
        keys = np.concatenate([kk[:t + 1], kk[f1], kk[f2]])
        vals = np.concatenate([v[:t + 1], v[f1], v[f2]])
        k_pos = np.arange(t + 1 + 2 * k)
        want = causal_attention(q[f2], keys, vals, t + 1 + k + np.arange(k), k_pos)
        np.testing.assert_allclose(out[N * k + t * k: N * k + (t + 1) * k], want, atol=1e-12)


def test_planted_staircase_off_by_one_is_caught():
    """A staircase that lets group t also see x_{t+1} breaks the closed form."""
    N, k = 6, 3
    m = ta.mask_single(N, k)
    bad = m.copy()
    for t in range(N - 1):
        bad[N + t * k:N + (t + 1) * k, t + 1] = True
    want = N * (N + 1) // 2 + k * N * (N + 1) // 2 + N * k * (k + 1) // 2
    assert int(m.sum()) == want and int(bad.sum()) != want
