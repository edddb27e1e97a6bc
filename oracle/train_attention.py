"""Training-time attention masks of K-Forcing (App. C.2, SingleForward and
DoubleForward) and dense masked attention over them.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Token layout of one sequence, indices into the full token list:
  context  x_1..x_N                      -> 0 .. N-1
  block 1  k tokens per context position  -> N + t k + a      (t = 0..N-1, a = 0..k-1)
  block 2  (DoubleForward only)           -> N + N k + t k + a
SingleForward: block 1 holds the noise tokens.  DoubleForward: block 1 holds
the first-round predictions (Future-1), block 2 the fresh noise (Future-2).
"""
import numpy as np


def mask_single(N: int, k: int) -> np.ndarray:
    """M_S in {0,1}^{(N+Nk) x (N+Nk)} (App. C.2), rows = queries, cols = keys:
    context -> context causal; the noise group at context position t (1-based)
    attends to x_1..x_t; noise -> noise causal inside each group of k."""
    T = N + N * k
    m = np.zeros((T, T), bool)
    for i in range(N):
        for j in range(i + 1):
            m[i, j] = True
    for t in range(N):                 # 0-based group t <-> context position t + 1
        for a in range(k):
            q = N + t * k + a
            for j in range(t + 1):
                m[q, j] = True
            for b in range(a + 1):
                m[q, N + t * k + b] = True
    return m


def mask_double(N: int, k: int) -> np.ndarray:
    """M_D in {0,1}^{2Nk x (N+2Nk)} (App. C.2): queries Future-1 then
    Future-2, keys context, Future-1, Future-2.  Future-1 rows are M_S's
    noise rows; a Future-2 token of window t sees x_1..x_t, all k Future-1
    tokens of its window, and the Future-2 tokens of its window up to itself."""
    T = N + 2 * N * k
    m = np.zeros((2 * N * k, T), bool)
    ms = mask_single(N, k)
    m[:N * k, :N + N * k] = ms[N:, :]
    for t in range(N):
        for a in range(k):
            q = N * k + t * k + a
            for j in range(t + 1):
                m[q, j] = True
            for b in range(k):
                m[q, N + t * k + b] = True
            for b in range(a + 1):
                m[q, N + N * k + t * k + b] = True
    return m


def mask_full(N: int, k: int, blocks: int) -> np.ndarray:
    """The mask over every token of the layout as queries: M_S (blocks = 1),
    or the context rows of M_S stacked on M_D (blocks = 2)."""
    if blocks == 1:
        return mask_single(N, k)
    T = N + 2 * N * k
    m = np.zeros((T, T), bool)
    ms = mask_single(N, k)
    m[:N, :N] = ms[:N, :N]
    m[N:, :] = mask_double(N, k)
    return m


def masked_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, mask: np.ndarray) -> np.ndarray:
    """softmax(q k^T / sqrt(hd) restricted to mask) v in fp64.
    q [n, H, hd], k, v [m, H, hd], mask [n, m] (every row has a visible key)."""
    q, k, v = (np.asarray(a, np.float64) for a in (q, k, v))
    hd = q.shape[-1]
    s = np.einsum("nhd,mhd->hnm", q, k) / np.sqrt(hd)
    s = np.where(mask[None, :, :], s, -np.inf)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=-1, keepdims=True)
    return np.einsum("hnm,mhd->nhd", p, v)
