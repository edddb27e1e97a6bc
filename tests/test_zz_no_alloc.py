"""kf_op_head_tokens_noalloc: the LM-head noise -> token map for callers that
must not allocate device memory (its scratch is a fixed array in the
library's device image).  Its tokens must equal those of kf_op_head_tokens,
which allocates its scratch, on two calls in a row.

This file is collected last on purpose: it must pass both alone in a fresh
process and after every other test.
"""
import ctypes

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

KF_E_CAPACITY = -2


@pytest.fixture(scope="module")
def env():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2606_10820_gb300 import kforcing as kf
    lib = kf.load_library()
    args = [ctypes.c_int32] * 3 + [ctypes.c_void_p] * 3 + \
        [ctypes.c_float, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p]
    for fn in ("kf_op_head_tokens", "kf_op_head_tokens_noalloc"):
        getattr(lib, fn).argtypes = args
        getattr(lib, fn).restype = ctypes.c_int
    return torch, lib, kf


def _tokens(torch, lib, fn, x, w, z, tau, map_kind):
    rows, d = x.shape
    out = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
    rc = getattr(lib, fn)(rows, w.shape[0], d, x.data_ptr(), w.data_ptr(), z.data_ptr(), tau,
                          map_kind, out.data_ptr(), None)
    assert rc == 0, rc
    torch.cuda.synchronize()
    return out.cpu().numpy()


@pytest.mark.parametrize("rows,V,d", [(64, 30522, 768), (5, 1000, 128), (160, 50257, 768)])
@pytest.mark.parametrize("map_kind", [0, 1])
def test_noalloc_matches_allocating_entry(env, rows, V, d, map_kind):
    torch, lib, _ = env
    g = torch.Generator(device="cuda").manual_seed(rows * 131 + V)
    x = torch.randn(rows, d, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(V, d, device="cuda", generator=g) * 0.05).to(torch.bfloat16)
    z = torch.rand(rows, device="cuda", generator=g)
    want = _tokens(torch, lib, "kf_op_head_tokens", x, w, z, 1.0, map_kind)
    # two calls in a row: the shared scratch keeps the previous call's contents
    first = _tokens(torch, lib, "kf_op_head_tokens_noalloc", x, w, z, 1.0, map_kind)
    z2 = torch.rand(rows, device="cuda", generator=g)
    want2 = _tokens(torch, lib, "kf_op_head_tokens", x, w, z2, 0.7, map_kind)
    second = _tokens(torch, lib, "kf_op_head_tokens_noalloc", x, w, z2, 0.7, map_kind)
    np.testing.assert_array_equal(first, want)
    np.testing.assert_array_equal(second, want2)
    assert ((first >= 0) & (first < V)).all()


def test_noalloc_rejects_oversize(env):
    torch, lib, kf = env
    rows, V, d = 300, 30522, 64        # 300 * 954 records > 262144
    x = torch.zeros(rows, d, dtype=torch.bfloat16, device="cuda")
    w = torch.zeros(V, d, dtype=torch.bfloat16, device="cuda")
    z = torch.zeros(rows, device="cuda")
    out = torch.zeros(rows, dtype=torch.int32, device="cuda")
    rc = lib.kf_op_head_tokens_noalloc(rows, V, d, x.data_ptr(), w.data_ptr(), z.data_ptr(), 1.0,
                                       0, out.data_ptr(), None)
    assert rc == KF_E_CAPACITY
    assert "static scratch" in kf.kf_last_error()
