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
    lib.kf_op_status.argtypes = [ctypes.c_void_p]
    lib.kf_op_status.restype = ctypes.c_int
    return torch, lib, kf


def _tokens(torch, lib, fn, x, w, z, tau, map_kind):
    rows, d = x.shape
    out = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
    rc = getattr(lib, fn)(rows, w.shape[0], d, x.data_ptr(), w.data_ptr(), z.data_ptr(), tau,
                          map_kind, out.data_ptr(), None)
    assert rc == 0, rc
    assert lib.kf_op_status(None) == 0     # no kernel of the call flagged an error
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


def test_noalloc_matches_oracle(env):
    """The no-allocation entry against the oracle's inverse-CDF and argmax maps
    on fp64 logits of the same bf16 operands (the rule of test_gpu_head_op)."""
    torch, lib, _ = env
    from test_gpu_head_op import check_against_oracle
    g = torch.Generator(device="cuda").manual_seed(77)
    x = torch.randn(40, 256, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(5000, 256, device="cuda", generator=g) * 0.05).to(torch.bfloat16)
    z = torch.rand(40, device="cuda", generator=g)
    for map_kind in (0, 1):
        got = _tokens(torch, lib, "kf_op_head_tokens_noalloc", x, w, z, 0.8, map_kind)
        assert check_against_oracle(x, w, z, 0.8, map_kind, got) == 0


_NO_ALLOC_PROBE = r"""
import ctypes, sys
import torch
sys.path.insert(0, sys.argv[1])
from paper_2606_10820_gb300 import kforcing as kf
lib = kf.load_library()
fn = lib.kf_op_head_tokens_noalloc
fn.argtypes = [ctypes.c_int32] * 3 + [ctypes.c_void_p] * 3 + [ctypes.c_float, ctypes.c_int32,
                                                               ctypes.c_void_p, ctypes.c_void_p]
fn.restype = ctypes.c_int
g = torch.Generator(device="cuda").manual_seed(3)
cases = []
for rows, V, d in [(64, 30522, 768), (200, 1000, 128), (3, 50257, 256)]:
    x = torch.randn(rows, d, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(V, d, device="cuda", generator=g) * 0.05).to(torch.bfloat16)
    z = torch.rand(2, rows, device="cuda", generator=g)
    out = torch.zeros(rows, dtype=torch.int32, device="cuda")
    cases.append((rows, V, d, x, w, z, out))
torch.cuda.synchronize()
def run(i):
    for rows, V, d, x, w, z, out in cases:
        for m in (0, 1):
            rc = fn(rows, V, d, x.data_ptr(), w.data_ptr(), z[i].data_ptr(), 1.0, m, out.data_ptr(), None)
            assert rc == 0, rc
    torch.cuda.synchronize()
run(0)                       # module load and every kernel variant once
before = torch.cuda.mem_get_info()[0]
for _ in range(3):
    run(1)
after = torch.cuda.mem_get_info()[0]
print("free bytes before", before, "after", after)
assert before == after, (before, after)
"""


def test_noalloc_allocates_nothing():
    """In a fresh process that calls only the no-allocation entry: after one
    warm-up round (module load, every kernel variant), repeated calls of three
    shapes leave the device's free memory (cudaMemGetInfo) unchanged."""
    import os
    import subprocess
    import sys
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    p = subprocess.run([sys.executable, "-c", _NO_ALLOC_PROBE, root], capture_output=True, text=True,
                       timeout=600)
    assert p.returncode == 0, p.stdout + p.stderr
