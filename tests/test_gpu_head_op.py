"""The fused LM-head noise -> token map alone (kf_op_head_tokens) against
the oracle's maps on logits from a plain fp64 matmul of the same bf16
operands.  The GPU never writes logits: only the chunk records and tokens."""
import ctypes

import numpy as np
import pytest

import oracle

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
    lib.kf_op_head_tokens.argtypes = [ctypes.c_int32] * 3 + [ctypes.c_void_p] * 3 + \
        [ctypes.c_float, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p]
    lib.kf_op_head_tokens.restype = ctypes.c_int
    lib.kf_op_status.argtypes = [ctypes.c_void_p]
    lib.kf_op_status.restype = ctypes.c_int
    return torch, lib


def _case(torch, rows, V, d, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    x = torch.randn(rows, d, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(V, d, device="cuda", generator=g) * 0.05).to(torch.bfloat16)
    z = torch.rand(rows, device="cuda", generator=g)
    return x, w, z


def run_op(lib, torch, x, w, z, tau, map_kind, fn="kf_op_head_tokens"):
    rows, d = x.shape
    V = w.shape[0]
    out = torch.full((rows,), -1, dtype=torch.int32, device="cuda")
    rc = getattr(lib, fn)(rows, V, d, x.data_ptr(), w.data_ptr(), z.data_ptr(), tau, map_kind,
                          out.data_ptr(), None)
    assert rc == 0
    assert lib.kf_op_status(None) == 0
    return out.cpu().numpy()


def check_against_oracle(x, w, z, tau, map_kind, got):
    lg = (x.double() @ w.double().T).cpu().numpy() / tau
    zz = z.cpu().numpy()
    bad = 0
    for i in range(lg.shape[0]):
        if map_kind == 0:
            want = oracle.icdf_token(lg[i], zz[i], np.float32)
            if got[i] != want:
                p = np.exp(lg[i] - lg[i].max())
                F = np.cumsum(p / p.sum())
                # fp32 accumulation-order error of the logits and the sums: z
                # must lie that close to every CDF boundary between the two
                # tokens' bins, F(lo) .. F(hi - 1)
                lo, hi = sorted((int(got[i]), int(want)))
                if np.abs(zz[i] - F[lo:hi]).max() > 1e-4:
                    bad += 1
        else:
            want = oracle.argmax_token(lg[i])
            if got[i] != want and lg[i][want] - lg[i][got[i]] > 1e-4:
                bad += 1
    return bad


# (8 rows at V = 50,257: the persistent loop over 128-wide tiles of one M tile;
# 130 and 520 rows: the persistent loop over 256-wide tiles, a ragged last M tile)
@pytest.mark.parametrize("rows,V,d,tau", [(3, 1000, 128, 1.0), (64, 30522, 768, 1.0),
                                          (8, 50257, 768, 1.0), (130, 50257, 768, 0.5),
                                          (520, 50257, 768, 1.0), (256, 32, 64, 1.0)])
@pytest.mark.parametrize("map_kind", [0, 1])
def test_head_tokens_match_oracle(env, rows, V, d, tau, map_kind):
    torch, lib = env
    x, w, z = _case(torch, rows, V, d, rows + V + map_kind)
    got = run_op(lib, torch, x, w, z, tau, map_kind)
    assert ((got >= 0) & (got < V)).all()
    assert check_against_oracle(x, w, z, tau, map_kind, got) == 0


def test_head_tokens_noise_extremes(env):
    """z = 0 picks the first id with mass; z just below 1 the last one."""
    torch, lib = env
    x, w, _ = _case(torch, 8, 4000, 256, 5)
    z = torch.tensor([0.0, 0.0, 0.5, 0.5, 0.9999999, 0.9999999, 0.25, 0.75], device="cuda")
    got = run_op(lib, torch, x, w, z, 1.0, 0)
    assert got[0] == 0 and got[1] == 0
    assert got[4] >= 3990 and got[5] >= 3990
    assert check_against_oracle(x, w, z, 1.0, 0, got) == 0


def test_head_tokens_rejects_bad_args(env):
    torch, lib = env
    x, w, z = _case(torch, 2, 100, 64, 1)
    out = torch.zeros(2, dtype=torch.int32, device="cuda")
    assert lib.kf_op_head_tokens(2, 100, 60, x.data_ptr(), w.data_ptr(), z.data_ptr(), 1.0, 0,
                                 out.data_ptr(), None) != 0
    assert lib.kf_op_head_tokens(2, 100, 64, x.data_ptr(), w.data_ptr(), z.data_ptr(), 0.0, 0,
                                 out.data_ptr(), None) != 0
