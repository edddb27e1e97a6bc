"""tcgen05 GEMM (and the SIMT GEMM) against a plain PyTorch fp32 matmul of
the same bf16 operands, through the C ABI of include/kforcing_ops.h."""
import ctypes

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

SHAPES = [
    (1, 128, 64),        # one row, one K block
    (5, 256, 768),       # tiny M, split-K
    (130, 384, 768),     # ragged M across two row tiles
    (64, 768, 3072),     # AR-step MLP-down shape, deep split-K
    (512, 2304, 768),    # LM1B k=4 QKV
    (512, 768, 3072),    # LM1B k=4 MLP-down: 128-wide tiles, split-K 4
    (320, 3072, 768),    # first-step rows (P=1), MLP-up
    (256, 30720, 768),   # LM-head shape (vocab padded to 256)
    (1000, 200, 128),    # N not a multiple of the tile
    (200, 640, 320),     # odd number of 64-wide K blocks: a short last pipeline stage
    (4096, 768, 3072),   # OWT batch 512 k=4 MLP-down: one wave of 128 192-wide tiles
    (3900, 700, 768),    # 192-wide tiles with ragged M and N (the last W box partly past N)
    (4096, 768, 768),    # OWT batch 512 k=4 O projection: 192-wide tiles
    (2100, 2340, 768),   # persistent 256-wide tiles with ragged M and N
    (4096, 2304, 768),   # OWT batch 512 k=4 QKV shape: two tiles per CTA
    (4096, 3072, 768),   # OWT batch 512 k=4 MLP-up shape: 384 tiles on the persistent loop
]

PERSISTENT = [(2100, 2340, 768), (4096, 2304, 768), (4096, 3072, 768)]

# the skinny warp-MMA kernel (M <= 64): one K range per CTA, or K split over
# clusters of 2, 4 and 8 CTAs; ragged M (one 8-row box, several n-blocks)
# and N (the last 16-column block partly past N)
SKINNY = [
    (1, 128, 64),        # one row, one K atom
    (8, 2304, 768),      # OWT batch 1, k = 4 QKV rows
    (6, 3072, 768),      # MLP-up, a partial 8-row box
    (64, 768, 3072),     # batch 8, k = 4 MLP-down: K over a cluster of 8
    (33, 768, 768),      # five n-blocks, K split 2
    (17, 200, 128),      # N not a multiple of 16
    (40, 768, 832),      # 13 K atoms: no power-of-two split divides them
    (16, 1000, 3072),    # K split 4, ragged N
]


@pytest.fixture(scope="module")
def env():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g
    g.build()
    from paper_2606_10820_gb300 import kforcing as kf
    lib = kf.load_library()
    lib.kf_op_gemm_bf16.argtypes = [ctypes.c_int32] * 4 + [ctypes.c_void_p] * 4
    lib.kf_op_gemm_bf16.restype = ctypes.c_int
    return torch, lib


def _run(torch, lib, impl, A, W):
    M, K = A.shape
    N = W.shape[0]
    out = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    rc = lib.kf_op_gemm_bf16(impl, M, N, K, A.data_ptr(), W.data_ptr(), out.data_ptr(), None)
    assert rc == 0
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("M,N,K", SHAPES)
def test_gemm_matches_fp32_matmul(env, M, N, K):
    torch, lib = env
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N * 3 + K)
    A = (torch.randn(M, K, device="cuda", generator=g) * 0.5).to(torch.bfloat16)
    W = (torch.randn(N, K, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    ref = (A.double() @ W.double().T).float()
    scale = ref.abs().max().item()
    for impl in (0, 1, 2):     # tcgen05, SIMT, tcgen05 one CTA per tile
        out = _run(torch, lib, impl, A, W)
        assert torch.isfinite(out).all()
        err = (out - ref).abs().max().item()
        assert err <= 1e-4 * scale + 1e-6, (impl, err, scale)


@pytest.mark.parametrize("M,N,K", PERSISTENT)
def test_persistent_tiles_equal_per_tile_ctas(env, M, N, K):
    """Past a wave of tiles the persistent tile loop computes each 128 x 256
    tile with the same K order as a CTA per tile: identical bits."""
    torch, lib = env
    g = torch.Generator(device="cuda").manual_seed(M + N + K)
    A = (torch.randn(M, K, device="cuda", generator=g) * 0.5).to(torch.bfloat16)
    W = (torch.randn(N, K, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    assert torch.equal(_run(torch, lib, 0, A, W), _run(torch, lib, 2, A, W))


def test_gemm_repeat_is_deterministic(env):
    """Split-K partials are reduced in split order: identical bits each run."""
    torch, lib = env
    g = torch.Generator(device="cuda").manual_seed(1)
    A = torch.randn(64, 3072, device="cuda", generator=g).to(torch.bfloat16)
    W = (torch.randn(768, 3072, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    a = _run(torch, lib, 0, A, W)
    b = _run(torch, lib, 0, A, W)
    assert torch.equal(a, b)


@pytest.mark.parametrize("M,N,K", SKINNY)
def test_skinny_gemm_matches_fp32_matmul(env, M, N, K):
    torch, lib = env
    g = torch.Generator(device="cuda").manual_seed(M * 11 + N * 5 + K)
    A = (torch.randn(M, K, device="cuda", generator=g) * 0.5).to(torch.bfloat16)
    W = (torch.randn(N, K, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    ref = (A.double() @ W.double().T).float()
    scale = ref.abs().max().item()
    out = _run(torch, lib, 3, A, W)
    assert torch.isfinite(out).all()
    err = (out - ref).abs().max().item()
    assert err <= 1e-4 * scale + 1e-6, (err, scale)
    # split partials are summed in split order: identical bits each run
    assert torch.equal(out, _run(torch, lib, 3, A, W))
