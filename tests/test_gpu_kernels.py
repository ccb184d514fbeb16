"""Kernel-level numerics against plain PyTorch references of the same op."""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _cos_ref(h64: torch.Tensor) -> torch.Tensor:
    n = h64.norm(dim=1).clamp_min(1e-12)
    x = h64 / n[:, None]
    return x @ x.T


@pytest.mark.parametrize("B,gh,gw,D,tlens,dtype", [
    (1, 36, 36, 3584, [64], torch.bfloat16),        # 11 x 11 tiles, ragged last tile
    (1, 16, 8, 256, [5], torch.bfloat16),          # exactly one 128-row tile
    (3, 10, 20, 512, [7, 1, 30], torch.bfloat16),  # shifted last tile, ragged text offsets
    (2, 24, 24, 4096, [32, 32], torch.bfloat16),
    (2, 12, 12, 128, [9, 1], torch.bfloat16),      # 2 x 2 tiles, 16-row ragged edge, T_b = 1
    (1, 13, 11, 256, [4], torch.bfloat16),         # N % 4 != 0: CUDA-core path
    (1, 10, 10, 40, [3], torch.float32),           # CUDA-core path
    # the general kernel's symmetric mode (its tiles fill the GPU at least once):
    (1, 64, 64, 256, [17], torch.bfloat16),        # document page grid, 128 x 256 tiles
    (6, 36, 36, 640, [64, 3, 40, 1, 64, 16], torch.bfloat16),  # a batch, ragged text
    (4, 50, 50, 200, [8, 8, 8, 8], torch.bfloat16),  # ragged row and column tiles, D % 64 != 0
])
def test_cosine_matches_fp64_reference(B, gh, gw, D, tlens, dtype):
    from paper_2608_02134_gb300 import gmc
    N = gh * gw
    r = np.random.default_rng(N + D)
    ragged = len(set(tlens)) > 1
    rows = [r.standard_normal((N + t, D), dtype=np.float32) * r.uniform(0.2, 3.0, size=(N + t, 1)).astype(np.float32)
            for t in tlens]
    hid = torch.from_numpy(np.concatenate(rows)).to(dtype).cuda()
    off = torch.tensor(np.concatenate([[0], np.cumsum(tlens)]), dtype=torch.int32, device="cuda")
    prob = gmc.problem(B, gh, gw, 1, gmc.GMC_BF16 if dtype == torch.bfloat16 else gmc.GMC_F32,
                       off if ragged else None)
    out = torch.full((B, N, N), float("nan"), dtype=torch.float32, device="cuda")
    ws = gmc.cosine(prob, gmc.default_params(), hid, N, max(tlens), D, out)
    torch.cuda.synchronize()
    assert gmc.read_status(ws) == 0
    start = 0
    for b in range(B):
        h = hid[start:start + N].double()
        ref = _cos_ref(h)
        got = out[b].double()
        assert torch.isfinite(got).all(), "unwritten entries"
        err = (got - ref).abs().max().item()
        assert err < 2e-5, (b, err)
        start += N + tlens[b]
