"""gmc_transport_noalloc against gmc_transport.

The no-allocation entry point exists for callers that must not allocate
device memory (an engine plugin inside enqueue(), code inside a CUDA graph
capture, a server with a fixed memory pool).  It keeps its scratch in a
fixed array inside libgmc.so instead of a caller workspace, so it must give
the same results as the workspace entry point, call after call, even though
every call reuses the same array.  This file is collected last on purpose.
"""

import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

ROW_TOL = 2e-2      # the bf16 transport tolerance of the parity tests
ROW_TOL_F32 = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _case(B, gh, gw, T, Hkv, d, D, K, dtype, seed):
    """Random inputs plus a valid support / assignment / weights for every image."""
    r = np.random.default_rng(seed)
    N = gh * gw
    tdt = torch.bfloat16 if dtype == 1 else torch.float32
    R = N + T
    hidden = torch.from_numpy(r.standard_normal((B * R, D), dtype=np.float32)).to(tdt).cuda()
    keys = torch.from_numpy(r.standard_normal((2 * B * R, Hkv, d), dtype=np.float32)).to(tdt).cuda()
    pos = torch.from_numpy(r.integers(0, 1000, size=3 * B * R, dtype=np.int32)).cuda()
    sup, asg = [], []
    for _ in range(B):
        s = np.sort(r.choice(N, size=K, replace=False)).astype(np.int32)
        a = s[r.integers(0, K, size=N)].astype(np.int32)
        a[s] = s
        sup.append(s)
        asg.append(a)
    support = torch.from_numpy(np.concatenate(sup)).cuda()
    assign = torch.from_numpy(np.concatenate(asg)).cuda()
    weights = torch.from_numpy(r.uniform(0.5, 2.0, size=B * N).astype(np.float32)).cuda()
    return dict(B=B, gh=gh, gw=gw, N=N, T=T, Hkv=Hkv, d=d, D=D, K=K, dtype=dtype, tdt=tdt,
                hidden=hidden, keys=keys, pos=pos, support=support, assign=assign, weights=weights)


def _outputs(c):
    rows = c["B"] * (c["K"] + c["T"])
    return (torch.empty(c["B"] * c["K"], dtype=torch.int32, device="cuda"),
            torch.empty((rows, c["D"]), dtype=c["tdt"], device="cuda"),
            torch.empty((2 * rows, c["Hkv"], c["d"]), dtype=c["tdt"], device="cuda"),
            torch.empty(3 * rows, dtype=torch.int32, device="cuda"))


def _run_both(c):
    from paper_2608_02134_gb300 import gmc
    prob = gmc.problem(c["B"], c["gh"], c["gw"], c["Hkv"], c["dtype"])
    p = gmc.default_params()
    ref = _outputs(c)
    ws = gmc.alloc_workspace(gmc.transport_workspace_size(prob, c["N"], c["T"], c["K"]))
    gmc.transport(prob, p, c["hidden"], c["keys"], c["pos"], c["support"], c["assign"],
                  c["weights"], c["N"], c["T"], c["d"], c["D"], c["K"], *ref, ws)
    got = _outputs(c)
    status = torch.full((1,), 0xFFFF, dtype=torch.int32, device="cuda")
    gmc.transport_noalloc(prob, p, c["hidden"], c["keys"], c["pos"], c["support"], c["assign"],
                          c["weights"], c["N"], c["T"], c["d"], c["D"], c["K"], *got,
                          device_status=status)
    torch.cuda.synchronize()
    assert gmc.read_status(ws) == 0
    assert int(status.item()) == 0
    return ref, got


def _compare(ref, got, tol):
    from tests import parity
    idx_r, hid_r, kv_r, pos_r = (t.cpu() for t in ref)
    idx_g, hid_g, kv_g, pos_g = (t.cpu() for t in got)
    assert torch.equal(idx_r, idx_g)
    assert torch.equal(pos_r, pos_g)
    assert torch.equal(kv_r.view(torch.uint8) if kv_r.dtype == torch.bfloat16 else kv_r,
                       kv_g.view(torch.uint8) if kv_g.dtype == torch.bfloat16 else kv_g)
    err = parity.rel_row_err(hid_g.float().numpy().astype(np.float64),
                             hid_r.float().numpy().astype(np.float64))
    assert err <= tol, err


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls():
    # first call: two bf16 images; second call: a different fp32 problem reusing the array
    c1 = _case(B=2, gh=12, gw=12, T=9, Hkv=2, d=64, D=256, K=30, dtype=1, seed=5)
    ref, got = _run_both(c1)
    _compare(ref, got, ROW_TOL)
    c2 = _case(B=1, gh=8, gw=8, T=4, Hkv=4, d=16, D=64, K=16, dtype=0, seed=6)
    ref, got = _run_both(c2)
    _compare(ref, got, ROW_TOL_F32)


def test_noalloc_rejects_problems_above_its_fixed_scratch():
    from paper_2608_02134_gb300 import gmc
    prob = gmc.problem(64, 36, 36, 4, gmc.GMC_BF16)        # 64 * 1296 rows > 65536
    fake = ctypes.c_void_p(1 << 20)
    rc = gmc.lib().gmc_transport_noalloc(ctypes.byref(prob), None, fake, fake, fake, fake, fake,
                                         fake, 1296, 8, 128, 3584, 257, fake, fake, fake, fake,
                                         None, None)
    assert rc == gmc.GMC_ERR_UNSUPPORTED
