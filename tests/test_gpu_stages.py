"""GPU parity of the staged entry points gmc_select and gmc_transport.

gmc_select gets the very same fp32 client matrix the oracle reads, so only
the solver's arithmetic differs; gmc_transport gets the oracle's own support,
assignment and population weights.
"""

import numpy as np
import pytest
import torch

from oracle import gmc_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _select_gpu(C: np.ndarray, K: int, **pk):
    from paper_2608_02134_gb300 import gmc
    from tests import parity
    B, M, N = C.shape
    p = gmc.default_params(**pk)
    ws = gmc.alloc_workspace(gmc.select_workspace_size(B, M, N, K, p))
    L = gmc.TraceLayout()
    prob = gmc.problem(B, 1, N, 1, gmc.GMC_F32)
    import ctypes
    assert gmc.lib().gmc_get_trace_layout(ctypes.byref(prob), ctypes.byref(p), N, 1, 0, K,
                                          ctypes.byref(L)) == 0
    tr = torch.zeros(B * L.bytes_per_image, dtype=torch.uint8, device="cuda")
    Cd = torch.from_numpy(np.ascontiguousarray(C, dtype=np.float32)).cuda()
    out = torch.empty(B * K, dtype=torch.int32, device="cuda")
    gmc.select(Cd, B, M, N, K, p, out, ws, tr)
    torch.cuda.synchronize()
    st = gmc.read_status(ws)
    traces = parity.parse_trace(tr.cpu().numpy(), L, B, K, 0, N)
    assert np.array_equal(Cd.cpu().numpy(), C.astype(np.float32)), "clients were written"
    return out.cpu().numpy().reshape(B, K), traces, st


def _check_select(C, K, **pk):
    from tests import parity
    idx, traces, st = _select_gpu(C, K, **pk)
    assert st == 0
    p = O.params(**{k: v for k, v in pk.items()})
    fails, ties = [], 0
    for b in range(C.shape[0]):
        C64 = C[b].astype(np.float32).astype(np.float64)
        sel = O.select_support(C64, K, p, forced=traces[b].forced_rounds())
        dec = parity.Decisions()
        parity.check_selection(sel, p["pool_mult"] * p["batch_b"], dec, f"img{b}")
        fails += dec.failures
        ties += len(dec.near_ties)
        assert np.array_equal(idx[b], sel.support)
        assert traces[b].K == K and traces[b].rounds == len(sel.rounds)
        fs = O.facility_value(C64, sel.support)
        assert abs(traces[b].F_S[0] - fs) <= 1e-5 * max(fs, 1e-30)
        # batched certificate Eq. (6) along the same rounds
        assert abs(traces[b].c_B - O.batched_certificate(sel)) <= 1e-4, (traces[b].c_B,
                                                                          O.batched_certificate(sel))
    assert not fails, "\n".join(fails[:10])
    return idx, traces, ties


def _structured_clients(B, M, N, seed):
    r = np.random.default_rng(seed)
    C = r.exponential(size=(B, M, N)) * (r.uniform(size=(B, M, N)) < 0.3)
    C *= np.exp(3 * r.standard_normal((B, M, 1)))           # rows of very different mass
    return (C / C.sum(axis=(1, 2), keepdims=True)).astype(np.float32)


@pytest.mark.parametrize("B,M,N,K", [(1, 200, 150, 37), (3, 1000, 700, 140), (2, 3344, 1296, 257)])
def test_select_matches_oracle_on_identical_clients(B, M, N, K):
    _check_select(_structured_clients(B, M, N, 7 + B), K)


def test_select_clients_of_a_real_boundary():
    """The oracle's own client matrix of the Qwen-shaped workload, in fp32."""
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("qwen", gh=18, gw=18, T=16)
    im = wl.image(0)
    f = lambda a: a.astype(np.float64)
    res = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos,
                     f(wl.probe()), wl.gh, wl.gw, 65)
    _check_select(res.clients.C[None].astype(np.float32), 65)


def test_select_zero_gain_fill_and_small_batches():
    # identical columns: one responsibility round, then an ascending fill
    col = np.random.default_rng(3).exponential(size=(40, 1)).astype(np.float32)
    C = np.repeat(col, 50, axis=1)[None]
    idx, tr, _ = _check_select(C, 30)
    assert idx[0].tolist() == list(range(30)) and tr[0].filled == 14
    # all-zero clients: the whole budget is filled in index order
    idx, tr, _ = _check_select(np.zeros((1, 10, 20), np.float32), 7)
    assert idx[0].tolist() == list(range(7)) and tr[0].rounds == 1
    # fewer positive gains than b: a short round, then the fill
    C = np.zeros((1, 6, 30), np.float32)
    C[0, np.arange(6), [2, 5, 9, 11, 20, 29]] = 1.0
    idx, tr, _ = _check_select(C, 10)
    assert set([2, 5, 9, 11, 20, 29]) <= set(idx[0].tolist())


def test_select_parameters_b1_and_k_equals_n():
    C = _structured_clients(1, 80, 60, 11)
    _check_select(C, 12, batch_b=1, pool_mult=4)
    _check_select(C, 60)


def test_select_beyond_the_cluster_runs_on_the_whole_gpu():
    """N = GMC_MAX_N with 4,800 client rows and a 128-token pool: the cluster
    solver's per-CTA state (a copy per token, 1/16 of the rows) exceeds a
    CTA's 227 KB, so every round runs on the whole GPU (4 launches a round,
    then the final one; the prep kernels and the certificate besides)."""
    from paper_2608_02134_gb300 import gmc
    B, M, N, K, b = 1, 4800, 8192, 600, 32
    n0 = gmc.launch_count()
    _check_select(_structured_clients(B, M, N, 91), K, batch_b=b)
    assert gmc.launch_count() - n0 == 3 + 4 * (-(-K // b)) + 1 + 1


def test_transport_with_oracle_decisions():
    from paper_2608_02134_gb300 import gmc, workloads
    from tests import gpu_harness as GH, parity
    wl = workloads.make("qwen", gh=12, gw=12, T=10, D=256, H=4, Hkv=2, K=25)
    im = wl.image(0)
    f = lambda a: a.astype(np.float64)
    res = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos, f(wl.probe()),
                     wl.gh, wl.gw, wl.K)
    inp = GH.to_device(wl)
    K, N, T = res.K, wl.N, wl.T[0]
    prob = gmc.problem(1, wl.gh, wl.gw, wl.Hkv, gmc.GMC_BF16)
    p = gmc.default_params()
    ws = gmc.alloc_workspace(gmc.transport_workspace_size(prob, N, T, K))
    sup = torch.tensor(res.support, dtype=torch.int32, device="cuda")
    pi = torch.tensor(res.assignment.pi, dtype=torch.int32, device="cuda")
    m = torch.tensor(res.m, dtype=torch.float32, device="cuda")
    oi = torch.empty(K, dtype=torch.int32, device="cuda")
    oh = torch.empty((K + T, wl.D), dtype=torch.bfloat16, device="cuda")
    okv = torch.empty((2 * (K + T), wl.Hkv, wl.d), dtype=torch.bfloat16, device="cuda")
    op = torch.empty(3 * (K + T), dtype=torch.int32, device="cuda")
    gmc.transport(prob, p, inp["hidden"], inp["keys"], inp["pos_ids"], sup, pi, m, N, T, wl.d,
                  wl.D, K, oi, oh, okv, op, ws)
    torch.cuda.synchronize()
    assert gmc.read_status(ws) == 0
    assert np.array_equal(oi.cpu().numpy(), res.support)
    hid = oh.float().cpu().numpy().astype(np.float64)
    assert parity.rel_row_err(hid[:K], res.out_hidden[:K]) < 2e-2
    # bf16 rounding is the only loss: within one bf16 ulp of the fp64 value
    ref = res.out_hidden[:K]
    assert np.all(np.abs(hid[:K] - ref) <= np.abs(ref) * 2 ** -8 + 1e-6)
    assert np.array_equal(hid[K:], f(im.hidden[N:]))
    assert np.array_equal(okv.float().cpu().numpy().reshape(2, K + T, wl.Hkv, wl.d), res.out_kv)
    assert np.array_equal(op.cpu().numpy().reshape(3, K + T), res.out_pos)
