"""GPU parity of the long-prefix path (gmc_compress_long) and the wide solver.

Long prefixes use the bounded appearance bank (appendix "Appearance and
spatial clients", last paragraph; Table "Shared GMC configuration", long-prefix
row: a rank-128 Rademacher projection, at most M_V uniformly spaced appearance
clients, b = 512) and the N x K support cosines for the assignment.  Checked
here:
  * the wide solver (every round on the whole GPU, pools above 128) on the very
    same fp32 client matrix as the oracle, like the standard solver;
  * the client matrix with the bounded bank, entry by entry;
  * the whole step on the small long-prefix workload (N = 1600, pool 256)
    against the forced oracle: every decision, the transported rows, the
    bit-exact gathers and the bank values;
  * the paper's long-prefix shape (N = 15,876, K = 4,096, b = 512) at full
    size, on sampled outputs the oracle computes one by one: appearance client
    rows, assignments, transported carriers, and the bit-exact text, K/V and
    position rows.
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


# ---------------------------------------------------------------------------
# wide solver on identical clients
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("B,M,N,K,b", [(1, 300, 700, 140, 64), (2, 3344, 1296, 257, 64),
                                       (1, 800, 4096, 1024, 256), (1, 500, 12000, 1500, 512)])
def test_wide_select_matches_oracle_on_identical_clients(B, M, N, K, b):
    from tests.test_gpu_stages import _check_select, _structured_clients
    _check_select(_structured_clients(B, M, N, 40 + B + b), K, batch_b=b)


def test_wide_select_fill_and_short_rounds():
    from tests.test_gpu_stages import _check_select
    # identical columns: one responsibility round, then an ascending fill
    col = np.random.default_rng(5).exponential(size=(40, 1)).astype(np.float32)
    C = np.repeat(col, 600, axis=1)[None]
    idx, tr, _ = _check_select(C, 300, batch_b=64)
    assert idx[0].tolist() == list(range(300)) and tr[0].filled == 300 - 64
    # all-zero clients: the whole budget is filled in index order
    idx, tr, _ = _check_select(np.zeros((1, 10, 400), np.float32), 150, batch_b=64)
    assert idx[0].tolist() == list(range(150)) and tr[0].rounds == 1
    # fewer positive gains than b: a short round, then the fill
    C = np.zeros((1, 6, 300), np.float32)
    C[0, np.arange(6), [2, 5, 90, 111, 200, 299]] = 1.0
    idx, tr, _ = _check_select(C, 100, batch_b=64)
    assert {2, 5, 90, 111, 200, 299} <= set(idx[0].tolist())


# ---------------------------------------------------------------------------
# the bounded bank's client matrix, entry by entry
# ---------------------------------------------------------------------------
def _long_inputs(wl):
    from paper_2608_02134_gb300 import gmc
    from tests import gpu_harness as GH
    lpo, b = GH.long_prefix_of(wl)
    R = torch.from_numpy(lpo["R"]).to(torch.bfloat16).cuda()
    lp = gmc.long_prefix(R, lpo["max_clients"])
    lp._keep = R
    return lpo, lp, gmc.default_params(batch_b=b)


def _gpu_long_clients(wl):
    from paper_2608_02134_gb300 import gmc
    from tests import gpu_harness as GH, parity
    lpo, lp, params = _long_inputs(wl)
    inp = GH.to_device(wl)
    comp = gmc.Compressor(wl.B, wl.gh, wl.gw, wl.T_max, wl.H, wl.Hkv, wl.d, wl.D, wl.K,
                          gmc.GMC_BF16, text_lengths=wl.T if wl.ragged else None, params=params,
                          trace=True, long_prefix=lp)
    MV = min(wl.N, lpo["max_clients"])
    M = wl.H * wl.T_max + MV + params.landmarks ** 2
    out = torch.full((wl.B, M, wl.N), float("nan"), dtype=torch.float32, device="cuda")
    gmc.clients_long(comp.prob, comp.params, lp, None, inp["hidden"], inp["keys"], inp["queries"],
                     inp["pos_ids"], inp["vo_probe"], wl.N, wl.T_max, wl.H, wl.d, wl.D, wl.K, out,
                     comp.workspace, comp.trace)
    torch.cuda.synchronize()
    assert comp.status() == 0
    traces = parity.parse_trace(comp.trace.cpu().numpy(), comp.layout, wl.B, comp.K, wl.H, wl.N,
                                comp.params.max_head_clusters)
    return out, traces, comp, lpo


def test_long_clients_match_oracle_entrywise():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH, parity
    wl = workloads.make("longsmall")
    out, traces, comp, lpo = _gpu_long_clients(wl)
    C = out.cpu().numpy().astype(np.float64)
    p = GH.oracle_params(comp.params)
    f = lambda a: np.asarray(a, dtype=np.float64)
    im = wl.image(0)
    tr = traces[0]
    nc = min(p["max_head_clusters"], wl.H)
    forced = dict(centres=tr.centres[:nc].tolist(), head_assign=tr.head_assign.tolist())
    res = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos, f(wl.probe()),
                     wl.gh, wl.gw, wl.K, p, forced=forced, long_prefix=lpo)
    ref = res.clients.C
    got = C[0, :ref.shape[0]]
    assert ref.shape[0] == wl.H * wl.T_max + lpo["max_clients"] + 256
    assert np.all(np.isfinite(got))
    err = parity.rel_row_err(got, ref)
    app = res.clients.banks["appearance"]
    err_app = parity.rel_row_err(got[app], ref[app])
    print(f"longsmall: client rows max rel err {err:.2e} (appearance bank {err_app:.2e})")
    assert err <= 1e-3
    # the split bf16 product keeps the projected cosines near fp32 accuracy
    assert err_app <= 1e-4
    assert abs(got.sum() - ref.sum()) <= 1e-5 * ref.sum()


# ---------------------------------------------------------------------------
# the whole step against the forced oracle
# ---------------------------------------------------------------------------
def _parity(wl, images, tol=2e-2):
    from tests import gpu_harness as GH
    g = GH.run(wl)
    assert g.status == 0, hex(g.status)
    fails, ties, checked = [], 0, 0
    for b in images:
        rep = GH.compare_image(g, b, tol)
        fails += rep.dec.failures
        ties += len(rep.dec.near_ties)
        checked += rep.dec.checked
    assert not fails, "\n".join(fails[:10])
    print(f"{wl.name}: {checked} decisions checked, {ties} near-ties followed")
    return g


def test_long_small_parity():
    from paper_2608_02134_gb300 import workloads
    g = _parity(workloads.make("longsmall"), [0])
    tr = g.traces[0]
    assert tr.K == 320 and tr.rounds >= 5
    assert g.comp.layout.pool_size == 256


def test_long_small_ragged_batch():
    from paper_2608_02134_gb300 import workloads
    _parity(workloads.make("longsmall", B=3, T=[16, 5, 11]), [0, 1, 2])


def test_long_small_budget_edges():
    from paper_2608_02134_gb300 import workloads
    _parity(workloads.make("longsmall", K=64), [0])    # one round of b = 64
    _parity(workloads.make("longsmall", K=1), [0])     # a single carrier
    # K = N returns the input unchanged
    from tests import gpu_harness as GH
    wl = workloads.make("longsmall", K=5000)
    g = GH.run(wl, trace=False)
    assert g.status == 0
    inp = wl.image(0)
    assert np.array_equal(g.idx, np.arange(wl.N))
    assert np.array_equal(g.hidden, inp.hidden.astype(np.float64))


# ---------------------------------------------------------------------------
# the paper's long-prefix shape at full size, on sampled outputs
# ---------------------------------------------------------------------------
def test_long_doc_full_size_sampled():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH, parity
    wl = workloads.make("longdoc")
    N, T, K, D = wl.N, wl.T_max, wl.K, wl.D
    g = GH.run(wl)
    assert g.status == 0, hex(g.status)
    tr = g.traces[0]
    idx = g.idx
    assert idx.size == K and np.all(np.diff(idx) > 0) and idx[0] >= 0 and idx[-1] < N
    assert tr.K == K and tr.rounds <= -(-K // 512) + 1
    im = wl.image(0)
    f = lambda a: np.asarray(a, dtype=np.float64)
    hid = f(im.hidden)
    hvis = hid[:N]
    # bit-exact gathers: text rows, compact K/V and position ids at the kept rows
    rows = np.concatenate([idx, N + np.arange(T)])
    assert np.array_equal(g.hidden[K:], hid[N:])
    kv = g.kv.reshape(2, K + T, wl.Hkv, wl.d)
    assert np.array_equal(kv[0], f(im.keys)[rows]) and np.array_equal(kv[1], f(im.values)[rows])
    assert np.array_equal(g.pos.reshape(3, K + T), im.pos[:, rows])
    # the banks' values: F(S) <= F(V) per bank, and the bounded bank's F(V)
    for q in range(3):
        assert 0.0 < tr.F_S[q] <= tr.F_V[q] * (1 + 1e-5)
    rng = np.random.default_rng(0)
    p = GH.oracle_params(g.comp.params)
    xn = O.unit_states(hvis, p)
    # assignment of sampled discarded tokens: a valid argmax of kappa (Eq.
    # (cond-assignment)) at the GPU's separability gate, fp64 cosines
    inS = np.zeros(N, bool)
    inS[idx] = True
    disc = np.flatnonzero(~inS)
    P = O.grid_coords(wl.gh, wl.gw)
    for i in rng.choice(disc, size=48, replace=False):
        cs = xn[idx] @ xn[i]
        top = np.sort(cs)[::-1]
        delta = top[0] - top[1]
        gi = np.exp(-((delta / p["ambig_margin"]) ** p["gate_pow"]))
        d2 = np.sum((P[idx] - P[i]) ** 2, axis=1)
        kappa = cs + p["assign_spatial_w"] * tr.s_x * gi * np.exp(-d2 / p["tau_s"])
        got = kappa[np.searchsorted(idx, tr.pi[i])]
        assert tr.pi[i] in set(idx.tolist())
        assert got >= kappa.max() - parity.TOL * max(1.0, abs(kappa.max())), (i, got, kappa.max())
    # transported carriers from the GPU's assignment and weights, fp64 (Eq. (5))
    pi, m = tr.pi, tr.mass.astype(np.float64)
    for k in rng.choice(K, size=24, replace=False):
        j = idx[k]
        mem = np.flatnonzero(pi == j)
        assert j in mem
        c = (m[mem, None] * hvis[mem]).sum(axis=0) / m[mem].sum()
        want = c * O.rms(hvis[j]) / (O.rms(c) + p["rms_eps"])
        err = parity.rel_row_err(g.hidden[k][None], want[None])
        assert err < 2e-2, (k, err)
    # sampled appearance client rows of the bounded bank, against the oracle's
    # formula on those rows only (fp64 projected states of every token)
    out, _, comp, lpo = _gpu_long_clients(wl)
    xt = O.projected_states(hvis, f(lpo["R"]), p)
    ct = O.bounded_client_tokens(N, lpo["max_clients"])
    MV = ct.size
    a0 = wl.H * T
    for mrow in rng.choice(MV, size=8, replace=False):
        lg = (xt[ct[mrow]] @ xt.T) / p["tau_v"]
        e = np.exp(lg - lg.max())
        want = p["beta_V"] / MV * e / e.sum()
        got = out[0, a0 + mrow].cpu().numpy().astype(np.float64)
        assert parity.rel_row_err(got[None], want[None]) < 1e-4, mrow


def test_long_small_with_views_and_prefix_layers():
    """gmc_compress_long with a historical message view and two dense prefix
    layers: the view's grounded rows join the client matrix beside the bounded
    bank, and the prefix layers' K/V are gathered at the kept rows."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("longsmall")
    g = GH.run(wl, n_hist=1, n_prefix=2)
    assert g.status == 0, hex(g.status)
    rep = GH.compare_image(g, 0, 2e-2)
    assert not rep.dec.failures, "\n".join(rep.dec.failures[:10])
