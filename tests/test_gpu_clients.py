"""GPU client matrix against the oracle, element by element (gmc_clients).

gmc_clients stops the path after the client build, so the message slice
(Eq. (cond-native-message)), the probe values and mass coordinate (Eq. (1)),
the grounded clients (Eq. (2)), the head and query weights (Eq.
(cond-head-weight)), the cosines and the appearance and spatial banks (Eq.
(cond-aux-clients), (cond-coverage)) are all compared entry by entry with
the oracle's fp64 client matrix, which follows the GPU's head clustering
(checked separately against the oracle's fp64 pattern cosines).  Bar: every
row within a max relative error of 1e-3 of its largest entry, for bf16 inputs
with fp32 arithmetic as for fp32 inputs.
"""

import numpy as np
import pytest
import torch

from oracle import gmc_oracle as O

pytestmark = pytest.mark.gpu

ROW_TOL = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _gpu_clients(wl, n_hist=0):
    from paper_2608_02134_gb300 import gmc
    from tests import gpu_harness as GH, parity
    dt = gmc.GMC_BF16 if wl.dtype == "bf16" else gmc.GMC_F32
    inp = GH.to_device(wl)
    comp = gmc.Compressor(wl.B, wl.gh, wl.gw, wl.T_max, wl.H, wl.Hkv, wl.d, wl.D, wl.K, dt,
                          text_lengths=wl.T if wl.ragged else None, trace=True, n_views=n_hist)
    vw = None
    if n_hist:
        hv = [wl.history_abi_arrays(v) for v in range(n_hist)]
        vw = gmc.views([GH._dev(h["keys"]) for h in hv], [GH._dev(h["queries"]) for h in hv],
                       [GH._dev(h["vo_probe"]) for h in hv])
    M = (1 + n_hist) * wl.H * wl.T_max + wl.N + comp.params.landmarks ** 2
    out = torch.full((wl.B, M, wl.N), float("nan"), dtype=torch.float32, device="cuda")
    gmc.clients(comp.prob, comp.params, vw, inp["hidden"], inp["keys"], inp["queries"],
                inp["pos_ids"], inp["vo_probe"], wl.N, wl.T_max, wl.H, wl.d, wl.D, wl.K, out,
                comp.workspace, comp.trace)
    torch.cuda.synchronize()
    assert comp.status() == 0
    traces = parity.parse_trace(comp.trace.cpu().numpy(), comp.layout, wl.B, comp.K, wl.H, wl.N,
                                comp.params.max_head_clusters)
    return out.cpu().numpy().astype(np.float64), traces, comp


def _compare(wl, images, n_hist=0):
    from tests import gpu_harness as GH, parity
    C, traces, comp = _gpu_clients(wl, n_hist)
    p = GH.oracle_params(comp.params)
    f = lambda a: np.asarray(a, dtype=np.float64)
    worst = 0.0
    for b in images:
        im = wl.image(b)
        tr = traces[b]
        nc = min(p["max_head_clusters"], wl.H)
        forced = dict(centres=tr.centres[:nc].tolist(), head_assign=tr.head_assign.tolist())
        history = None
        if n_hist:
            history = [{k: f(a) for k, a in wl.history_view(b, v).items()} for v in range(n_hist)]
        res = O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos,
                         f(wl.probe()), wl.gh, wl.gw, wl.K, p, forced=forced, history=history)
        dec = parity.Decisions()
        parity.check_heads(res.heads, dec, f"{wl.name}[b={b}]")
        assert not dec.failures, dec.failures
        ref = res.clients.C
        got = C[b, :ref.shape[0]]
        assert np.all(np.isfinite(got))
        err = parity.rel_row_err(got, ref)
        worst = max(worst, err)
        assert err <= ROW_TOL, f"image {b}: client rows max rel err {err:.3e}"
        # bank masses (rows of each bank add up to its beta)
        assert abs(got.sum() - ref.sum()) <= 1e-5 * ref.sum()
    print(f"{wl.name}: worst client row error {worst:.2e}")


def test_clients_tiny_fp32():
    from paper_2608_02134_gb300 import workloads
    _compare(workloads.make("tiny"), [0])


def test_clients_qwen_shape():
    from paper_2608_02134_gb300 import workloads
    _compare(workloads.make("qwen"), [0])


def test_clients_llava_shape():
    from paper_2608_02134_gb300 import workloads
    _compare(workloads.make("llava", K=128), [0])


def test_clients_ragged_batch_and_views():
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make("qwen", B=3, T=[20, 7, 33], gh=12, gw=12, D=64, H=8, Hkv=2, K=30)
    _compare(wl, [0, 1, 2])
    _compare(wl, [0, 2], n_hist=2)
