"""Device-detected conditions reach the status word, and the context stays usable.

Nothing here faults, traps or hangs the GPU: the non-finite input is made on
the host, and the wait that runs out is a bounded wait on a barrier phase
nothing completes (gmc_selftest_bounded_wait), given a limit of about a
millisecond.
"""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _small():
    from paper_2608_02134_gb300 import workloads
    return workloads.make("qwen", gh=12, gw=12, T=20, D=64, H=8, Hkv=2, K=30)


def test_nonfinite_hidden_state_is_reported_with_check_mode():
    from paper_2608_02134_gb300 import gmc
    from tests import gpu_harness as GH
    wl = _small()
    inp = GH.to_device(wl)
    inp["hidden"].view(-1)[5 * wl.D + 3] = float("nan")   # one visual state's entry, set from the host
    g = GH.run(wl, params=gmc.default_params(check_mode=1), trace=False, inputs=inp)
    assert g.status & gmc.STATUS_NONFINITE
    assert not g.status & gmc.STATUS_TIMEOUT
    # every output index is still a valid, sorted support
    assert np.all(np.diff(g.idx) > 0) and g.idx[0] >= 0 and g.idx[-1] < wl.N
    # the next call on clean inputs runs normally
    g2 = GH.run(wl, trace=False)
    assert g2.status == 0


def test_check_mode_off_leaves_clean_status():
    from paper_2608_02134_gb300 import gmc
    from tests import gpu_harness as GH
    g = GH.run(_small(), params=gmc.default_params(check_mode=1), trace=False)
    assert g.status == 0


def test_bounded_wait_runs_out_and_reports_timeout():
    from paper_2608_02134_gb300 import gmc
    from tests import gpu_harness as GH
    ws = gmc.alloc_workspace(256)
    gmc.selftest_bounded_wait(2_000_000, ws)    # about 1 ms of SM clocks
    assert gmc.read_status(ws) == gmc.STATUS_TIMEOUT
    gmc.selftest_bounded_wait(0, ws)            # a limit already passed: gives up at once
    assert gmc.read_status(ws) == gmc.STATUS_TIMEOUT
    # the context is still usable afterwards
    g = GH.run(_small(), trace=False)
    assert g.status == 0
