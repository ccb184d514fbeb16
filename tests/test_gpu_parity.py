"""GPU parity: gmc_compress through the C-ABI against the fp64 oracle.

Bar (per image): every discrete choice is a valid choice of the oracle's
fp64 values within the relative margin 1e-4 (so the kept indices are
bit-exact wherever the margin exceeds it); transported rows within max
row-relative error 1e-3 (fp32 inputs) or 2e-2 (bf16 inputs, fp32
accumulation); text rows, compact K/V and position ids bit-exact.
"""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

TOL_F32, TOL_BF16 = 1e-3, 2e-2


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_02134_gb300 import gmc
    gmc.lib()


def _check(g, images, tol):
    from tests import gpu_harness as GH
    assert g.status == 0, f"device status {g.status:#x}"
    reports = [GH.compare_image(g, b, tol) for b in images]
    fails = [f for r in reports for f in r.dec.failures]
    ties = sum(len(r.dec.near_ties) for r in reports)
    checked = sum(r.dec.checked for r in reports)
    print(f"{g.wl.name}: {checked} decisions checked, {ties} near-ties followed, "
          f"max hidden err {max(r.hidden_err for r in reports):.2e}")
    assert not fails, "\n".join(fails[:20])
    return reports


def test_tiny_fp32():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("tiny")
    _check(GH.run(wl), [0], TOL_F32)


@pytest.mark.parametrize("K", [64, 128, 192])
def test_llava_shape(K):
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("llava", K=K)
    _check(GH.run(wl), [0], TOL_BF16)


def test_qwen_shape():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("qwen")
    _check(GH.run(wl), [0], TOL_BF16)


def test_document_shape():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("doc")
    _check(GH.run(wl), [0], TOL_BF16)


def test_largest_image():
    """N = GMC_MAX_N (a 128 x 64 page, K = 820): the cluster solver's state
    does not fit a CTA, so every selection round runs on the whole GPU; every
    decision is still checked against the oracle."""
    from paper_2608_02134_gb300 import gmc, workloads
    from tests import gpu_harness as GH
    wl = workloads.make("doc", gh=128, gw=64, K=820)
    assert wl.N == 8192  # GMC_MAX_N
    g = GH.run(wl)
    _check(g, [0], TOL_BF16)
    # the stages of a timed call: no cluster rounds
    inp = GH.to_device(wl)
    gmc.profile_enable(True)
    try:
        g.comp.run(inp["hidden"], inp["keys"], inp["queries"], inp["pos_ids"], inp["vo_probe"])
        torch.cuda.synchronize()
        stages = gmc.profile_read()
    finally:
        gmc.profile_enable(False)
    assert "select" in stages and "rounds_gpu" not in stages, sorted(stages)
    assert g.comp.status() == 0


def test_serving_batch_every_image():
    """32 ragged images in one call; the oracle checks every one of them."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("serving")
    g = GH.run(wl)
    _check(g, list(range(wl.B)), TOL_BF16)


@pytest.mark.parametrize("shape", [
    dict(gh=5, gw=7, H=3, Hkv=1, d=16, D=40, T=3, K=9),      # ragged tiles, GQA 3:1
    dict(gh=6, gw=6, H=2, Hkv=2, d=8, D=16, T=1, K=1),       # one text query, K = 1
    dict(gh=9, gw=11, H=8, Hkv=2, d=32, D=64, T=17, K=40),   # more heads than clusters
])
def test_small_shapes_fp32(shape):
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    K = shape.pop("K")
    T = shape.pop("T")
    wl = workloads.make("tiny", K=K, T=T, **shape)
    _check(GH.run(wl), [0], TOL_F32)


def test_small_shape_bf16_strong_gate():
    """Low hidden dimension spreads the cosines, so s_x > 0 and the spatial term acts."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("qwen", gh=12, gw=12, T=20, D=64, H=8, Hkv=2, K=30)
    g = GH.run(wl)
    reps = _check(g, [0], TOL_BF16)
    assert g.traces[0].s_x > 0.0


def test_identity_when_K_equals_N():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("tiny", K=64)
    g = GH.run(wl, trace=False)
    im = wl.image(0)
    assert np.array_equal(g.idx, np.arange(64))
    assert np.array_equal(g.hidden, im.hidden.astype(np.float64))
    assert np.array_equal(g.pos, im.pos.reshape(-1))
    wl2 = workloads.make("tiny", K=500)        # K_r > N clamps to N: identity
    g2 = GH.run(wl2, trace=False)
    assert np.array_equal(g2.hidden, im.hidden.astype(np.float64))


def test_deterministic_repeat():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("llava", K=128)
    inp = GH.to_device(wl)
    a = GH.run(wl, inputs=inp)
    b = GH.run(wl, inputs=inp)
    assert np.array_equal(a.idx, b.idx)
    assert np.array_equal(a.hidden_raw, b.hidden_raw)


def test_history_views_small_bf16():
    """Two completed historical message views (each with its own queries, keys, values, probe)."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("qwen", gh=12, gw=12, T=20, D=64, H=8, Hkv=2, K=30)
    _check(GH.run(wl, n_hist=2), [0], TOL_BF16)


def test_history_views_tiny_fp32_ragged_batch():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("tiny", B=2, T=[8, 5], K=16)
    _check(GH.run(wl, n_hist=1), [0, 1], TOL_F32)


def test_history_views_qwen_shape():
    """The deployed two-view setting (current view + two completed views) at the Qwen shape."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("qwen")
    _check(GH.run(wl, n_hist=2), [0], TOL_BF16)


def test_history_views_llava_shape():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("llava", K=128)
    _check(GH.run(wl, n_hist=2), [0], TOL_BF16)


@pytest.mark.parametrize("wlname,shape", [
    ("tiny", dict(H=1, Hkv=1)),
    ("qwen", dict(gh=12, gw=12, T=20, D=64, H=1, Hkv=1, K=30)),
])
def test_single_head(wlname, shape):
    """H = 1: one head cluster of weight 1."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    shape = dict(shape)
    K = shape.pop("K", None)
    T = shape.pop("T", None)
    wl = workloads.make(wlname, K=K, T=T, **shape)
    g = GH.run(wl)
    _check(g, [0], TOL_F32 if wl.dtype == "f32" else TOL_BF16)
    assert g.traces[0].n_clusters == 1 and abs(float(g.traces[0].omega[0]) - 1.0) < 1e-6


@pytest.mark.parametrize("resp_temp", [0.05, 0.02, 1.0])
def test_responsibility_temperature(resp_temp):
    """Temperatures away from the paper's 0.1 (the softmax is shifted by its row maximum)."""
    from paper_2608_02134_gb300 import gmc, workloads
    from tests import gpu_harness as GH
    wl = workloads.make("qwen", gh=18, gw=18, T=24, D=128, H=8, Hkv=2, K=60)
    g = GH.run(wl, params=gmc.default_params(resp_temp=resp_temp))
    _check(g, [0], TOL_BF16)


def test_prefix_layers_qwen_shape():
    """Cached path: two dense prefix layers gathered bit-exactly at the kept rows."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("qwen")
    _check(GH.run(wl, n_prefix=2), [0], TOL_BF16)


def test_prefix_layers_ragged_batch_with_views():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("qwen", B=3, T=[20, 7, 33], gh=12, gw=12, D=64, H=8, Hkv=2, K=30)
    _check(GH.run(wl, n_prefix=9, n_hist=2), [0, 1, 2], TOL_BF16)


def test_prefix_layers_fp32_and_identity():
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("tiny")
    _check(GH.run(wl, n_prefix=1), [0], TOL_F32)
    wl2 = workloads.make("tiny", K=64)                        # K = N: every layer unchanged
    g = GH.run(wl2, trace=False, n_prefix=3)
    for l in range(3):
        pk = wl2.prefix_kv(0, l)
        ref = np.stack([pk["K"], pk["V"]]).reshape(-1).astype(np.float64)
        assert np.array_equal(g.prefix[l].reshape(-1), ref)


def test_multi_image_prompt_qwen_shape():
    """Two Qwen-shaped images in one prompt: seeds, image-restricted banks, same-image clusters."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("multi")
    g = GH.run(wl)
    _check(g, [0], TOL_BF16)
    img = np.arange(wl.N) // wl.Ng
    pi = g.traces[0].pi
    assert np.all(img[pi] == img)


@pytest.mark.parametrize("I,K", [(3, 24), (4, 2)])
def test_multi_image_small_shapes(I, K):
    """Three and four images (K below the image count: one carrier each), ragged text, fp32 and bf16."""
    from paper_2608_02134_gb300 import workloads
    from tests import gpu_harness as GH
    wl = workloads.make("tiny", I=I, gh=6, gw=7, B=2, T=[5, 9], K=K)
    g = GH.run(wl)
    _check(g, [0, 1], TOL_F32)
    assert g.comp.K == max(K, I)
    wl2 = workloads.make("qwen", I=I, gh=8, gw=8, T=12, D=64, H=8, Hkv=2, K=K)
    _check(GH.run(wl2), [0], TOL_BF16)
