"""CPU tests of the C-ABI library: it builds, loads without a GPU, exports every
entry point include/gmc.h declares, and its host-side logic (defaults, sizing,
argument validation) behaves as documented.  No compute call is made."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def gmc():
    from paper_2608_02134_gb300 import build
    build.build()
    from paper_2608_02134_gb300 import gmc as g
    g.lib()
    return g


def declared_functions():
    src = open(os.path.join(ROOT, "include", "gmc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gmc_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(gmc):
    names = declared_functions()
    assert len(names) >= 12
    L = ctypes.CDLL(gmc.LIB_PATH)
    for n in names:
        assert hasattr(L, n), f"{n} declared in include/gmc.h but not exported"
    assert set(names) == set(gmc.EXPORTS)


def test_defaults_are_the_papers_configuration(gmc):
    """Table "Shared GMC configuration" (fixed-token settings)."""
    p = gmc.default_params()
    assert (p.batch_b, p.pool_mult, p.landmarks, p.max_head_clusters) == (16, 4, 16, 4)
    vals = dict(resp_temp=0.1, tau_v=0.2, tau_s=0.02, beta_V=0.5, beta_S=0.25, lambda_mass=1.0,
                eps_mass=1e-8, assign_spatial_w=0.5, gate_scale=0.08, gate_pow=8.0,
                ambig_margin=0.05, pop_strength=0.5, terminal_q_weight=2.0, head_eps=0.05)
    for k, v in vals.items():
        assert getattr(p, k) == pytest.approx(v, rel=1e-6), k
    assert p.check_mode == 0
    assert gmc.version().startswith("gmc ")


def test_struct_sizes_match_header(gmc):
    # 23 four-byte fields / 6 fields with one pointer
    assert ctypes.sizeof(gmc.Params) == 23 * 4
    assert ctypes.sizeof(gmc.TraceHeader) == 64


def test_workspace_and_trace_sizing(gmc):
    pr = gmc.problem(1, 36, 36, 4, gmc.GMC_BF16)
    ws = gmc.workspace_size(pr, 1296, 64, 28, 128, 3584, 257)
    # it holds at least the client matrix and the attention slice
    M = 28 * 64 + 1296 + 256
    assert ws >= M * 1296 * 4 + 28 * 64 * 1296 * 4
    pr32 = gmc.problem(32, 36, 36, 4, gmc.GMC_BF16)
    assert gmc.workspace_size(pr32, 1296, 64, 28, 128, 3584, 257) > 31 * ws
    assert gmc.workspace_size(gmc.problem(1, 36, 35, 4, 1), 1296, 64, 28, 128, 3584, 257) == 0
    assert gmc.workspace_size(pr, 1296, 64, 30, 128, 3584, 257) == 0      # H % Hkv != 0
    # head statistics of one token block must fit shared memory: H <= 56
    assert gmc.workspace_size(pr, 1296, 64, 56, 128, 3584, 257) > 0
    assert gmc.workspace_size(pr, 1296, 64, 60, 128, 3584, 257) == 0
    L = gmc.trace_layout(pr, gmc.default_params(), 1296, 64, 28, 257)
    assert L.rounds_max == 17 + 1 and L.pool_size == 64
    assert L.off_order >= 64 and L.bytes_per_image % 16 == 0
    assert L.off_mass + 4 * 1296 <= L.bytes_per_image
    assert gmc.lib().gmc_trace_size(ctypes.byref(pr32), None, 1296, 64, 28, 257) == 32 * L.bytes_per_image


def _compress_rc(gmc, prob=None, ws_bytes=1 << 40, null=None, params=None, **shape):
    lib = gmc.lib()
    sh = dict(N=64, T=8, H=4, d=64, D=256, K=16)
    sh.update(shape)
    prob = prob or gmc.problem(1, 8, 8, 4, gmc.GMC_F32)
    fake = ctypes.c_void_p(1 << 20)    # aligned, never dereferenced: validation fails first
    ptrs = [fake] * 9
    if null is not None:
        ptrs[null] = None
    h, k, q, pos, w, oi, oh, okv, op = ptrs
    return lib.gmc_compress(ctypes.byref(prob), params, h, k, q, pos, w, sh["N"], sh["T"], sh["H"],
                            sh["d"], sh["D"], sh["K"], oi, oh, okv, op, fake, ws_bytes, None, None)


def test_argument_validation(gmc):
    assert _compress_rc(gmc, null=0) == gmc.GMC_ERR_ARG
    assert _compress_rc(gmc, null=6) == gmc.GMC_ERR_ARG
    assert _compress_rc(gmc, N=63) == gmc.GMC_ERR_ARG                     # N != grid_h*grid_w
    assert _compress_rc(gmc, H=6) == gmc.GMC_ERR_ARG                      # H % Hkv
    assert _compress_rc(gmc, T=0) == gmc.GMC_ERR_ARG
    assert _compress_rc(gmc, H=128, prob=gmc.problem(1, 8, 8, 4, 0)) == gmc.GMC_ERR_UNSUPPORTED
    assert _compress_rc(gmc, H=60, prob=gmc.problem(1, 8, 8, 4, 0)) == gmc.GMC_ERR_UNSUPPORTED
    assert _compress_rc(gmc, D=250) == gmc.GMC_ERR_UNSUPPORTED           # D % 8
    assert _compress_rc(gmc, ws_bytes=1024) == gmc.GMC_ERR_WORKSPACE
    bad = gmc.default_params(batch_b=64, pool_mult=4)                    # pool 256 > GMC_MAX_POOL
    assert _compress_rc(gmc, params=ctypes.byref(bad)) == gmc.GMC_ERR_ARG
    assert _compress_rc(gmc, prob=gmc.problem(1, 8, 8, 4, 7)) == gmc.GMC_ERR_ARG   # dtype
    assert "WORKSPACE" in gmc.lib().gmc_error_string(gmc.GMC_ERR_WORKSPACE).decode()


def test_select_and_transport_validation(gmc):
    lib = gmc.lib()
    fake = ctypes.c_void_p(1 << 20)
    p = gmc.default_params()
    assert lib.gmc_select(fake, 1, 10, 20, 25, ctypes.byref(p), fake, fake, 1 << 30, None, None) \
        == gmc.GMC_ERR_ARG                                                 # K > N
    assert lib.gmc_select(fake, 1, 10, 20, 5, ctypes.byref(p), fake, fake, 16, None, None) \
        == gmc.GMC_ERR_WORKSPACE
    assert gmc.select_workspace_size(1, 10, 20, 5, p) >= 10 * 20 * 6
    pr = gmc.problem(1, 4, 5, 1, gmc.GMC_F32)
    assert gmc.transport_workspace_size(pr, 20, 3, 5) > 0
    assert lib.gmc_transport(ctypes.byref(pr), None, fake, fake, fake, fake, fake, fake, 20, 3, 8,
                             16, 0, fake, fake, fake, fake, fake, 1 << 30, None) == gmc.GMC_ERR_ARG
    assert lib.gmc_read_status(None, None, None) == gmc.GMC_ERR_ARG


def test_binding_raises_without_the_library(gmc, monkeypatch, tmp_path):
    """No fallback: a missing libgmc.so is an error, not a silent CPU path."""
    monkeypatch.setattr(gmc, "_lib", None)
    monkeypatch.setattr(gmc, "LIB_PATH", str(tmp_path / "libgmc.so"))
    with pytest.raises(RuntimeError, match="missing"):
        gmc.lib()


def _long_rc(gmc, prob, lp, params=None, ws_bytes=1 << 40, **shape):
    lib = gmc.lib()
    sh = dict(N=1600, T=16, H=4, d=64, D=256, K=320)
    sh.update(shape)
    fake = ctypes.c_void_p(1 << 20)
    return lib.gmc_compress_long(ctypes.byref(prob), params, ctypes.byref(lp) if lp else None,
                                 None, None, fake, fake, fake, fake, fake, sh["N"], sh["T"],
                                 sh["H"], sh["d"], sh["D"], sh["K"], fake, fake, fake, fake,
                                 fake, ws_bytes, None, None)


def test_long_prefix_sizing_and_validation(gmc):
    """gmc_compress_long: the bounded bank's limits (bf16, one image, N >= 256,
    rank a multiple of 8 up to GMC_MAX_RANK, N up to GMC_MAX_N_LONG, pools up
    to GMC_MAX_POOL_WIDE)."""
    assert ctypes.sizeof(gmc.LongPrefix) == 16
    lp = gmc.LongPrefix(128, 4096, 1 << 20)
    pr = gmc.problem(1, 126, 126, 4, gmc.GMC_BF16)
    p = gmc.default_params(batch_b=512)
    N = 126 * 126
    ws = gmc.workspace_size_long(pr, p, lp, 0, N, 128, 28, 128, 3584, 4096)
    # the client matrix with M_V = 4096 appearance rows, and the N x K support cosines
    M = 28 * 128 + 4096 + 256
    assert ws >= M * N * 4 + N * 4096 * 4
    # no N x N cosine matrix: far below what the exact bank would need
    assert ws < M * N * 6 + N * N * 4
    assert gmc.workspace_size_long(pr, gmc.default_params(), lp, 0, N, 128, 28, 128, 3584,
                                   4096) > 0
    assert gmc.workspace_size_long(pr, p, lp, 0, N, 128, 28, 128, 3584, 4096) > \
        gmc.workspace_size_long(pr, gmc.default_params(), lp, 0, N, 128, 28, 128, 3584, 4096)
    small = gmc.problem(1, 40, 40, 2, gmc.GMC_BF16)
    lps = gmc.LongPrefix(128, 512, 1 << 20)
    p64 = gmc.default_params(batch_b=64)
    assert _long_rc(gmc, small, lps, ctypes.byref(p64), ws_bytes=1024) == gmc.GMC_ERR_WORKSPACE
    assert _long_rc(gmc, small, None, ctypes.byref(p64)) == gmc.GMC_ERR_ARG
    assert _long_rc(gmc, small, gmc.LongPrefix(12, 512, 1 << 20), ctypes.byref(p64)) == gmc.GMC_ERR_ARG
    assert _long_rc(gmc, small, gmc.LongPrefix(128, 0, 1 << 20), ctypes.byref(p64)) == gmc.GMC_ERR_ARG
    assert _long_rc(gmc, small, gmc.LongPrefix(128, 512, 0), ctypes.byref(p64)) == gmc.GMC_ERR_ARG
    assert _long_rc(gmc, small, gmc.LongPrefix(264, 512, 1 << 20), ctypes.byref(p64)) == \
        gmc.GMC_ERR_UNSUPPORTED                                             # rank > 256
    assert _long_rc(gmc, gmc.problem(1, 40, 40, 2, gmc.GMC_F32), lps, ctypes.byref(p64)) == \
        gmc.GMC_ERR_UNSUPPORTED                                             # bf16 only
    assert _long_rc(gmc, gmc.problem(1, 8, 8, 2, gmc.GMC_BF16), lps, ctypes.byref(p64),
                    N=64) == gmc.GMC_ERR_UNSUPPORTED                        # N < 256
    assert _long_rc(gmc, gmc.problem(1, 12, 20, 2, gmc.GMC_BF16), lps, ctypes.byref(p64),
                    N=240) == gmc.GMC_ERR_UNSUPPORTED
    assert _long_rc(gmc, gmc.problem(1, 40, 40, 2, gmc.GMC_BF16, images=2), lps,
                    ctypes.byref(p64), N=3200) == gmc.GMC_ERR_UNSUPPORTED   # one image
    assert _long_rc(gmc, gmc.problem(1, 130, 130, 2, gmc.GMC_BF16), lps, ctypes.byref(p64),
                    N=16900) == gmc.GMC_ERR_UNSUPPORTED                     # N > 16384
    big = gmc.default_params(batch_b=2048, pool_mult=4)                     # pool 8192 > 4096
    assert _long_rc(gmc, small, lps, ctypes.byref(big)) == gmc.GMC_ERR_ARG
    # the standard entry point keeps its limits
    assert _compress_rc(gmc, prob=pr, N=N, T=128, H=28, d=128, D=3584, K=4096) == \
        gmc.GMC_ERR_UNSUPPORTED
    # gmc_select accepts wide pools (every round on the whole GPU) and longer N with them
    assert gmc.select_workspace_size(1, 500, 12000, 1500, p) > 500 * 12000 * 6
    assert gmc.select_workspace_size(1, 500, 12000, 1500, gmc.default_params()) == 0


def test_host_io_struct_and_validation(gmc):
    """gmc_host_io: 9 (pointer, pointer, size) triples; nothing is copied when an
    argument is missing or the problem is invalid."""
    assert ctypes.sizeof(gmc.HostIO) == 9 * 3 * 8
    lib = gmc.lib()
    pr = gmc.problem(1, 36, 36, 4, gmc.GMC_BF16)
    p = gmc.default_params()
    fake = ctypes.c_void_p(1 << 20)
    assert lib.gmc_compress_host(ctypes.byref(pr), ctypes.byref(p), None, 1296, 64, 28, 128, 3584,
                                 257, fake, 1 << 30, None, None) == gmc.GMC_ERR_ARG
    io = gmc.HostIO()
    assert lib.gmc_compress_host(ctypes.byref(pr), ctypes.byref(p), ctypes.byref(io), 1296, 64, 28,
                                 128, 3584, 257, fake, 1 << 30, None, None) == gmc.GMC_ERR_ARG
    for name, _ in gmc.HostIO._fields_:  # every pointer and size set: the problem decides
        setattr(io, name, 1 << 20)
    assert lib.gmc_compress_host(ctypes.byref(pr), ctypes.byref(p), ctypes.byref(io), 1295, 64, 28,
                                 128, 3584, 257, fake, 1 << 30, None, None) == gmc.GMC_ERR_ARG
