"""Python binding of libgmc.so: the same entry points as include/gmc.h.

Argument marshalling only: every step of the compression runs in the CUDA
library.  Tensors are torch tensors (device memory, or pinned host memory for
the staged host path); the library is loaded on first use and a missing or
unloadable build raises -- there is no fallback.
"""

from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass, fields

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libgmc.so")

GMC_OK, GMC_ERR_ARG, GMC_ERR_UNSUPPORTED, GMC_ERR_WORKSPACE, GMC_ERR_CUDA = range(5)
GMC_F32, GMC_BF16 = 0, 1
STATUS_NONFINITE, STATUS_TIMEOUT, STATUS_TEXT_LEN, STATUS_INTERNAL = 0x1, 0x2, 0x4, 0x8

EXPORTS = (
    "gmc_default_params", "gmc_workspace_size", "gmc_compress", "gmc_get_trace_layout",
    "gmc_trace_size", "gmc_select_workspace_size", "gmc_select",
    "gmc_transport_workspace_size", "gmc_transport", "gmc_read_status", "gmc_error_string",
    "gmc_version", "gmc_profile_enable", "gmc_profile_read", "gmc_launch_count",
    "gmc_transport_noalloc", "gmc_cosine_workspace_size", "gmc_cosine",
    "gmc_workspace_size_views", "gmc_compress_views", "gmc_clients", "gmc_selftest_bounded_wait",
    "gmc_compress_ex", "gmc_workspace_size_long", "gmc_compress_long", "gmc_clients_long",
    "gmc_compress_host",
)
MAX_VIEWS = 4
MAX_PREFIX_LAYERS = 64


class HostIO(ctypes.Structure):
    """gmc_host_io: (host, device, bytes) for every input, (device, host, bytes) for every output."""
    _fields_ = ([f for n in ("hidden", "keys", "queries", "pos_ids", "vo_probe")
                 for f in ((n, ctypes.c_void_p), ("d_" + n, ctypes.c_void_p),
                           (n + "_bytes", ctypes.c_size_t))] +
                [f for n in ("out_idx", "out_hidden", "out_kv", "out_pos")
                 for f in (("d_" + n, ctypes.c_void_p), (n, ctypes.c_void_p),
                           (n + "_bytes", ctypes.c_size_t))])


class Params(ctypes.Structure):
    _fields_ = [
        ("batch_b", ctypes.c_int), ("pool_mult", ctypes.c_int),
        ("resp_temp", ctypes.c_float), ("resp_eps", ctypes.c_float),
        ("tau_v", ctypes.c_float), ("tau_s", ctypes.c_float),
        ("beta_G", ctypes.c_float), ("beta_V", ctypes.c_float), ("beta_S", ctypes.c_float),
        ("landmarks", ctypes.c_int), ("max_head_clusters", ctypes.c_int),
        ("head_eps", ctypes.c_float), ("terminal_q_weight", ctypes.c_float),
        ("lambda_mass", ctypes.c_float), ("eps_mass", ctypes.c_float),
        ("assign_spatial_w", ctypes.c_float), ("gate_scale", ctypes.c_float),
        ("gate_pow", ctypes.c_float), ("ambig_margin", ctypes.c_float),
        ("pop_strength", ctypes.c_float), ("rms_eps", ctypes.c_float),
        ("norm_eps", ctypes.c_float), ("check_mode", ctypes.c_int),
    ]


class Problem(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("grid_h", ctypes.c_int), ("grid_w", ctypes.c_int),
                ("Hkv", ctypes.c_int), ("dtype", ctypes.c_int), ("text_offsets", ctypes.c_void_p),
                ("images", ctypes.c_int)]


class Views(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int), ("beta_hist", ctypes.c_float),
                ("keys", ctypes.c_void_p * (MAX_VIEWS - 1)),
                ("queries", ctypes.c_void_p * (MAX_VIEWS - 1)),
                ("vo_probe", ctypes.c_void_p * (MAX_VIEWS - 1))]


class PrefixKV(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int),
                ("keys", ctypes.c_void_p * MAX_PREFIX_LAYERS),
                ("out_kv", ctypes.c_void_p * MAX_PREFIX_LAYERS)]


class LongPrefix(ctypes.Structure):
    _fields_ = [("rank", ctypes.c_int), ("max_clients", ctypes.c_int),
                ("rademacher", ctypes.c_void_p)]


class TraceHeader(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("rounds", ctypes.c_int32), ("n_clusters", ctypes.c_int32),
                ("filled", ctypes.c_int32), ("s_x", ctypes.c_float), ("delta_bar", ctypes.c_float),
                ("F_S", ctypes.c_float * 3), ("F_V", ctypes.c_float * 3), ("c_B", ctypes.c_float),
                ("reserved", ctypes.c_int32 * 3)]


class TraceLayout(ctypes.Structure):
    _fields_ = [("bytes_per_image", ctypes.c_size_t), ("rounds_max", ctypes.c_int),
                ("pool_size", ctypes.c_int), ("off_order", ctypes.c_size_t),
                ("off_round_end", ctypes.c_size_t), ("off_pool", ctypes.c_size_t),
                ("off_centres", ctypes.c_size_t), ("off_head_assign", ctypes.c_size_t),
                ("off_omega", ctypes.c_size_t), ("off_pi", ctypes.c_size_t),
                ("off_ebar", ctypes.c_size_t), ("off_mass", ctypes.c_size_t),
                ("off_gains", ctypes.c_size_t), ("off_cover", ctypes.c_size_t)]


_lib = None


def lib() -> ctypes.CDLL:
    """Load libgmc.so (raises if it is missing: build it with __graft_entry__.build())."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing; build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    vp, sz, i = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int
    P, PP = ctypes.POINTER(Params), ctypes.POINTER(Problem)
    L.gmc_default_params.argtypes = [P]
    L.gmc_default_params.restype = None
    L.gmc_workspace_size.argtypes = [PP, i, i, i, i, i, i]
    L.gmc_workspace_size.restype = sz
    L.gmc_compress.argtypes = [PP, P, vp, vp, vp, vp, vp, i, i, i, i, i, i, vp, vp, vp, vp, vp,
                               sz, vp, vp]
    L.gmc_compress.restype = i
    L.gmc_compress_host.argtypes = [PP, P, ctypes.POINTER(HostIO), i, i, i, i, i, i, vp, sz, vp,
                                    vp]
    L.gmc_compress_host.restype = i
    L.gmc_workspace_size_views.argtypes = [PP, i, i, i, i, i, i, i]
    L.gmc_workspace_size_views.restype = sz
    L.gmc_compress_views.argtypes = [PP, P, ctypes.POINTER(Views), vp, vp, vp, vp, vp, i, i, i, i,
                                     i, i, vp, vp, vp, vp, vp, sz, vp, vp]
    L.gmc_compress_views.restype = i
    L.gmc_get_trace_layout.argtypes = [PP, P, i, i, i, i, ctypes.POINTER(TraceLayout)]
    L.gmc_get_trace_layout.restype = i
    L.gmc_trace_size.argtypes = [PP, P, i, i, i, i]
    L.gmc_trace_size.restype = sz
    L.gmc_select_workspace_size.argtypes = [i, i, i, i, P]
    L.gmc_select_workspace_size.restype = sz
    L.gmc_select.argtypes = [vp, i, i, i, i, P, vp, vp, sz, vp, vp]
    L.gmc_select.restype = i
    L.gmc_transport_workspace_size.argtypes = [PP, i, i, i]
    L.gmc_transport_workspace_size.restype = sz
    L.gmc_transport.argtypes = [PP, P, vp, vp, vp, vp, vp, vp, i, i, i, i, i, vp, vp, vp, vp, vp,
                                sz, vp]
    L.gmc_transport.restype = i
    L.gmc_read_status.argtypes = [vp, ctypes.POINTER(ctypes.c_uint32), vp]
    L.gmc_read_status.restype = i
    L.gmc_error_string.argtypes = [i]
    L.gmc_error_string.restype = ctypes.c_char_p
    L.gmc_version.argtypes = []
    L.gmc_version.restype = ctypes.c_char_p
    L.gmc_profile_enable.argtypes = [i]
    L.gmc_profile_enable.restype = i
    L.gmc_profile_read.argtypes = [ctypes.POINTER(ctypes.c_float), ctypes.POINTER(ctypes.c_char_p), i]
    L.gmc_profile_read.restype = i
    L.gmc_launch_count.argtypes = []
    L.gmc_launch_count.restype = ctypes.c_uint64
    L.gmc_transport_noalloc.argtypes = [PP, P, vp, vp, vp, vp, vp, vp, i, i, i, i, i, vp, vp, vp,
                                        vp, vp, vp]
    L.gmc_transport_noalloc.restype = i
    L.gmc_cosine_workspace_size.argtypes = [PP, i]
    L.gmc_cosine_workspace_size.restype = sz
    L.gmc_cosine.argtypes = [PP, P, vp, i, i, i, vp, vp, sz, vp]
    L.gmc_cosine.restype = i
    L.gmc_compress_ex.argtypes = [PP, P, ctypes.POINTER(Views), ctypes.POINTER(PrefixKV), vp, vp,
                                  vp, vp, vp, i, i, i, i, i, i, vp, vp, vp, vp, vp, sz, vp, vp]
    L.gmc_compress_ex.restype = i
    L.gmc_clients.argtypes = [PP, P, ctypes.POINTER(Views), vp, vp, vp, vp, vp, i, i, i, i, i, i,
                              vp, vp, sz, vp, vp]
    L.gmc_clients.restype = i
    LP = ctypes.POINTER(LongPrefix)
    L.gmc_workspace_size_long.argtypes = [PP, P, LP, i, i, i, i, i, i, i]
    L.gmc_workspace_size_long.restype = sz
    L.gmc_compress_long.argtypes = [PP, P, LP, ctypes.POINTER(Views), ctypes.POINTER(PrefixKV), vp,
                                    vp, vp, vp, vp, i, i, i, i, i, i, vp, vp, vp, vp, vp, sz, vp, vp]
    L.gmc_compress_long.restype = i
    L.gmc_clients_long.argtypes = [PP, P, LP, ctypes.POINTER(Views), vp, vp, vp, vp, vp, i, i, i,
                                   i, i, i, vp, vp, sz, vp, vp]
    L.gmc_clients_long.restype = i
    L.gmc_selftest_bounded_wait.argtypes = [ctypes.c_longlong, vp, sz, vp]
    L.gmc_selftest_bounded_wait.restype = i
    _lib = L
    return L


class GMCError(RuntimeError):
    pass


def _check(rc: int):
    if rc != GMC_OK:
        raise GMCError(lib().gmc_error_string(rc).decode())


def default_params(**overrides) -> Params:
    p = Params()
    lib().gmc_default_params(ctypes.byref(p))
    for k, v in overrides.items():
        if k not in {f[0] for f in Params._fields_}:
            raise KeyError(k)
        setattr(p, k, v)
    return p


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def problem(B, grid_h, grid_w, Hkv, dtype, text_offsets=None, images=1) -> Problem:
    return Problem(B, grid_h, grid_w, Hkv, dtype,
                   None if text_offsets is None else text_offsets.data_ptr(), images)


def workspace_size(prob: Problem, N, T, H, d, D, K) -> int:
    return int(lib().gmc_workspace_size(ctypes.byref(prob), N, T, H, d, D, K))


def trace_layout(prob: Problem, params: Params, N, T, H, K) -> TraceLayout:
    L = TraceLayout()
    _check(lib().gmc_get_trace_layout(ctypes.byref(prob), ctypes.byref(params), N, T, H, K, ctypes.byref(L)))
    return L


def alloc_workspace(nbytes: int, device="cuda") -> torch.Tensor:
    # torch's caching allocator returns 512-byte aligned blocks
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)


def compress(prob: Problem, params: Params, hidden, keys, queries, pos_ids, vo_probe,
             N, T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace, trace=None,
             stream=None):
    """gmc_compress on device tensors (see include/gmc.h for layouts)."""
    _check(lib().gmc_compress(
        ctypes.byref(prob), ctypes.byref(params), _ptr(hidden), _ptr(keys), _ptr(queries),
        _ptr(pos_ids), _ptr(vo_probe), N, T, H, d, D, K, _ptr(out_idx), _ptr(out_hidden),
        _ptr(out_kv), _ptr(out_pos), _ptr(workspace), workspace.numel(), _ptr(trace),
        _stream(stream)))


def _nbytes(t) -> int:
    return t.numel() * t.element_size()


def compress_host(prob: Problem, params: Params, host_in, dev_in, dev_out, host_out, N, T, H, d,
                  D, K, workspace, trace=None, stream=None):
    """gmc_compress_host: inputs from page-locked host tensors through the device
    tensors `dev_in`, outputs back into page-locked host tensors.  host_in / dev_in:
    dicts with hidden, keys, queries, pos_ids, vo_probe; dev_out / host_out: dicts
    with idx, hidden, kv, pos."""
    io = HostIO()
    for n in ("hidden", "keys", "queries", "pos_ids", "vo_probe"):
        setattr(io, n, _ptr(host_in[n]))
        setattr(io, "d_" + n, _ptr(dev_in[n]))
        setattr(io, n + "_bytes", _nbytes(host_in[n]))
    for n, k in (("out_idx", "idx"), ("out_hidden", "hidden"), ("out_kv", "kv"), ("out_pos", "pos")):
        setattr(io, "d_" + n, _ptr(dev_out[k]))
        setattr(io, n, _ptr(host_out[k]))
        setattr(io, n + "_bytes", _nbytes(host_out[k]))
    _check(lib().gmc_compress_host(ctypes.byref(prob), ctypes.byref(params), ctypes.byref(io), N,
                                   T, H, d, D, K, _ptr(workspace), workspace.numel(), _ptr(trace),
                                   _stream(stream)))


def views(keys, queries, vo_probe, beta_hist=0.5) -> Views:
    """Historical message views from per-view device tensors (keys, queries, probes)."""
    v = Views()
    v.n = len(keys)
    v.beta_hist = beta_hist
    for k in range(v.n):
        v.keys[k], v.queries[k], v.vo_probe[k] = _ptr(keys[k]), _ptr(queries[k]), _ptr(vo_probe[k])
    return v


def prefix_kv(keys, outs) -> PrefixKV:
    """Dense prefix layers from per-layer device tensors (inputs as `keys`, outputs as `out_kv`)."""
    if len(keys) != len(outs) or len(keys) > MAX_PREFIX_LAYERS:
        raise GMCError("prefix layers: one output per input, at most 64")
    pf = PrefixKV()
    pf.n_layers = len(keys)
    for l, (k, o) in enumerate(zip(keys, outs)):
        pf.keys[l], pf.out_kv[l] = _ptr(k), _ptr(o)
    return pf


def compress_ex(prob: Problem, params: Params, vw, pf, hidden, keys, queries, pos_ids, vo_probe,
                N, T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace, trace=None,
                stream=None):
    """gmc_compress_ex on device tensors (vw, pf: Views / PrefixKV or None; see include/gmc.h)."""
    _check(lib().gmc_compress_ex(
        ctypes.byref(prob), ctypes.byref(params), ctypes.byref(vw) if vw is not None else None,
        ctypes.byref(pf) if pf is not None else None, _ptr(hidden), _ptr(keys), _ptr(queries),
        _ptr(pos_ids), _ptr(vo_probe), N, T, H, d, D, K, _ptr(out_idx), _ptr(out_hidden),
        _ptr(out_kv), _ptr(out_pos), _ptr(workspace), workspace.numel(), _ptr(trace),
        _stream(stream)))


def workspace_size_views(prob: Problem, n_views, N, T, H, d, D, K) -> int:
    return int(lib().gmc_workspace_size_views(ctypes.byref(prob), n_views, N, T, H, d, D, K))


def compress_views(prob: Problem, params: Params, vw: Views, hidden, keys, queries, pos_ids,
                   vo_probe, N, T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace,
                   trace=None, stream=None):
    """gmc_compress_views on device tensors (see include/gmc.h)."""
    _check(lib().gmc_compress_views(
        ctypes.byref(prob), ctypes.byref(params), ctypes.byref(vw), _ptr(hidden), _ptr(keys),
        _ptr(queries), _ptr(pos_ids), _ptr(vo_probe), N, T, H, d, D, K, _ptr(out_idx),
        _ptr(out_hidden), _ptr(out_kv), _ptr(out_pos), _ptr(workspace), workspace.numel(),
        _ptr(trace), _stream(stream)))


def clients(prob: Problem, params: Params, vw: Views | None, hidden, keys, queries, pos_ids,
            vo_probe, N, T, H, d, D, K, out_clients, workspace, trace=None, stream=None):
    """gmc_clients: the client matrix alone, float[B][M][N] into out_clients (see include/gmc.h)."""
    _check(lib().gmc_clients(
        ctypes.byref(prob), ctypes.byref(params), ctypes.byref(vw) if vw is not None else None,
        _ptr(hidden), _ptr(keys), _ptr(queries), _ptr(pos_ids), _ptr(vo_probe), N, T, H, d, D, K,
        _ptr(out_clients), _ptr(workspace), workspace.numel(), _ptr(trace), _stream(stream)))


def long_prefix(rademacher, max_clients=4096) -> LongPrefix:
    """The bounded appearance bank of long prefixes: rademacher is the device
    bf16 [r][D] map (entries +-1), max_clients the M_V cap."""
    return LongPrefix(int(rademacher.shape[0]), int(max_clients), rademacher.data_ptr())


def workspace_size_long(prob: Problem, params: Params, lp: LongPrefix, n_views, N, T, H, d, D,
                        K) -> int:
    return int(lib().gmc_workspace_size_long(ctypes.byref(prob), ctypes.byref(params),
                                             ctypes.byref(lp), n_views, N, T, H, d, D, K))


def compress_long(prob: Problem, params: Params, lp: LongPrefix, vw, pf, hidden, keys, queries,
                  pos_ids, vo_probe, N, T, H, d, D, K, out_idx, out_hidden, out_kv, out_pos,
                  workspace, trace=None, stream=None):
    """gmc_compress_long on device tensors (vw, pf: Views / PrefixKV or None; see include/gmc.h)."""
    _check(lib().gmc_compress_long(
        ctypes.byref(prob), ctypes.byref(params), ctypes.byref(lp),
        ctypes.byref(vw) if vw is not None else None, ctypes.byref(pf) if pf is not None else None,
        _ptr(hidden), _ptr(keys), _ptr(queries), _ptr(pos_ids), _ptr(vo_probe), N, T, H, d, D, K,
        _ptr(out_idx), _ptr(out_hidden), _ptr(out_kv), _ptr(out_pos), _ptr(workspace),
        workspace.numel(), _ptr(trace), _stream(stream)))


def clients_long(prob: Problem, params: Params, lp: LongPrefix, vw, hidden, keys, queries,
                 pos_ids, vo_probe, N, T, H, d, D, K, out_clients, workspace, trace=None,
                 stream=None):
    """gmc_clients_long: the client matrix with the bounded appearance bank."""
    _check(lib().gmc_clients_long(
        ctypes.byref(prob), ctypes.byref(params), ctypes.byref(lp),
        ctypes.byref(vw) if vw is not None else None, _ptr(hidden), _ptr(keys), _ptr(queries),
        _ptr(pos_ids), _ptr(vo_probe), N, T, H, d, D, K, _ptr(out_clients), _ptr(workspace),
        workspace.numel(), _ptr(trace), _stream(stream)))


def selftest_bounded_wait(cycles: int, workspace, stream=None):
    """gmc_selftest_bounded_wait: a device wait that nothing ends, bounded by `cycles` clocks."""
    _check(lib().gmc_selftest_bounded_wait(cycles, _ptr(workspace), workspace.numel(),
                                           _stream(stream)))


def select(clients, B, M, N, K, params: Params, out_idx, workspace, trace=None, stream=None):
    _check(lib().gmc_select(_ptr(clients), B, M, N, K, ctypes.byref(params), _ptr(out_idx),
                            _ptr(workspace), workspace.numel(), _ptr(trace), _stream(stream)))


def select_workspace_size(B, M, N, K, params: Params) -> int:
    return int(lib().gmc_select_workspace_size(B, M, N, K, ctypes.byref(params)))


def transport(prob: Problem, params: Params, hidden, keys, pos_ids, support, assign, weights,
              N, T, d, D, K, out_idx, out_hidden, out_kv, out_pos, workspace, stream=None):
    _check(lib().gmc_transport(
        ctypes.byref(prob), ctypes.byref(params), _ptr(hidden), _ptr(keys), _ptr(pos_ids),
        _ptr(support), _ptr(assign), _ptr(weights), N, T, d, D, K, _ptr(out_idx),
        _ptr(out_hidden), _ptr(out_kv), _ptr(out_pos), _ptr(workspace), workspace.numel(),
        _stream(stream)))


def transport_noalloc(prob: Problem, params: Params, hidden, keys, pos_ids, support, assign,
                      weights, N, T, d, D, K, out_idx, out_hidden, out_kv, out_pos,
                      device_status=None, stream=None):
    """gmc_transport_noalloc: gmc_transport without a workspace (scratch inside the library)."""
    _check(lib().gmc_transport_noalloc(
        ctypes.byref(prob), ctypes.byref(params), _ptr(hidden), _ptr(keys), _ptr(pos_ids),
        _ptr(support), _ptr(assign), _ptr(weights), N, T, d, D, K, _ptr(out_idx),
        _ptr(out_hidden), _ptr(out_kv), _ptr(out_pos), _ptr(device_status), _stream(stream)))


def cosine(prob: Problem, params: Params, hidden, N, T, D, out_cos, workspace=None, stream=None):
    """gmc_cosine: cos [B][N][N] of the visual states (the Gram stage alone)."""
    if workspace is None:
        workspace = alloc_workspace(int(lib().gmc_cosine_workspace_size(ctypes.byref(prob), N)),
                                    out_cos.device)
    _check(lib().gmc_cosine(ctypes.byref(prob), ctypes.byref(params), _ptr(hidden), N, T, D,
                            _ptr(out_cos), _ptr(workspace), workspace.numel(), _stream(stream)))
    return workspace


def transport_workspace_size(prob: Problem, N, T, K) -> int:
    return int(lib().gmc_transport_workspace_size(ctypes.byref(prob), N, T, K))


def read_status(workspace, stream=None) -> int:
    st = ctypes.c_uint32(0)
    _check(lib().gmc_read_status(_ptr(workspace), ctypes.byref(st), _stream(stream)))
    return int(st.value)


def version() -> str:
    return lib().gmc_version().decode()


def profile_enable(on: bool):
    lib().gmc_profile_enable(1 if on else 0)


def profile_read() -> dict:
    """Per-stage milliseconds of the last profiled gmc_compress call."""
    ms = (ctypes.c_float * 16)()
    names = (ctypes.c_char_p * 16)()
    n = lib().gmc_profile_read(ms, names, 16)
    return {names[k].decode(): float(ms[k]) for k in range(max(n, 0))}


def launch_count() -> int:
    return int(lib().gmc_launch_count())


# ---------------------------------------------------------------------------
# Convenience: one call on a workload, outputs as torch tensors
# ---------------------------------------------------------------------------
@dataclass
class Outputs:
    idx: torch.Tensor
    hidden: torch.Tensor
    kv: torch.Tensor
    pos: torch.Tensor
    K: int
    trace: torch.Tensor | None = None
    layout: TraceLayout | None = None


class Compressor:
    """Holds device buffers for repeated gmc_compress calls on one problem shape.

    Inputs are device tensors in the C-ABI layout; ``run`` launches one call
    on the current stream.  ``run_host`` stages pinned host inputs in, runs,
    and copies the outputs back (the end-to-end path through host memory).
    """

    def __init__(self, B, grid_h, grid_w, T, H, Hkv, d, D, K, dtype, text_lengths=None,
                 params: Params | None = None, trace=False, device="cuda", n_views=0, images=1,
                 long_prefix: LongPrefix | None = None):
        self.B, self.gh, self.gw, self.T, self.H, self.Hkv, self.d, self.D = B, grid_h, grid_w, T, H, Hkv, d, D
        self.images = images
        self.N = grid_h * grid_w * images
        self.Kr = K
        self.K = min(self.N, max(images, K))
        self.dtype = dtype
        self.tdt = torch.bfloat16 if dtype == GMC_BF16 else torch.float32
        self.params = params or default_params()
        self.device = device
        lens = list(text_lengths) if text_lengths is not None else [T] * B
        self.text_lengths = lens
        off = [0]
        for t in lens:
            off.append(off[-1] + t)
        self.offsets = torch.tensor(off, dtype=torch.int32, device=device) if text_lengths is not None else None
        self.prob = problem(B, grid_h, grid_w, Hkv, dtype, self.offsets, images)
        self.n_views = n_views
        self.long_prefix = long_prefix
        if long_prefix is not None:
            ws = workspace_size_long(self.prob, self.params, long_prefix, n_views, self.N, T, H, d,
                                     D, K)
        else:
            ws = workspace_size_views(self.prob, n_views, self.N, T, H, d, D, K)
        if ws == 0:
            raise GMCError("invalid problem for gmc_workspace_size")
        self.workspace = alloc_workspace(ws, device)
        tot_text = off[-1]
        Kx = self.K
        self.out_idx = torch.empty(B * Kx, dtype=torch.int32, device=device)
        self.out_hidden = torch.empty((B * Kx + tot_text, D), dtype=self.tdt, device=device)
        self.out_kv = torch.empty((2 * (B * Kx + tot_text), Hkv, d), dtype=self.tdt, device=device)
        self.out_pos = torch.empty(3 * (B * Kx + tot_text), dtype=torch.int32, device=device)
        self.trace = None
        self.layout = None
        if trace:
            self.layout = trace_layout(self.prob, self.params, self.N, T, H, K)
            self.trace = torch.zeros(B * self.layout.bytes_per_image, dtype=torch.uint8, device=device)

    def run(self, hidden, keys, queries, pos_ids, vo_probe, stream=None, history=None,
            beta_hist=0.5, prefix=None):
        """history: None, or (keys, queries, vo_probe) lists of the historical views;
        prefix: None, or the dense prefix layers' K/V tensors (layout of `keys`),
        gathered into self.out_prefix (one tensor per layer, layout of out_kv)."""
        if history is not None and len(history[0]) > self.n_views:
            raise GMCError("more historical views than the workspace was sized for")
        if self.long_prefix is not None:
            pf = None
            if prefix is not None:
                if getattr(self, "out_prefix", None) is None or len(self.out_prefix) != len(prefix):
                    self.out_prefix = [torch.empty_like(self.out_kv) for _ in prefix]
                pf = prefix_kv(prefix, self.out_prefix)
            vw = views(*history, beta_hist=beta_hist) if history is not None else None
            compress_long(self.prob, self.params, self.long_prefix, vw, pf, hidden, keys, queries,
                          pos_ids, vo_probe, self.N, self.T, self.H, self.d, self.D, self.Kr,
                          self.out_idx, self.out_hidden, self.out_kv, self.out_pos,
                          self.workspace, self.trace, stream)
        elif prefix is not None:
            if history is not None and len(history[0]) > self.n_views:
                raise GMCError("more historical views than the workspace was sized for")
            if getattr(self, "out_prefix", None) is None or len(self.out_prefix) != len(prefix):
                self.out_prefix = [torch.empty_like(self.out_kv) for _ in prefix]
            vw = views(*history, beta_hist=beta_hist) if history is not None else None
            compress_ex(self.prob, self.params, vw, prefix_kv(prefix, self.out_prefix), hidden,
                        keys, queries, pos_ids, vo_probe, self.N, self.T, self.H, self.d, self.D,
                        self.Kr, self.out_idx, self.out_hidden, self.out_kv, self.out_pos,
                        self.workspace, self.trace, stream)
        elif history is None:
            compress(self.prob, self.params, hidden, keys, queries, pos_ids, vo_probe, self.N,
                     self.T, self.H, self.d, self.D, self.Kr, self.out_idx, self.out_hidden,
                     self.out_kv, self.out_pos, self.workspace, self.trace, stream)
        else:
            if len(history[0]) > self.n_views:
                raise GMCError("more historical views than the workspace was sized for")
            vw = views(*history, beta_hist=beta_hist)
            compress_views(self.prob, self.params, vw, hidden, keys, queries, pos_ids, vo_probe,
                           self.N, self.T, self.H, self.d, self.D, self.Kr, self.out_idx,
                           self.out_hidden, self.out_kv, self.out_pos, self.workspace, self.trace,
                           stream)
        return Outputs(self.out_idx, self.out_hidden, self.out_kv, self.out_pos, self.K, self.trace,
                       self.layout)

    def run_host(self, host_in, dev_in, host_out, stream=None):
        """gmc_compress_host: the inputs in page-locked host tensors (dict: hidden, keys,
        queries, pos_ids, vo_probe) copied through the device tensors `dev_in`, the outputs
        (this Compressor's device buffers) copied back into `host_out` (dict: idx, hidden,
        kv, pos).  Synchronise the stream before reading host_out."""
        if self.long_prefix is not None:
            raise GMCError("run_host covers gmc_compress (no long-prefix bank)")
        compress_host(self.prob, self.params, host_in, dev_in,
                      {"idx": self.out_idx, "hidden": self.out_hidden, "kv": self.out_kv,
                       "pos": self.out_pos}, host_out, self.N, self.T, self.H, self.d, self.D,
                      self.Kr, self.workspace, self.trace, stream)

    def status(self, stream=None) -> int:
        return read_status(self.workspace, stream)
